// Dense projections of the layer on CUDA cores (fp32 FMA).  This is the path for fp32 storage
// and the reference shape for the tensor-core kernels.
//
// Forward, per destination type t and block of 64 rows (Eq. 7 with one W_r per relation, Eq. 11):
//   Z = sum_{r -> t} M_r W_r        (relation means of Eq. 10 concatenated along K)
//   U = Z W_agg[t] + b[t],  Y = act(U) + H_in,  H_out = LayerNorm_t(Y) (optional)
//   saved: Z, U (storage type), (mean, rstd) per row.
// Backward, per destination type t and block of 64 rows (chain rule of the above):
//   dY  = LayerNorm backward of dH_out (or dH_out), dU = dY * act'(U)
//   dZ  = dU W_agg^T,  dMs_r = (dZ W_r^T) / deg_r(j)  (pre-scaled for the transposed gather)
//   column partials of db = sum dU, dgamma = sum dH_out * x_hat, dbeta = sum dH_out
// Weight gradients (split over rows, fixed-order reduction):
//   dW_agg[t] = Z^T dU,  dW_r = M_r^T dZ
#include <algorithm>

#include "layer_kernels.cuh"
#include "simt_tile.cuh"

namespace hg {

// ---------------------------------------------------------------------------------------------
// forward projection
// ---------------------------------------------------------------------------------------------

template <typename T, int D>
__global__ void __launch_bounds__(256) proj_fwd_simt(FwdArgs a) {
  using TL = Tile<T, D>;
  constexpr int RM = TL::RM, CN = TL::CN;
  extern __shared__ __align__(16) float smem[];
  float(*As)[kAPad] = reinterpret_cast<float(*)[kAPad]>(smem);
  float* Bs = smem + kBM * kAPad;
  float* Zs = Bs + kKC * D;  // kBM x (D + 4)
  constexpr int ZLD = D + 4;
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
  const int64_t m0 = (int64_t)blockIdx.x * kBM;
  const int64_t nv = min((int64_t)kBM, a.n - m0);

  float acc[RM][CN];
#pragma unroll
  for (int i = 0; i < RM; ++i)
#pragma unroll
    for (int j = 0; j < CN; ++j) acc[i][j] = 0.f;
  for (int r = 0; r < a.nrel; ++r) {
    for (int k0 = 0; k0 < D; k0 += kKC) {
      stage_a<T, D>(As, (const T*)a.M, a.mrow0[r] + m0, nv, k0, a.mrow, a.msent);
      stage_b<T, D>(Bs, (const T*)a.W_rel[r], k0);
      __syncthreads();
      mma_chunk<D, RM, CN>(&As[0][0], kAPad, 0, Bs, acc);
      __syncthreads();
    }
  }
  // Z (rounded to the storage type) -> saved and smem operand of the second product
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int m = ty * RM + i;
    float z[CN];
#pragma unroll
    for (int j = 0; j < CN; ++j) {
      z[j] = round_to<T>(acc[i][j]);
      Zs[m * ZLD + tx * CN + j] = z[j];
      acc[i][j] = 0.f;
    }
    if (m < nv) store_cols<T, CN>((T*)a.Z + (a.off + m0 + m) * D + tx * CN, z);
  }
  __syncthreads();
  for (int k0 = 0; k0 < D; k0 += kKC) {
    stage_b<T, D>(Bs, (const T*)a.W_agg, k0);
    __syncthreads();
    mma_chunk<D, RM, CN>(Zs, ZLD, k0, Bs, acc);
    __syncthreads();
  }
  float bias[CN], g[CN], be[CN];
  load_cols<T, CN>((const T*)a.b + tx * CN, bias);
  if (a.ln) {
    load_cols<T, CN>((const T*)a.gamma + tx * CN, g);
    load_cols<T, CN>((const T*)a.beta + tx * CN, be);
  }
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int m = ty * RM + i;
    const bool live = m < nv;
    const int64_t node = a.off + m0 + (live ? m : 0);
    float h[CN], u[CN], y[CN];
    if (live) load_cols<T, CN>((const T*)a.H_in + node * D + tx * CN, h);
    float s = 0.f;
#pragma unroll
    for (int j = 0; j < CN; ++j) {
      u[j] = round_to<T>(acc[i][j] + bias[j]);
      y[j] = act_apply(u[j], a.act) + (live ? h[j] : 0.f);
      s += y[j];
    }
    if (live) store_cols<T, CN>((T*)a.U + node * D + tx * CN, u);
    if (a.ln) {
      const float mean = row_sum16(s) * (1.f / D);
      float q = 0.f;
#pragma unroll
      for (int j = 0; j < CN; ++j) q += (y[j] - mean) * (y[j] - mean);
      const float var = row_sum16(q) * (1.f / D);
      const float rstd = rsqrtf(var + a.eps);
#pragma unroll
      for (int j = 0; j < CN; ++j) y[j] = (y[j] - mean) * rstd * g[j] + be[j];
      if (live && tx == 0) a.stats[node] = make_float2(mean, rstd);
    }
    if (live) store_cols<T, CN>((T*)a.H_out + node * D + tx * CN, y);
  }
}

// ---------------------------------------------------------------------------------------------
// backward, row side
// ---------------------------------------------------------------------------------------------

template <typename T, int D>
__global__ void __launch_bounds__(256) proj_bwd_simt(BwdArgs a) {
  using TL = Tile<T, D>;
  constexpr int RM = TL::RM, CN = TL::CN;
  constexpr int LD = D + 4;
  extern __shared__ __align__(16) float smem[];
  float* Us = smem;               // kBM x LD: dU operand
  float* Zs = Us + kBM * LD;      // kBM x LD: dZ operand
  float* Bs = Zs + kBM * LD;      // kKC x D
  float* red = Bs + kKC * D;      // 16 x 3 x D column partials
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
  const int64_t m0 = (int64_t)blockIdx.x * kBM;
  const int64_t nv = min((int64_t)kBM, a.n - m0);

  float g[CN];
  if (a.ln) load_cols<T, CN>((const T*)a.gamma + tx * CN, g);
  float cdb[CN], cdg[CN], cdbe[CN];
#pragma unroll
  for (int j = 0; j < CN; ++j) cdb[j] = cdg[j] = cdbe[j] = 0.f;
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int m = ty * RM + i;
    const bool live = m < nv;
    const int64_t node = a.off + m0 + (live ? m : 0);
    float dout[CN], u[CN], h[CN], dy[CN], du[CN];
    if (live) {
      load_cols<T, CN>((const T*)a.dH_out + node * D + tx * CN, dout);
      load_cols<T, CN>((const T*)a.U + node * D + tx * CN, u);
      load_cols<T, CN>((const T*)a.H_in + node * D + tx * CN, h);
    } else {
#pragma unroll
      for (int j = 0; j < CN; ++j) dout[j] = u[j] = h[j] = 0.f;
    }
    if (a.ln) {
      const float2 st = live ? a.stats[node] : make_float2(0.f, 0.f);
      float xh[CN], dxh[CN], s1 = 0.f, s2 = 0.f;
#pragma unroll
      for (int j = 0; j < CN; ++j) {
        xh[j] = (act_apply(u[j], a.act) + h[j] - st.x) * st.y;
        dxh[j] = dout[j] * g[j];
        s1 += dxh[j];
        s2 += dxh[j] * xh[j];
        cdg[j] += dout[j] * xh[j];
        cdbe[j] += dout[j];
      }
      const float mean1 = row_sum16(s1) * (1.f / D), mean2 = row_sum16(s2) * (1.f / D);
#pragma unroll
      for (int j = 0; j < CN; ++j) dy[j] = st.y * (dxh[j] - mean1 - xh[j] * mean2);
    } else {
#pragma unroll
      for (int j = 0; j < CN; ++j) dy[j] = dout[j];
    }
#pragma unroll
    for (int j = 0; j < CN; ++j) {
      du[j] = round_to<T>(dy[j] * act_grad(u[j], a.act));
      if (!live) du[j] = 0.f;
      cdb[j] += du[j];
      Us[m * LD + tx * CN + j] = du[j];
    }
    if (live) {
      store_cols<T, CN>((T*)a.dY + node * D + tx * CN, dy);
      store_cols<T, CN>((T*)a.dU + node * D + tx * CN, du);
    }
  }
  // column partials of this block: reduce the 16 row groups in fixed order
#pragma unroll
  for (int j = 0; j < CN; ++j) {
    red[(ty * 3 + 0) * D + tx * CN + j] = cdb[j];
    red[(ty * 3 + 1) * D + tx * CN + j] = cdg[j];
    red[(ty * 3 + 2) * D + tx * CN + j] = cdbe[j];
  }
  __syncthreads();
  for (int k = threadIdx.x; k < 3 * D; k += blockDim.x) {
    float s = 0.f;
    for (int r = 0; r < 16; ++r) s += red[r * 3 * D + k];
    a.part[(int64_t)blockIdx.x * 3 * D + k] = s;
  }
  // dZ = dU W_agg^T
  float acc[RM][CN];
#pragma unroll
  for (int i = 0; i < RM; ++i)
#pragma unroll
    for (int j = 0; j < CN; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < D; k0 += kKC) {
    stage_b<T, D>(Bs, (const T*)a.W_aggT, k0);
    __syncthreads();
    mma_chunk<D, RM, CN>(Us, LD, k0, Bs, acc);
    __syncthreads();
  }
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int m = ty * RM + i;
    float z[CN];
#pragma unroll
    for (int j = 0; j < CN; ++j) {
      z[j] = round_to<T>(acc[i][j]);
      Zs[m * LD + tx * CN + j] = z[j];
    }
    if (m < nv) store_cols<T, CN>((T*)a.dZ + (a.off + m0 + m) * D + tx * CN, z);
  }
  __syncthreads();
  // dMs_r = (dZ W_r^T) / deg_r
  for (int r = 0; r < a.nrel; ++r) {
#pragma unroll
    for (int i = 0; i < RM; ++i)
#pragma unroll
      for (int j = 0; j < CN; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < D; k0 += kKC) {
      stage_b<T, D>(Bs, (const T*)a.W_relT[r], k0);
      __syncthreads();
      mma_chunk<D, RM, CN>(Zs, LD, k0, Bs, acc);
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < RM; ++i) {
      const int m = ty * RM + i;
      if (m >= nv) continue;
      const int64_t row = a.mrow0[r] + m0 + m;
      const int64_t out = a.mrow ? (int64_t)a.mrow[row] : row;  // compact rows: empty rows are not stored
      if (a.mrow && out >= a.msent) continue;
      const int deg = a.csr_ptr ? a.csr_ptr[row + 1] - a.csr_ptr[row] : 0;
      const float sc = !a.csr_ptr ? 1.f : (deg > 0 ? __fdiv_rn(1.0f, (float)deg) : 0.f);
      float v[CN];
#pragma unroll
      for (int j = 0; j < CN; ++j) v[j] = acc[i][j] * sc;
      store_cols<T, CN>((T*)a.dMs + out * D + tx * CN, v);
    }
  }
}

// ---------------------------------------------------------------------------------------------
// weight gradients: out = X^T Y over rows, split over row ranges, fixed-order reduction
// ---------------------------------------------------------------------------------------------
constexpr int kWT = 128;  // output tile edge (D >= 128) or D
constexpr int kWR = 32;   // rows per step

template <typename T, int D>
__global__ void __launch_bounds__(256) wgrad_partial(const T* __restrict__ X, int64_t x0, const T* __restrict__ Y,
                                                     int64_t y0, int64_t n, int64_t rows_per_split,
                                                     float* __restrict__ part, const int32_t* __restrict__ xmap,
                                                     int64_t xsent) {
  constexpr int TW = D < kWT ? D : kWT;
  constexpr int TPT = TW / 16;  // outputs per thread per dim
  constexpr int VEC = VecTraits<T>::kElems;
  __shared__ __align__(16) float Xs[kWR][TW];
  __shared__ __align__(16) float Ys[kWR][TW];
  const int tiles_per_dim = D / TW;
  const int ti = blockIdx.x / tiles_per_dim, tj = blockIdx.x % tiles_per_dim;
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
  const int64_t r0 = (int64_t)blockIdx.y * rows_per_split;
  const int64_t r1 = min(n, r0 + rows_per_split);
  float acc[TPT][TPT];
#pragma unroll
  for (int i = 0; i < TPT; ++i)
#pragma unroll
    for (int j = 0; j < TPT; ++j) acc[i][j] = 0.f;
  for (int64_t rb = r0; rb < r1; rb += kWR) {
    for (int idx = threadIdx.x; idx < kWR * TW / VEC; idx += blockDim.x) {
      const int k = idx / (TW / VEC), cv = idx % (TW / VEC);
      float fx[VEC], fy[VEC];
      const int64_t xr = rb + k < r1 ? (xmap ? (int64_t)xmap[x0 + rb + k] : x0 + rb + k) : 0;
      if (rb + k < r1 && (!xmap || xr < xsent)) {
        unpack(ldg16(X + xr * D + ti * TW + cv * VEC), fx, T());
        unpack(ldg16(Y + (y0 + rb + k) * D + tj * TW + cv * VEC), fy, T());
      } else {
#pragma unroll
        for (int q = 0; q < VEC; ++q) fx[q] = fy[q] = 0.f;
      }
#pragma unroll
      for (int q = 0; q < VEC; ++q) {
        Xs[k][cv * VEC + q] = fx[q];
        Ys[k][cv * VEC + q] = fy[q];
      }
    }
    __syncthreads();
#pragma unroll 4
    for (int k = 0; k < kWR; ++k) {
      float xa[TPT], yb[TPT];
#pragma unroll
      for (int i = 0; i < TPT; i += 4) {
        float4 v = *reinterpret_cast<const float4*>(&Xs[k][ty * TPT + i]);
        xa[i] = v.x; xa[i + 1] = v.y; xa[i + 2] = v.z; xa[i + 3] = v.w;
        float4 w = *reinterpret_cast<const float4*>(&Ys[k][tx * TPT + i]);
        yb[i] = w.x; yb[i + 1] = w.y; yb[i + 2] = w.z; yb[i + 3] = w.w;
      }
#pragma unroll
      for (int i = 0; i < TPT; ++i)
#pragma unroll
        for (int j = 0; j < TPT; ++j) acc[i][j] = fmaf(xa[i], yb[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* out = part + (int64_t)blockIdx.y * D * D;
#pragma unroll
  for (int i = 0; i < TPT; ++i) {
    const int row = ti * TW + ty * TPT + i;
#pragma unroll
    for (int j = 0; j < TPT; j += 4)
      *reinterpret_cast<float4*>(out + (int64_t)row * D + tj * TW + tx * TPT + j) =
          make_float4(acc[i][j], acc[i][j + 1], acc[i][j + 2], acc[i][j + 3]);
  }
}

// out[i] = sum over splits k of part[k * stride + i] in a fixed order: a block owns 32 consecutive
// outputs (one per lane); warp w sums the splits k = w, w + kRedLanes, ... in ascending order, and the
// kRedLanes warp sums are added in warp order.
constexpr int kRedLanes = 32;
// Outputs i in [k * seg, (k + 1) * seg) go to outs.p[k][i - k * seg] (up to three segments).
struct RedOuts {
  float* p[3];
};
__global__ void __launch_bounds__(32 * kRedLanes) reduce_lanes(const float* __restrict__ part, int64_t stride,
                                                             int splits, int64_t count, int64_t seg, RedOuts outs) {
  __shared__ float red[kRedLanes][33];
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int64_t i = (int64_t)blockIdx.x * 32 + lane;
  float s = 0.f;
  if (i < count) {
    int k = w;
    for (; k + 3 * kRedLanes < splits; k += 4 * kRedLanes) {
      float v[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) v[u] = __ldg(part + (int64_t)(k + u * kRedLanes) * stride + i);
#pragma unroll
      for (int u = 0; u < 4; ++u) s += v[u];
    }
    for (; k < splits; k += kRedLanes) s += __ldg(part + (int64_t)k * stride + i);
  }
  red[w][lane] = s;
  __syncthreads();
  if (w == 0 && i < count) {
    float t = 0.f;
#pragma unroll
    for (int k = 0; k < kRedLanes; ++k) t += red[k][lane];
    const int64_t q = i / seg;
    outs.p[q][i - q * seg] = t;
  }
}


template <typename T>
__global__ void transpose_square(const T* __restrict__ W, T* __restrict__ Wt, int d, int count) {
  const int64_t total = (int64_t)count * d * d;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = i / ((int64_t)d * d), rc = i % ((int64_t)d * d);
    const int r = (int)(rc / d), c = (int)(rc % d);
    Wt[m * d * d + (int64_t)c * d + r] = W[i];
  }
}

// ---------------------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------------------
template <typename T, int D>
static size_t fwd_smem() { return sizeof(float) * (kBM * kAPad + kKC * D + kBM * (D + 4)); }
template <typename T, int D>
static size_t bwd_smem() { return sizeof(float) * (2 * kBM * (D + 4) + kKC * D + 16 * 3 * D); }

template <typename T, int D>
static hg_status set_smem_once() {
  static bool done = false;  // per instantiation; attribute is per function and device-wide
  if (!done) {
    HG_CUDA(cudaFuncSetAttribute(proj_fwd_simt<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)fwd_smem<T, D>()));
    HG_CUDA(cudaFuncSetAttribute(proj_bwd_simt<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bwd_smem<T, D>()));
    done = true;
  }
  return HG_OK;
}

template <typename T, int D>
static hg_status proj_fwd_t(const FwdArgs& a, cudaStream_t s) {
  HG_TRY((set_smem_once<T, D>()));
  return launch("proj_fwd_simt", proj_fwd_simt<T, D>, dim3((unsigned)ceil_div(a.n, kBM)), dim3(256), fwd_smem<T, D>(), s, a);
}

template <typename T, int D>
static hg_status proj_bwd_t(const BwdArgs& a, cudaStream_t s) {
  HG_TRY((set_smem_once<T, D>()));
  return launch("proj_bwd_simt", proj_bwd_simt<T, D>, dim3((unsigned)ceil_div(a.n, kBM)), dim3(256), bwd_smem<T, D>(), s, a);
}

int wgrad_splits(int64_t n) {
  return (int)std::max<int64_t>(1, std::min<int64_t>(304, ceil_div(n, 256)));
}

hg_status reduce_partials(const float* part, int64_t stride, int splits, int64_t count, float* out, float* tmp,
                          cudaStream_t s);

template <typename T, int D>
static hg_status wgrad_t(const void* X, int64_t x0, const void* Y, int64_t y0, int64_t n, float* part, float* out,
                         float* tmp, const int32_t* xmap, int64_t xsent, cudaStream_t s) {
  const int splits = wgrad_splits(n);
  const int64_t rps = ceil_div(std::max<int64_t>(n, 1), splits);
  constexpr int TW = D < kWT ? D : kWT;
  const int tiles = (D / TW) * (D / TW);
  HG_TRY(launch("wgrad_partial", wgrad_partial<T, D>, dim3(tiles, splits), dim3(256), 0, s, (const T*)X, x0,
                (const T*)Y, y0, n, rps, part, xmap, xsent));
  return reduce_partials(part, (int64_t)D * D, splits, (int64_t)D * D, out, tmp, s);
}

template <typename T, int D>
static hg_status transpose_t(const void* W, void* Wt, int count, cudaStream_t s) {
  return launch("transpose_square", transpose_square<T>, dim3((unsigned)std::min<int64_t>(ceil_div((int64_t)count * D * D, 256), 1024)),
                dim3(256), 0, s, (const T*)W, (T*)Wt, D, count);
}

#define HG_DISPATCH_TD2(dtype, d, FN, ...)                                                  \
  do {                                                                                      \
    if (dtype == HG_F32) {                                                                  \
      if (d == 64) return FN<float, 64>(__VA_ARGS__);                                       \
      if (d == 128) return FN<float, 128>(__VA_ARGS__);                                     \
      if (d == 256) return FN<float, 256>(__VA_ARGS__);                                     \
    } else {                                                                                \
      if (d == 64) return FN<__nv_bfloat16, 64>(__VA_ARGS__);                               \
      if (d == 128) return FN<__nv_bfloat16, 128>(__VA_ARGS__);                             \
      if (d == 256) return FN<__nv_bfloat16, 256>(__VA_ARGS__);                             \
    }                                                                                       \
    set_error("unsupported feature width %d", d);                                           \
    return HG_ERR_UNSUPPORTED;                                                              \
  } while (0)

hg_status proj_forward(hg_dtype dt, int d, const FwdArgs& a, cudaStream_t s) { HG_DISPATCH_TD2(dt, d, proj_fwd_t, a, s); }
hg_status proj_backward(hg_dtype dt, int d, const BwdArgs& a, cudaStream_t s) { HG_DISPATCH_TD2(dt, d, proj_bwd_t, a, s); }
hg_status weight_grad(hg_dtype dt, int d, const void* X, int64_t x0, const void* Y, int64_t y0, int64_t n, float* part,
                      float* out, float* tmp, cudaStream_t s, const int32_t* xmap, int64_t xsent) {
  HG_DISPATCH_TD2(dt, d, wgrad_t, X, x0, Y, y0, n, part, out, tmp, xmap, xsent, s);
}
hg_status transpose_weights(hg_dtype dt, int d, const void* W, void* Wt, int count, cudaStream_t s) {
  HG_DISPATCH_TD2(dt, d, transpose_t, W, Wt, count, s);
}
size_t reduce_tmp_floats(int splits, int64_t count) {
  (void)splits;
  return (size_t)count;  // reduce_partials needs no temporaries; one slot keeps callers' layouts valid
}

// Fixed-order sum over `splits` partial arrays in one pass (reduce_lanes).
hg_status reduce_partials(const float* part, int64_t stride, int splits, int64_t count, float* out, float* tmp,
                          cudaStream_t s) {
  (void)tmp;
  if (count <= 0) return HG_OK;
  RedOuts o{{out, nullptr, nullptr}};
  return launch("reduce_lanes", reduce_lanes, dim3((unsigned)ceil_div(count, 32)), dim3(32 * kRedLanes), 0, s, part,
                stride, splits, count, count, o);
}

hg_status reduce_partials3(const float* part, int64_t stride, int splits, int64_t seg, float* out0, float* out1,
                           float* out2, cudaStream_t s) {
  const int nseg = out1 ? (out2 ? 3 : 2) : 1;
  const int64_t count = seg * nseg;
  if (count <= 0) return HG_OK;
  RedOuts o{{out0, out1, out2}};
  return launch("reduce_lanes", reduce_lanes, dim3((unsigned)ceil_div(count, 32)), dim3(32 * kRedLanes), 0, s, part,
                stride, splits, count, seg, o);
}

}  // namespace hg
