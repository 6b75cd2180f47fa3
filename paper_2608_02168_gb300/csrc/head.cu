// Prediction head and joint objective (Section 3.4, Eq. 18-20; the MeanAgg / MLP / loss steps of
// Algorithm 1).
//
// Forward (hg_head_loss), for the labelled rows r < n of one subgraph:
//   MeanAgg   h_r = H[lab[r]], or (H[lab[r]] + H_rep[j]) / 2 when row lab[r] has a replica j in
//             the second view (the overlap pairs idx_a -> idx_b); the pre-activation uses that
//             mean unrounded (fp32 here, two tensor-core chains for bf16), the rows saved for dW1
//             are rounded to the storage type
//   Eq. 18    a_r = h_r W1 + b1, z_r = relu(a_r) . w2 + b2                 (hidden width d)
//   Eq. 19    L_BCE = (1/n) sum_r [y_r softplus(-z_r) + (1 - y_r) softplus(z_r)]
//   Eq. 20    L_total = L_BCE + lambda_CCA L_CCA
// The gradient of L_BCE per row depends only on that row, so the forward also stores the unit
// gradient dA_r = (sigmoid(z_r) - y_r)/n * w2 * [a_r > 0] and the unit bias / w2 sums; the
// backward (hg_head_bwd) scales them by dloss, forms dh_r = dloss dA_r W1^T (split in halves over
// the two replicas of an overlap row) and dW1 = dloss sum_r h_r^T dA_r.
//
// fp32 storage: row tiles of 64 rows on CUDA cores (fp32 FMA).  bf16 storage: 128-row tiles on the
// tensor cores (head_tc.cu), dW1 by the tensor-core weight-gradient kernel.  Every sum over rows is
// a fixed-order reduction of per-block partials (deterministic).
#include <cuda_bf16.h>

#include <algorithm>

#include "hg_internal.cuh"
#include "head_kernels.cuh"
#include "layer_kernels.cuh"
#include "simt_tile.cuh"

namespace hg {

namespace {

__device__ __forceinline__ float softplus_f(float x) { return fmaxf(x, 0.f) + log1pf(expf(-fabsf(x))); }

__device__ __forceinline__ float sigmoid_f(float z) {
  const float e = expf(-fabsf(z));
  return z >= 0.f ? 1.f / (1.f + e) : e / (1.f + e);
}

// map[idx_a[k]] = idx_b[k] for the k < n overlap pairs whose rows are in range.
__global__ void head_rep_map(const int32_t* __restrict__ ia, const int32_t* __restrict__ ib, int64_t n_max,
                             const int64_t* __restrict__ n_dev, int64_t rows, int64_t rows_rep, int32_t* __restrict__ map) {
  int64_t n = n_max;
  if (n_dev) n = max((int64_t)0, min(n_max, *n_dev));
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < n; k += (int64_t)gridDim.x * blockDim.x) {
    const int32_t a = ia[k], b = ib[k];
    if (a >= 0 && a < rows && b >= 0 && b < rows_rep) map[a] = b;
  }
}

template <typename T, int D>
struct HeadSmem {
  static constexpr int kLda = D + 4;
  static constexpr size_t kFloats = (size_t)kBM * kLda + (size_t)kKC * D + 3 * kBM;
  static constexpr size_t kBytes = kFloats * sizeof(float) + 2 * kBM * sizeof(int32_t);
};

// One block per 64 labelled rows: MeanAgg gather, A = Hm W1 + b1, the logit, the loss term and the
// unit gradients, block partials of the row sums.
template <typename T, int D>
__global__ void __launch_bounds__(256) head_fwd_simt(HeadFwdArgs a) {
  using Tl = Tile<T, D>;
  constexpr int CN = Tl::CN, RM = Tl::RM, VEC = Tl::kVec;
  constexpr int LDA = HeadSmem<T, D>::kLda;
  extern __shared__ __align__(16) float smem[];
  float* As = smem;                       // [kBM][LDA]
  float* Bs = As + kBM * LDA;             // [kKC][D]
  float* yv = Bs + kKC * D;               // [kBM]
  float* red_loss = yv + kBM;             // [kBM]
  float* red_dz = red_loss + kBM;         // [kBM]
  int32_t* rowi = reinterpret_cast<int32_t*>(red_dz + kBM);  // [kBM] labelled row, -1 invalid
  int32_t* repi = rowi + kBM;                                 // [kBM]
  const T* H = (const T*)a.H;
  const T* Hr = (const T*)a.H_rep;
  const int64_t r0 = (int64_t)blockIdx.x * kBM;
  const int tid = threadIdx.x;
  if (tid < kBM) {
    const int64_t r = r0 + tid;
    int32_t i = -1, j = -1;
    float y = 0.f;
    if (r < a.n) {
      const int32_t li = a.lab[r];
      y = a.y[r];
      if (li >= 0 && li < a.rows) {
        i = li;
        j = a.map[li];
      }
      a.rep_row[r] = i >= 0 ? j : -2;
    }
    rowi[tid] = i;
    repi[tid] = j;
    yv[tid] = y;
    red_loss[tid] = 0.f;
    red_dz[tid] = 0.f;
  }
  __syncthreads();
  // MeanAgg rows into As (fp32) and the saved Hm (storage type)
  for (int idx = tid; idx < kBM * (D / VEC); idx += blockDim.x) {
    const int m = idx / (D / VEC), cv = idx % (D / VEC);
    const int64_t r = r0 + m;
    float f[VEC];
#pragma unroll
    for (int q = 0; q < VEC; ++q) f[q] = 0.f;
    if (r < a.n) {
      const int32_t i = rowi[m];
      if (i >= 0) {
        unpack(ldg16(H + (int64_t)i * D + cv * VEC), f, T());
        const int32_t j = repi[m];
        if (j >= 0) {
          float g[VEC];
          unpack(ldg16(Hr + (int64_t)j * D + cv * VEC), g, T());
#pragma unroll
          for (int q = 0; q < VEC; ++q) f[q] = 0.5f * (f[q] + g[q]);
        }
      }
      st16((T*)a.Hm + r * D + cv * VEC, pack(f, T()));
    }
#pragma unroll
    for (int q = 0; q < VEC; ++q) As[m * LDA + cv * VEC + q] = f[q];
  }
  __syncthreads();
  float acc[RM][CN];
#pragma unroll
  for (int i = 0; i < RM; ++i)
#pragma unroll
    for (int j = 0; j < CN; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < D; k0 += kKC) {
    stage_b<T, D>(Bs, (const T*)a.W1, k0);
    __syncthreads();
    mma_chunk<D, RM, CN>(As, LDA, k0, Bs, acc);
    __syncthreads();
  }
  const int ty = tid / 16, tx = tid % 16;
  float b1v[CN], w2v[CN];
  load_cols<T, CN>((const T*)a.b1 + tx * CN, b1v);
  load_cols<T, CN>((const T*)a.w2 + tx * CN, w2v);
  const float b2 = to_f32(((const T*)a.b2)[0]);
  float db1c[CN], dw2c[CN];
#pragma unroll
  for (int j = 0; j < CN; ++j) db1c[j] = dw2c[j] = 0.f;
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int m = ty * RM + i;
    const int64_t r = r0 + m;
    float part = 0.f;
#pragma unroll
    for (int j = 0; j < CN; ++j) {
      acc[i][j] += b1v[j];
      part = fmaf(fmaxf(acc[i][j], 0.f), w2v[j], part);
    }
    const float z = row_sum16(part) + b2;
    float dz = 0.f, term = 0.f;
    if (r < a.n) {
      const float y = yv[m];
      if (rowi[m] >= 0) {
        term = y * softplus_f(-z) + (1.f - y) * softplus_f(z);
        dz = (sigmoid_f(z) - y) * a.inv_n;
      } else {
        term = __int_as_float(0x7fc00000);  // an out-of-range row makes the loss NaN
      }
    }
    float da[CN];
#pragma unroll
    for (int j = 0; j < CN; ++j) {
      da[j] = acc[i][j] > 0.f ? dz * w2v[j] : 0.f;
      db1c[j] += da[j];
      dw2c[j] = fmaf(dz, fmaxf(acc[i][j], 0.f), dw2c[j]);
    }
    if (r < a.n) {
      store_cols<T, CN>((T*)a.dA + r * D + tx * CN, da);
      if (tx == 0) {
        red_loss[m] = term;
        red_dz[m] = dz;
        if (a.logits) a.logits[r] = z;
      }
    }
  }
  // block partials: column sums over the 16 row groups in order, row sums in row order
  float* red = As;  // [16][2D]
#pragma unroll
  for (int j = 0; j < CN; ++j) {
    red[ty * 2 * D + tx * CN + j] = db1c[j];
    red[ty * 2 * D + D + tx * CN + j] = dw2c[j];
  }
  __syncthreads();
  float* out = a.part + (int64_t)blockIdx.x * (2 + 2 * D);
  for (int c = tid; c < 2 * D; c += blockDim.x) {
    float s = 0.f;
    for (int g = 0; g < 16; ++g) s += red[g * 2 * D + c];
    out[2 + c] = s;
  }
  if (tid == 0) {
    float sl = 0.f, sd = 0.f;
    for (int m = 0; m < kBM; ++m) {
      sl += red_loss[m];
      sd += red_dz[m];
    }
    out[0] = sl;
    out[1] = sd;
  }
}

// loss_out[1] = L_BCE = sums[0] / n; loss_out[0] = L_BCE + lambda_CCA * cca[0] (Eq. 20).
__global__ void head_loss_finish(const float* __restrict__ sums, int64_t n, const float* __restrict__ cca, float lam,
                                 float* __restrict__ loss_out) {
  if (threadIdx.x == 0 && blockIdx.x == 0) {
    const float bce = n > 0 ? sums[0] / (float)n : 0.f;
    loss_out[1] = bce;
    loss_out[0] = cca ? bce + lam * cca[0] : bce;
  }
}

// One block per 64 labelled rows: dh = dloss * dA W1^T, added to the row of H (or, for a row with
// a replica, half to it and half to the replica's row of H_rep).  Labelled rows are distinct, so
// every destination row has one writer.
template <typename T, int D>
__global__ void __launch_bounds__(256) head_bwd_dx_simt(HeadBwdArgs a) {
  using Tl = Tile<T, D>;
  constexpr int CN = Tl::CN, RM = Tl::RM;
  extern __shared__ __align__(16) float smem[];
  float(*As)[kAPad] = reinterpret_cast<float(*)[kAPad]>(smem);  // [kBM][kAPad]
  float* Bs = smem + kBM * kAPad;                                // [kKC][D]
  const int64_t r0 = (int64_t)blockIdx.x * kBM;
  const int64_t valid = a.n - r0;
  float acc[RM][CN];
#pragma unroll
  for (int i = 0; i < RM; ++i)
#pragma unroll
    for (int j = 0; j < CN; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < D; k0 += kKC) {
    stage_a<T, D>(As, (const T*)a.dA, r0, valid, k0);
    stage_b<T, D>(Bs, (const T*)a.W1t, k0);
    __syncthreads();
    mma_chunk<D, RM, CN>(&As[0][0], kAPad, 0, Bs, acc);
    __syncthreads();
  }
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int64_t r = r0 + ty * RM + i;
    if (r >= a.n) continue;
    const int32_t rep = a.rep_row[r];
    if (rep == -2) continue;  // out-of-range labelled row: no gradient
    const int64_t li = a.lab[r];
    const float scale = rep >= 0 ? 0.5f * a.dloss : a.dloss;
    float g[CN], v[CN];
#pragma unroll
    for (int j = 0; j < CN; ++j) g[j] = scale * acc[i][j];
    if (a.dH) {
      T* p = (T*)a.dH + li * D + tx * CN;
      load_cols<T, CN>(p, v);
#pragma unroll
      for (int j = 0; j < CN; ++j) v[j] += g[j];
      store_cols<T, CN>(p, v);
    }
    if (rep >= 0 && a.dH_rep) {
      T* p = (T*)a.dH_rep + (int64_t)rep * D + tx * CN;
      load_cols<T, CN>(p, v);
#pragma unroll
      for (int j = 0; j < CN; ++j) v[j] += g[j];
      store_cols<T, CN>(p, v);
    }
  }
}

// dW1 *= dloss (it holds sum_r h_r^T dA_r); db1, dw2, db2 = dloss * the saved unit sums.
__global__ void head_grad_finish(float* __restrict__ dW1, const float* __restrict__ sums, float dloss, int d,
                                 float* __restrict__ db1, float* __restrict__ dw2, float* __restrict__ db2) {
  const int64_t dd = (int64_t)d * d;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < dd; i += (int64_t)gridDim.x * blockDim.x) {
    dW1[i] *= dloss;
    if (i < d) {
      db1[i] = dloss * sums[2 + i];
      dw2[i] = dloss * sums[2 + d + i];
    }
    if (i == 0) db2[0] = dloss * sums[1];
  }
}

// ---------------------------------------------------------------------------------------------
// buffers
// ---------------------------------------------------------------------------------------------
struct HeadLayout {
  void* Hm;
  void* dA;
  int32_t* rep_row;
  float* sums;  // [2 + 2d]
  // forward scratch
  int32_t* map;
  float* part;
  float* tmp;
  // backward scratch (overlaps the forward's)
  void* W1t;
  float* wpart;
  float* wtmp;
};

inline int head_blocks(int64_t n) { return (int)std::max<int64_t>(1, ceil_div(n, kBM)); }

inline int head_wgrad_splits(hg_dtype dt, int64_t n, int d) {
  return dt == HG_BF16 ? wgrad_tc_splits(n, d) : wgrad_splits(n);
}

void carve_head(void* saved, void* scratch, int64_t rows, int64_t n, int d, hg_dtype dt, HeadLayout* L,
                size_t* saved_bytes, size_t* scratch_bytes) {
  const size_t esz = dt == HG_BF16 ? 2 : 4;
  Carve s(saved);
  L->Hm = s.take<char>((size_t)n * d * esz);
  L->dA = s.take<char>((size_t)n * d * esz);
  L->rep_row = s.take<int32_t>((size_t)std::max<int64_t>(n, 1));
  L->sums = s.take<float>(2 + 2 * (size_t)d);
  const int blocks = head_blocks(n);
  Carve f(scratch);
  L->map = f.take<int32_t>((size_t)std::max<int64_t>(rows, 1));
  L->part = f.take<float>((size_t)blocks * (2 + 2 * d));
  L->tmp = f.take<float>(reduce_tmp_floats(blocks, 2 + 2 * d));
  const int splits = head_wgrad_splits(dt, n, d);
  Carve b(scratch);
  L->W1t = b.take<char>((size_t)d * d * esz);
  L->wpart = b.take<float>((size_t)splits * d * d);
  L->wtmp = b.take<float>(reduce_tmp_floats(splits, (int64_t)d * d));
  if (saved_bytes) *saved_bytes = s.used;
  if (scratch_bytes) *scratch_bytes = std::max(f.used, b.used);
}

template <typename T, int D>
hg_status head_smem_once() {
  static bool done = false;
  if (!done) {
    HG_CUDA(cudaFuncSetAttribute(head_fwd_simt<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)HeadSmem<T, D>::kBytes));
    done = true;
  }
  return HG_OK;
}

struct HeadIn {
  const hg_head_params* p;
  const void* H;
  int64_t rows;
  const void* H_rep;
  int64_t rows_rep;
  const int32_t* ia;
  const int32_t* ib;
  int64_t n_rep_max;
  const int64_t* n_rep_dev;
  const int32_t* lab;
  const float* y;
  int64_t n;
};

template <typename T, int D>
hg_status head_loss_t(const HeadIn& in, const float* cca, float lam, float* loss_out, float* logits,
                      const HeadLayout& L, cudaStream_t s) {
  HG_TRY((head_smem_once<T, D>()));
  if (in.n == 0) {
    HG_CUDA(cudaMemsetAsync(L.sums, 0, (2 + 2 * D) * sizeof(float), s));
    return launch("head_loss_finish", head_loss_finish, dim3(1), dim3(32), 0, s, (const float*)L.sums, in.n, cca, lam,
                  loss_out);
  }
  HG_CUDA(cudaMemsetAsync(L.map, 0xFF, (size_t)in.rows * sizeof(int32_t), s));
  if (in.n_rep_max > 0) {
    const unsigned g = (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(in.n_rep_max, 256), 152 * 8));
    HG_TRY(launch("head_rep_map", head_rep_map, dim3(g), dim3(256), 0, s, in.ia, in.ib, in.n_rep_max, in.n_rep_dev,
                  in.rows, in.rows_rep, L.map));
  }
  HeadFwdArgs a;
  a.H = in.H;
  a.rows = in.rows;
  a.H_rep = in.H_rep;
  a.map = L.map;
  a.lab = in.lab;
  a.y = in.y;
  a.n = in.n;
  a.inv_n = 1.f / (float)in.n;
  a.W1 = in.p->W1;
  a.b1 = in.p->b1;
  a.w2 = in.p->w2;
  a.b2 = in.p->b2;
  a.Hm = L.Hm;
  a.dA = L.dA;
  a.rep_row = L.rep_row;
  a.logits = logits;
  a.part = L.part;
  a.status = device_status_ptr();
  int blocks;
  if constexpr (sizeof(T) == 2) {  // bf16: tensor cores
    blocks = (int)ceil_div(in.n, kHeadTcRows);
    HG_TRY(head_fwd_tc(D, a, s));
  } else {
    blocks = head_blocks(in.n);
    HG_TRY(launch("head_fwd_simt", head_fwd_simt<T, D>, dim3(blocks), dim3(256), HeadSmem<T, D>::kBytes, s, a));
  }
  HG_TRY(reduce_partials(L.part, 2 + 2 * D, blocks, 2 + 2 * D, L.sums, L.tmp, s));
  return launch("head_loss_finish", head_loss_finish, dim3(1), dim3(32), 0, s, (const float*)L.sums, in.n, cca, lam,
                loss_out);
}

template <typename T, int D>
hg_status head_bwd_t(const hg_head_params* p, const int32_t* lab, int64_t n, int64_t rows, float dloss,
                     const HeadLayout& L, void* dH, void* dH_rep, const hg_head_grads* g, cudaStream_t s) {
  constexpr hg_dtype kDt = sizeof(T) == 2 ? HG_BF16 : HG_F32;
  if (n > 0 && (dH || dH_rep)) {
    HeadBwdArgs a{L.dA, lab, L.rep_row, n, rows, p->W1, L.W1t, dloss, dH, dH_rep, device_status_ptr()};
    if constexpr (sizeof(T) == 2) {  // bf16: tensor cores, W1 read as it is
      HG_TRY(head_dx_tc(D, a, s));
    } else {
      HG_TRY(transpose_weights(kDt, D, p->W1, L.W1t, 1, s));
      const size_t smem = sizeof(float) * ((size_t)kBM * kAPad + (size_t)kKC * D);
      HG_TRY(launch("head_bwd_dx_simt", head_bwd_dx_simt<T, D>, dim3(head_blocks(n)), dim3(256), smem, s, a));
    }
  }
  if (kDt == HG_BF16) {
    const int64_t x0 = 0;
    float* outs[1] = {g->dW1};
    HG_TRY(tc_weight_grad(D, L.Hm, &x0, 1, L.dA, 0, n, L.wpart, outs, L.wtmp, s));
  } else {
    HG_TRY(weight_grad(kDt, D, L.Hm, 0, L.dA, 0, n, L.wpart, g->dW1, L.wtmp, s));
  }
  return launch("head_grad_finish", head_grad_finish, dim3((unsigned)ceil_div((int64_t)D * D, 256)), dim3(256), 0, s,
                g->dW1, (const float*)L.sums, dloss, D, g->db1, g->dw2, g->db2);
}

#define HG_HEAD_DISPATCH(dtype, d, FN, ...)                                                 \
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

hg_status head_loss_dispatch(const HeadIn& in, const float* cca, float lam, float* loss_out, float* logits,
                             const HeadLayout& L, cudaStream_t s) {
  HG_HEAD_DISPATCH(in.p->dtype, in.p->d, head_loss_t, in, cca, lam, loss_out, logits, L, s);
}

hg_status head_bwd_dispatch(const hg_head_params* p, const int32_t* lab, int64_t n, int64_t rows, float dloss,
                            const HeadLayout& L, void* dH, void* dH_rep, const hg_head_grads* g, cudaStream_t s) {
  HG_HEAD_DISPATCH(p->dtype, p->d, head_bwd_t, p, lab, n, rows, dloss, L, dH, dH_rep, g, s);
}

hg_status check_head_params(const hg_head_params* p) {
  HG_REQUIRE(p != nullptr, "params must be non-null");
  if (!(p->d == 64 || p->d == 128 || p->d == 256) || !(p->dtype == HG_F32 || p->dtype == HG_BF16)) {
    set_error("unsupported d=%d / dtype=%d", p->d, (int)p->dtype);
    return HG_ERR_UNSUPPORTED;
  }
  HG_REQUIRE(p->W1 && p->b1 && p->w2 && p->b2, "W1, b1, w2, b2 must be non-null");
  HG_REQUIRE(((uintptr_t)p->W1 & 15) == 0 && ((uintptr_t)p->b1 & 15) == 0 && ((uintptr_t)p->w2 & 15) == 0,
             "W1, b1 and w2 must be 16-byte aligned");
  return HG_OK;
}

}  // namespace
}  // namespace hg

using namespace hg;

extern "C" hg_status hg_head_workspace_size(int64_t rows, int64_t n_lab, int32_t d, hg_dtype dtype,
                                           size_t* saved_bytes, size_t* scratch_bytes) {
  clear_error();
  HG_REQUIRE(saved_bytes && scratch_bytes, "saved_bytes and scratch_bytes must be non-null");
  HG_REQUIRE(rows >= 0 && n_lab >= 0 && rows < (int64_t(1) << 31) && n_lab < (int64_t(1) << 31),
             "rows and n_lab must be in [0, 2^31)");
  if (!(d == 64 || d == 128 || d == 256) || !(dtype == HG_F32 || dtype == HG_BF16)) {
    set_error("unsupported d=%d / dtype=%d", d, (int)dtype);
    return HG_ERR_UNSUPPORTED;
  }
  HeadLayout L;
  carve_head(nullptr, nullptr, rows, n_lab, d, dtype, &L, saved_bytes, scratch_bytes);
  return HG_OK;
}

extern "C" hg_status hg_head_loss(const hg_head_params* params, const void* H, int64_t rows, const void* H_rep,
                                 int64_t rows_rep, const int32_t* idx_a, const int32_t* idx_b, int64_t n_rep_max,
                                 const int64_t* n_rep_dev, const int32_t* lab_idx, const float* lab_y, int64_t n_lab,
                                 const float* cca_loss, float lambda_cca, float* loss_out, float* logits, void* saved,
                                 void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_head_params(params));
  HG_REQUIRE(loss_out && saved && scratch, "loss_out, saved and scratch must be non-null");
  HG_REQUIRE(((uintptr_t)saved & 255) == 0 && ((uintptr_t)scratch & 255) == 0, "buffers must be 256-byte aligned");
  HG_REQUIRE(rows >= 0 && n_lab >= 0 && n_rep_max >= 0 && rows < (int64_t(1) << 31) && n_lab < (int64_t(1) << 31) &&
                 n_rep_max < (int64_t(1) << 31),
             "rows, n_lab and n_rep_max must be in [0, 2^31)");
  HG_REQUIRE(n_lab == 0 || (H && rows > 0 && lab_idx && lab_y), "H, rows > 0, lab_idx and lab_y are needed when n_lab > 0");
  HG_REQUIRE(n_rep_max == 0 || n_lab == 0 || (H_rep && rows_rep > 0 && idx_a && idx_b),
             "H_rep, rows_rep > 0, idx_a and idx_b are needed when n_rep_max > 0");
  HG_REQUIRE(((uintptr_t)H & 15) == 0 && ((uintptr_t)H_rep & 15) == 0, "H and H_rep must be 16-byte aligned");
  HeadLayout L;
  carve_head(saved, scratch, rows, n_lab, params->d, params->dtype, &L, nullptr, nullptr);
  const HeadIn in{params, H, rows, H_rep, rows_rep, idx_a, idx_b, n_lab > 0 ? n_rep_max : 0, n_rep_dev, lab_idx, lab_y,
                  n_lab};
  return head_loss_dispatch(in, cca_loss, lambda_cca, loss_out, logits, L, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" hg_status hg_head_bwd(const hg_head_params* params, const int32_t* lab_idx, int64_t n_lab, float dloss,
                                const void* saved, void* dH, int64_t rows, void* dH_rep, int64_t rows_rep,
                                int32_t overwrite, const hg_head_grads* grads, void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_head_params(params));
  HG_REQUIRE(saved && scratch && grads, "saved, scratch and grads must be non-null");
  HG_REQUIRE(grads->dW1 && grads->db1 && grads->dw2 && grads->db2, "every gradient pointer must be non-null");
  HG_REQUIRE(((uintptr_t)saved & 255) == 0 && ((uintptr_t)scratch & 255) == 0, "buffers must be 256-byte aligned");
  HG_REQUIRE(n_lab >= 0 && n_lab < (int64_t(1) << 31), "n_lab must be in [0, 2^31)");
  HG_REQUIRE(n_lab == 0 || lab_idx, "lab_idx is needed when n_lab > 0");
  HG_REQUIRE(((uintptr_t)dH & 15) == 0 && ((uintptr_t)dH_rep & 15) == 0, "dH and dH_rep must be 16-byte aligned");
  HG_REQUIRE(rows >= 0 && rows_rep >= 0, "rows and rows_rep must be >= 0");
  HeadLayout L;
  carve_head(const_cast<void*>(saved), scratch, 0, n_lab, params->d, params->dtype, &L, nullptr, nullptr);
  if (overwrite) {
    const size_t row_bytes = (size_t)params->d * (params->dtype == HG_BF16 ? 2 : 4);
    cudaStream_t s0 = reinterpret_cast<cudaStream_t>(stream);
    if (dH && rows > 0) HG_CUDA(cudaMemsetAsync(dH, 0, (size_t)rows * row_bytes, s0));
    if (dH_rep && rows_rep > 0) HG_CUDA(cudaMemsetAsync(dH_rep, 0, (size_t)rows_rep * row_bytes, s0));
  }
  return head_bwd_dispatch(params, lab_idx, n_lab, 0, dloss, L, dH, dH_rep, grads,
                           reinterpret_cast<cudaStream_t>(stream));
}
