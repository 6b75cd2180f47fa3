// Temporal module (Section 3.2, Eq. 12-13): attention over each node's last w states and the GRU
// cell, forward and backward.
//
//   Eq. 12   u_k = tanh(c_k W_a), e_k = r . u_k, a = softmax_k(e), H~ = sum_k a_k c_k
//            (W_a = Q^T; c_k = the node's state k snapshots back, rows of the context C)
//   Eq. 13   r = sigmoid(x W_ir + b_ir + H~ W_hr + b_hr), z = sigmoid(x W_iz + b_iz + H~ W_hz + b_hz)
//            n = tanh(x W_in + b_in + r * (H~ W_hn + b_hn)),  H^t = (1 - z) n + z H~
// with x = h^t, the spatial embedding.  The context is an input of the step (earlier snapshots'
// outputs): no gradient flows into it.  H~ is rounded to the storage type (the tensor the GRU's
// products read).  The forward saves H~ and the attention weights a; the backward recomputes
// the rest.
//
// This file holds the CUDA-core path (fp32 storage; bf16 at d = 256 or with (w + 1) d > 512): row-tile
// GEMMs on CUDA cores into fp32 scratch and fused elementwise kernels.  bf16 at d <= 128 runs the
// tensor-core kernels of temporal_tc.cu.
#include <cuda_bf16.h>

#include <algorithm>

#include "hg_internal.cuh"
#include "layer_kernels.cuh"
#include "simt_tile.cuh"
#include "temporal_kernels.cuh"

namespace hg {

namespace {

// out[rows][ocol0 + 0..D) (+)= A[rows][0..K) . B[0..K)[bcol0 + 0..D)  (fp32 out, row stride ldo).
// A: row-major, row stride lda (type TA); B: row-major, row stride ldb (type TB).  One block per 64
// rows; K a multiple of 32.
// blockIdx.y selects the column block: B columns bcol0 + y D, output columns ocol0 + y D.
template <typename TA, typename TB, int D>
__global__ void __launch_bounds__(256) tgemm_simt(const TA* __restrict__ A, int64_t lda, const TB* __restrict__ B,
                                                  int64_t ldb, int bcol0, int K, int64_t n, float* __restrict__ out,
                                                  int64_t ldo, int ocol0, int accumulate) {
  bcol0 += blockIdx.y * D;
  ocol0 += blockIdx.y * D;
  using Tl = Tile<float, D>;
  constexpr int CN = Tl::CN, RM = Tl::RM;
  __shared__ __align__(16) float As[kBM][kAPad];
  extern __shared__ __align__(16) float Bs[];  // [kKC][D]
  const int64_t r0 = (int64_t)blockIdx.x * kBM;
  float acc[RM][CN];
#pragma unroll
  for (int i = 0; i < RM; ++i)
#pragma unroll
    for (int j = 0; j < CN; ++j) acc[i][j] = 0.f;
  for (int k0 = 0; k0 < K; k0 += kKC) {
    for (int idx = threadIdx.x; idx < kBM * kKC; idx += blockDim.x) {
      const int m = idx / kKC, k = idx % kKC;
      As[m][k] = r0 + m < n ? to_f32(A[(r0 + m) * lda + k0 + k]) : 0.f;
    }
    for (int idx = threadIdx.x; idx < kKC * D; idx += blockDim.x) {
      const int k = idx / D, c = idx % D;
      Bs[k * D + c] = to_f32(B[(int64_t)(k0 + k) * ldb + bcol0 + c]);
    }
    __syncthreads();
    mma_chunk<D, RM, CN>(&As[0][0], kAPad, 0, Bs, acc);
    __syncthreads();
  }
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int64_t r = r0 + ty * RM + i;
    if (r >= n) continue;
    float* o = out + r * ldo + ocol0 + tx * CN;
#pragma unroll
    for (int j = 0; j < CN; ++j) o[j] = accumulate ? o[j] + acc[i][j] : acc[i][j];
  }
}

__device__ __forceinline__ float sigm(float x) {
  const float e = expf(-fabsf(x));
  return x >= 0.f ? 1.f / (1.f + e) : e / (1.f + e);
}

// Eq. 12 per node from U (fp32, w blocks of n x D): a (saved), H~ (storage type).  One warp per node.
template <typename T, int D>
__global__ void temporal_attn_simt(const float* __restrict__ U, const T* __restrict__ C, const T* __restrict__ rvec,
                                   int64_t n, int w, T* __restrict__ Ht, float* __restrict__ a_out) {
  const int lane = threadIdx.x & 31;
  const int64_t v = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (v >= n) return;
  float e[kTemporalMaxW];
  float m = -INFINITY;
  for (int k = 0; k < w; ++k) {
    float s = 0.f;
    for (int c = lane; c < D; c += 32) s = fmaf(to_f32(rvec[c]), tanhf(U[((int64_t)k * n + v) * D + c]), s);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
    e[k] = s;
    m = fmaxf(m, s);
  }
  float sum = 0.f;
  for (int k = 0; k < w; ++k) {
    e[k] = expf(e[k] - m);
    sum += e[k];
  }
  for (int k = 0; k < w; ++k) e[k] /= sum;
  for (int c = lane; c < D; c += 32) {
    float h = 0.f;
    for (int k = 0; k < w; ++k) h = fmaf(e[k], to_f32(C[((int64_t)k * n + v) * D + c]), h);
    Ht[v * D + c] = from_f32<T>(h);
  }
  if (lane < w) {
    float ak = 0.f;
    for (int k = 0; k < w; ++k)
      if (k == lane) ak = e[k];
    a_out[v * w + lane] = ak;
  }
}

// Eq. 13 per element from Gi = x W_i, Gh = H~ W_h (fp32, n x 3D).
template <typename T, int D>
__global__ void temporal_gru_simt(const float* __restrict__ Gi, const float* __restrict__ Gh, const T* __restrict__ Ht,
                                  const T* __restrict__ b_i, const T* __restrict__ b_h, int64_t n, T* __restrict__ out) {
  const int64_t total = n * D;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < total; q += (int64_t)gridDim.x * blockDim.x) {
    const int64_t v = q / D;
    const int c = (int)(q % D);
    const float* gi = Gi + v * 3 * D;
    const float* gh = Gh + v * 3 * D;
    const float r = sigm(gi[c] + to_f32(b_i[c]) + gh[c] + to_f32(b_h[c]));
    const float z = sigm(gi[D + c] + to_f32(b_i[D + c]) + gh[D + c] + to_f32(b_h[D + c]));
    const float hn = gh[2 * D + c] + to_f32(b_h[2 * D + c]);
    const float nn = tanhf(gi[2 * D + c] + to_f32(b_i[2 * D + c]) + r * hn);
    const float h = to_f32(Ht[q]);
    out[q] = from_f32<T>((1.f - z) * nn + z * h);
  }
}

// Backward of Eq. 13 per element: dG_i = [dpre_r | dpre_z | dpre_n] and dG_h = [dpre_r | dpre_z | dhn]
// as gate-major arrays of n x D (storage type), and dh = dOut * z (fp32).
template <typename T, int D>
__global__ void temporal_gru_bwd_simt(const float* __restrict__ Gi, const float* __restrict__ Gh,
                                      const T* __restrict__ Ht, const T* __restrict__ b_i, const T* __restrict__ b_h,
                                      const T* __restrict__ dOut, int64_t n, T* __restrict__ dgi,
                                      T* __restrict__ dgh_n, float* __restrict__ dh) {
  const int64_t total = n * D;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < total; q += (int64_t)gridDim.x * blockDim.x) {
    const int64_t v = q / D;
    const int c = (int)(q % D);
    const float* gi = Gi + v * 3 * D;
    const float* gh = Gh + v * 3 * D;
    const float r = sigm(gi[c] + to_f32(b_i[c]) + gh[c] + to_f32(b_h[c]));
    const float z = sigm(gi[D + c] + to_f32(b_i[D + c]) + gh[D + c] + to_f32(b_h[D + c]));
    const float hn = gh[2 * D + c] + to_f32(b_h[2 * D + c]);
    const float nn = tanhf(gi[2 * D + c] + to_f32(b_i[2 * D + c]) + r * hn);
    const float h = to_f32(Ht[q]);
    const float g = to_f32(dOut[q]);
    const float dn = g * (1.f - z);
    const float dz = g * (h - nn);
    const float dpn = dn * (1.f - nn * nn);
    const float dpr = dpn * hn * r * (1.f - r);
    const float dpz = dz * z * (1.f - z);
    dgi[q] = from_f32<T>(dpr);
    dgi[total + q] = from_f32<T>(dpz);
    dgi[2 * total + q] = from_f32<T>(dpn);
    dgh_n[q] = from_f32<T>(dpn * r);
    dh[q] = g * z;
  }
}

// Backward of Eq. 12 per node (one warp): da_k = <dH~, c_k>, de = a (da - sum a da), and
// dpre_u_k = de_k r (1 - u_k^2) into dpre (storage type, w blocks of n x D); dr column partials
// de_k u_k accumulated per block (fixed order: lanes own columns, nodes in order).
template <typename T, int D>
__global__ void __launch_bounds__(256) temporal_attn_bwd_simt(const float* __restrict__ U, const T* __restrict__ C,
                                                              const T* __restrict__ rvec, const float* __restrict__ a_in,
                                                              const float* __restrict__ dHt, int64_t n, int w,
                                                              int64_t nodes_per_block, T* __restrict__ dpre,
                                                              float* __restrict__ dr_part) {
  constexpr int PL = D / 32;
  __shared__ float red[8][D];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float drl[PL];
#pragma unroll
  for (int i = 0; i < PL; ++i) drl[i] = 0.f;
  const int64_t v0 = (int64_t)blockIdx.x * nodes_per_block;
  const int64_t v1 = min(n, v0 + nodes_per_block);
  for (int64_t v = v0 + warp; v < v1; v += 8) {
    float da[kTemporalMaxW];
    float s = 0.f;
    for (int k = 0; k < w; ++k) {
      float p = 0.f;
#pragma unroll
      for (int i = 0; i < PL; ++i) {
        const int c = lane + 32 * i;
        p = fmaf(dHt[v * D + c], to_f32(C[((int64_t)k * n + v) * D + c]), p);
      }
#pragma unroll
      for (int o = 16; o > 0; o >>= 1) p += __shfl_xor_sync(0xffffffffu, p, o);
      da[k] = p;
      s = fmaf(a_in[v * w + k], p, s);
    }
    for (int k = 0; k < w; ++k) {
      const float de = a_in[v * w + k] * (da[k] - s);
#pragma unroll
      for (int i = 0; i < PL; ++i) {
        const int c = lane + 32 * i;
        const float u = tanhf(U[((int64_t)k * n + v) * D + c]);
        drl[i] = fmaf(de, u, drl[i]);
        dpre[((int64_t)k * n + v) * D + c] = from_f32<T>(de * to_f32(rvec[c]) * (1.f - u * u));
      }
    }
  }
#pragma unroll
  for (int i = 0; i < PL; ++i) red[warp][lane + 32 * i] = drl[i];
  __syncthreads();
  for (int c = threadIdx.x; c < D; c += blockDim.x) {
    float t = 0.f;
    for (int q = 0; q < 8; ++q) t += red[q][c];
    dr_part[(int64_t)blockIdx.x * D + c] = t;
  }
}

// part[block][c] = sum over the block's rows of X[row][c] (rows in order), for G column blocks of
// n x D arrays X_g (gate-major), written at part[block][g D + c].
template <typename T, int D>
__global__ void temporal_colsum(const T* __restrict__ X0, const T* __restrict__ X1, const T* __restrict__ X2,
                                int64_t n, int64_t rows_per_block, float* __restrict__ part) {
  const T* Xs[3] = {X0, X1, X2};
  const int64_t r0 = (int64_t)blockIdx.x * rows_per_block, r1 = min(n, r0 + rows_per_block);
  for (int q = threadIdx.x; q < 3 * D; q += blockDim.x) {
    const T* X = Xs[q / D];
    const int c = q % D;
    float s = 0.f;
    for (int64_t r = r0; r < r1; ++r) s += to_f32(X[r * D + c]);
    part[(int64_t)blockIdx.x * 3 * D + q] = s;
  }
}

// out[i][j] = W[j][i] for a rows x cols matrix W (storage type).
template <typename T>
__global__ void temporal_transpose(const T* __restrict__ W, int rows, int cols, T* __restrict__ out) {
  for (int q = blockIdx.x * blockDim.x + threadIdx.x; q < rows * cols; q += gridDim.x * blockDim.x) {
    const int i = q / rows, j = q % rows;
    out[q] = W[(int64_t)j * cols + i];
  }
}

// dst[row][g D + c] = scale * G[row][c] (a d x d block into a d x 3d gradient).
__global__ void temporal_place(const float* __restrict__ G, int d, int g, float* __restrict__ dst) {
  for (int q = blockIdx.x * blockDim.x + threadIdx.x; q < d * d; q += gridDim.x * blockDim.x) {
    const int row = q / d, c = q % d;
    dst[(int64_t)row * 3 * d + g * d + c] = G[q];
  }
}

template <typename T>
__global__ void temporal_to_storage(const float* __restrict__ x, int64_t count, T* __restrict__ out) {
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < count; q += (int64_t)gridDim.x * blockDim.x)
    out[q] = from_f32<T>(x[q]);
}

// ---------------------------------------------------------------------------------------------
// buffers
// ---------------------------------------------------------------------------------------------
inline int64_t tgrid(int64_t count, int threads = 256) {
  return std::max<int64_t>(1, std::min<int64_t>(ceil_div(count, threads), 152 * 16));
}
constexpr int64_t kColsumRows = 2048;  // rows per block of the bias sums
constexpr int64_t kAttnBwdNodes = 512;  // nodes per block of the attention backward

}  // namespace

struct TemporalLayout {
  // saved
  void* Ht;
  float* a;
  // scratch
  float* U;      // w n x d
  float* Gi;     // n x 3d
  float* Gh;     // n x 3d
  void* dgi;     // 3 x n x d (storage type)
  void* dghn;    // n x d
  float* dh;     // n x d
  float* dXf;    // n x d
  void* WiT;     // 3d x d
  void* WhT;     // 3d x d
  void* dpre;    // w n x d
  float* part;   // partial sums
  float* G;      // d x d (3 d x d on the tensor-core path)
  float* tmp;
  // tensor-core path
  void* dG;      // 4 x n x d bf16
  void* dhb;     // n x d bf16
  void* dHtb;    // n x d bf16
  float* sums;   // 4 d
};

int64_t temporal_part_floats(int64_t n, int d, int w) {
  const int64_t wsplit = (int64_t)wgrad_splits(std::max<int64_t>(n, 1) * std::max(w, 1)) * d * d;
  const int64_t cs = ceil_div(std::max<int64_t>(n, 1), kColsumRows) * 3 * d;
  const int64_t ab = ceil_div(std::max<int64_t>(n, 1), kAttnBwdNodes) * d;
  return std::max(wsplit, std::max(cs, ab));
}

void carve_temporal(void* saved, void* scratch, int64_t n, int d, int w, hg_dtype dt, TemporalLayout* L,
                    size_t* saved_bytes, size_t* scratch_bytes) {
  const size_t esz = dt == HG_BF16 ? 2 : 4;
  const size_t nd = (size_t)std::max<int64_t>(n, 1) * d;
  Carve s(saved);
  L->Ht = s.take<char>(nd * esz);
  L->a = s.take<float>((size_t)std::max<int64_t>(n, 1) * w);
  Carve k(scratch);
  if (temporal_tc_supported(dt, d, w)) {
    L->dG = k.take<char>(nd * 4 * esz);
    L->dhb = k.take<char>(nd * esz);
    L->dHtb = k.take<char>(nd * esz);
    L->part = k.take<float>(temporal_tc_part_floats(n, d));
    L->sums = k.take<float>((size_t)4 * d);
    L->G = k.take<float>((size_t)3 * d * d);
    L->tmp = k.take<float>(reduce_tmp_floats(1, (int64_t)d * d) + 4 * (size_t)d);
    if (saved_bytes) *saved_bytes = s.used;
    if (scratch_bytes) *scratch_bytes = k.used;
    return;
  }
  L->U = k.take<float>(nd * w);
  L->Gi = k.take<float>(nd * 3);
  L->Gh = k.take<float>(nd * 3);
  L->dgi = k.take<char>(nd * 3 * esz);
  L->dghn = k.take<char>(nd * esz);
  L->dh = k.take<float>(nd);
  L->dXf = k.take<float>(nd);
  L->WiT = k.take<char>((size_t)3 * d * d * esz);
  L->WhT = k.take<char>((size_t)3 * d * d * esz);
  L->dpre = k.take<char>(nd * w * esz);
  L->part = k.take<float>((size_t)temporal_part_floats(n, d, w));
  L->G = k.take<float>((size_t)d * d);
  L->tmp = k.take<float>(reduce_tmp_floats(1, (int64_t)d * d) + 3 * (size_t)d);
  if (saved_bytes) *saved_bytes = s.used;
  if (scratch_bytes) *scratch_bytes = k.used;
}

namespace {

template <typename TA, typename TB, int D>
hg_status gemm(const void* A, int64_t lda, const void* B, int64_t ldb, int bcol0, int K, int64_t n, float* out,
               int64_t ldo, int ocol0, int accumulate, int col_blocks, cudaStream_t s) {
  static bool done = false;
  if (!done) {
    HG_CUDA(cudaFuncSetAttribute(tgemm_simt<TA, TB, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)(sizeof(float) * kKC * D)));
    done = true;
  }
  return launch("temporal_gemm_simt", tgemm_simt<TA, TB, D>, dim3((unsigned)ceil_div(n, kBM), col_blocks), dim3(256),
                sizeof(float) * kKC * D, s, (const TA*)A, lda, (const TB*)B, ldb, bcol0, K, n, out, ldo, ocol0,
                accumulate);
}

template <typename T, int D>
hg_status fwd_simt(const hg_temporal_params* p, const void* X, const void* C, int64_t n, void* H_out,
                   const TemporalLayout& L, cudaStream_t s) {
  const int w = p->w;
  HG_TRY((gemm<T, T, D>(C, D, p->Wa, D, 0, D, w * n, L.U, D, 0, 0, 1, s)));
  HG_TRY(launch("temporal_attn_simt", temporal_attn_simt<T, D>, dim3((unsigned)ceil_div(n * 32, 256)), dim3(256), 0, s,
                (const float*)L.U, (const T*)C, (const T*)p->r, n, w, (T*)L.Ht, L.a));
  HG_TRY((gemm<T, T, D>(X, D, p->W_i, 3 * D, 0, D, n, L.Gi, 3 * D, 0, 0, 3, s)));
  HG_TRY((gemm<T, T, D>(L.Ht, D, p->W_h, 3 * D, 0, D, n, L.Gh, 3 * D, 0, 0, 3, s)));
  return launch("temporal_gru_simt", temporal_gru_simt<T, D>, dim3((unsigned)tgrid(n * D)), dim3(256), 0, s,
                (const float*)L.Gi, (const float*)L.Gh, (const T*)L.Ht, (const T*)p->b_i, (const T*)p->b_h, n,
                (T*)H_out);
}

template <typename T, int D>
hg_status bwd_simt(const hg_temporal_params* p, const void* X, const void* C, int64_t n, const void* dOut, void* dX,
                   const hg_temporal_grads* g, const TemporalLayout& L, cudaStream_t s) {
  constexpr hg_dtype kDt = sizeof(T) == 2 ? HG_BF16 : HG_F32;
  const int w = p->w;
  const int64_t nd = n * D;
  const T* dgi = (const T*)L.dgi;
  // recompute the gate products, then the elementwise backward of Eq. 13
  HG_TRY((gemm<T, T, D>(X, D, p->W_i, 3 * D, 0, D, n, L.Gi, 3 * D, 0, 0, 3, s)));
  HG_TRY((gemm<T, T, D>(L.Ht, D, p->W_h, 3 * D, 0, D, n, L.Gh, 3 * D, 0, 0, 3, s)));
  HG_TRY(launch("temporal_gru_bwd_simt", temporal_gru_bwd_simt<T, D>, dim3((unsigned)tgrid(nd)), dim3(256), 0, s,
                (const float*)L.Gi, (const float*)L.Gh, (const T*)L.Ht, (const T*)p->b_i, (const T*)p->b_h,
                (const T*)dOut, n, (T*)L.dgi, (T*)L.dghn, L.dh));
  // dX = dG_i W_i^T and dH~ = dh + dG_h W_h^T (K = 3d as three d-wide products, in gate order)
  HG_TRY(launch("temporal_transpose", temporal_transpose<T>, dim3((unsigned)tgrid(3 * D * D)), dim3(256), 0, s,
                (const T*)p->W_i, D, 3 * D, (T*)L.WiT));
  HG_TRY(launch("temporal_transpose", temporal_transpose<T>, dim3((unsigned)tgrid(3 * D * D)), dim3(256), 0, s,
                (const T*)p->W_h, D, 3 * D, (T*)L.WhT));
  for (int q = 0; q < 3; ++q)
    HG_TRY((gemm<T, T, D>(dgi + q * nd, D, (const T*)L.WiT + (int64_t)q * D * D, D, 0, D, n, L.dXf, D, 0, q > 0, 1,
                          s)));
  const T* dgh[3] = {dgi, dgi + nd, (const T*)L.dghn};
  for (int q = 0; q < 3; ++q)
    HG_TRY((gemm<T, T, D>(dgh[q], D, (const T*)L.WhT + (int64_t)q * D * D, D, 0, D, n, L.dh, D, 0, 1, 1, s)));
  HG_TRY(launch("temporal_to_storage", temporal_to_storage<T>, dim3((unsigned)tgrid(nd)), dim3(256), 0, s,
                (const float*)L.dXf, nd, (T*)dX));
  // backward of Eq. 12 (U recomputed), dr and dW_a
  HG_TRY((gemm<T, T, D>(C, D, p->Wa, D, 0, D, w * n, L.U, D, 0, 0, 1, s)));
  const int ab = (int)ceil_div(n, kAttnBwdNodes);
  HG_TRY(launch("temporal_attn_bwd_simt", temporal_attn_bwd_simt<T, D>, dim3(ab), dim3(256), 0, s, (const float*)L.U,
                (const T*)C, (const T*)p->r, (const float*)L.a, (const float*)L.dh, n, w, kAttnBwdNodes, (T*)L.dpre,
                L.part));
  HG_TRY(reduce_partials(L.part, D, ab, D, g->dr, L.tmp, s));
  HG_TRY(weight_grad(kDt, D, C, 0, L.dpre, 0, w * n, L.part, g->dWa, L.tmp, s));
  // dW_i = x^T dG_i, dW_h = H~^T dG_h (one d x d block per gate)
  for (int q = 0; q < 3; ++q) {
    HG_TRY(weight_grad(kDt, D, X, 0, dgi + q * nd, 0, n, L.part, L.G, L.tmp, s));
    HG_TRY(launch("temporal_place", temporal_place, dim3((unsigned)tgrid(D * D)), dim3(256), 0, s, (const float*)L.G,
                  D, q, g->dW_i));
    HG_TRY(weight_grad(kDt, D, L.Ht, 0, dgh[q], 0, n, L.part, L.G, L.tmp, s));
    HG_TRY(launch("temporal_place", temporal_place, dim3((unsigned)tgrid(D * D)), dim3(256), 0, s, (const float*)L.G,
                  D, q, g->dW_h));
  }
  // bias gradients: column sums in row order, then the blocks in order
  const int cb = (int)ceil_div(n, kColsumRows);
  HG_TRY(launch("temporal_colsum", temporal_colsum<T, D>, dim3(cb), dim3(256), 0, s, dgi, dgi + nd, dgi + 2 * nd, n,
                kColsumRows, L.part));
  HG_TRY(reduce_partials(L.part, 3 * D, cb, 3 * D, g->db_i, L.tmp, s));
  HG_TRY(launch("temporal_colsum", temporal_colsum<T, D>, dim3(cb), dim3(256), 0, s, dgi, dgi + nd, (const T*)L.dghn,
                n, kColsumRows, L.part));
  return reduce_partials(L.part, 3 * D, cb, 3 * D, g->db_h, L.tmp, s);
}

}  // namespace
}  // namespace hg

namespace hg {
namespace {

#define HG_TEMPORAL_DISPATCH(dtype, d, FN, ...)                                             \
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

hg_status check_temporal(const hg_temporal_params* p, int64_t n) {
  HG_REQUIRE(p != nullptr, "params must be non-null");
  if (!(p->d == 64 || p->d == 128 || p->d == 256) || !(p->dtype == HG_F32 || p->dtype == HG_BF16)) {
    set_error("unsupported d=%d / dtype=%d", p->d, (int)p->dtype);
    return HG_ERR_UNSUPPORTED;
  }
  HG_REQUIRE(p->w >= 1 && p->w <= kTemporalMaxW, "w must be in [1, %d]", kTemporalMaxW);
  HG_REQUIRE(p->Wa && p->r && p->W_i && p->W_h && p->b_i && p->b_h, "every parameter pointer must be non-null");
  HG_REQUIRE(n >= 0 && n * p->w < (int64_t(1) << 31), "n * w must be in [0, 2^31)");
  return HG_OK;
}

}  // namespace
}  // namespace hg

using namespace hg;

extern "C" hg_status hg_temporal_workspace_size(int64_t n, int32_t d, int32_t w, hg_dtype dtype, size_t* saved_bytes,
                                               size_t* scratch_bytes) {
  clear_error();
  HG_REQUIRE(saved_bytes && scratch_bytes, "saved_bytes and scratch_bytes must be non-null");
  HG_REQUIRE(n >= 0 && w >= 1 && w <= kTemporalMaxW && n * w < (int64_t(1) << 31), "bad n or w");
  if (!(d == 64 || d == 128 || d == 256) || !(dtype == HG_F32 || dtype == HG_BF16)) {
    set_error("unsupported d=%d / dtype=%d", d, (int)dtype);
    return HG_ERR_UNSUPPORTED;
  }
  TemporalLayout L;
  carve_temporal(nullptr, nullptr, n, d, w, dtype, &L, saved_bytes, scratch_bytes);
  return HG_OK;
}

extern "C" hg_status hg_temporal_fwd(const hg_temporal_params* params, const void* X, const void* C, int64_t n,
                                    void* H_out, void* saved, void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_temporal(params, n));
  HG_REQUIRE(saved && scratch, "saved and scratch must be non-null");
  HG_REQUIRE(((uintptr_t)saved & 255) == 0 && ((uintptr_t)scratch & 255) == 0, "buffers must be 256-byte aligned");
  HG_REQUIRE(n == 0 || (X && C && H_out), "X, C and H_out must be non-null");
  if (n == 0) return HG_OK;
  TemporalLayout L;
  carve_temporal(saved, scratch, n, params->d, params->w, params->dtype, &L, nullptr, nullptr);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (temporal_tc_supported(params->dtype, params->d, params->w)) {
    const TemporalTcIn in{params, X, C, n, L.Ht, L.a};
    return temporal_fwd_tc(in, H_out, s);
  }
  HG_TEMPORAL_DISPATCH(params->dtype, params->d, fwd_simt, params, X, C, n, H_out, L, s);
}

extern "C" hg_status hg_temporal_bwd(const hg_temporal_params* params, const void* X, const void* C, int64_t n,
                                    const void* saved, const void* dH_out, void* dX, const hg_temporal_grads* grads,
                                    void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_temporal(params, n));
  HG_REQUIRE(saved && scratch && grads, "saved, scratch and grads must be non-null");
  HG_REQUIRE(grads->dWa && grads->dr && grads->dW_i && grads->dW_h && grads->db_i && grads->db_h,
             "every gradient pointer must be non-null");
  HG_REQUIRE(((uintptr_t)saved & 255) == 0 && ((uintptr_t)scratch & 255) == 0, "buffers must be 256-byte aligned");
  HG_REQUIRE(n == 0 || (X && C && dH_out && dX), "X, C, dH_out and dX must be non-null");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int d = params->d;
  if (n == 0) {
    HG_CUDA(cudaMemsetAsync(grads->dWa, 0, sizeof(float) * d * d, s));
    HG_CUDA(cudaMemsetAsync(grads->dr, 0, sizeof(float) * d, s));
    HG_CUDA(cudaMemsetAsync(grads->dW_i, 0, sizeof(float) * 3 * d * d, s));
    HG_CUDA(cudaMemsetAsync(grads->dW_h, 0, sizeof(float) * 3 * d * d, s));
    HG_CUDA(cudaMemsetAsync(grads->db_i, 0, sizeof(float) * 3 * d, s));
    HG_CUDA(cudaMemsetAsync(grads->db_h, 0, sizeof(float) * 3 * d, s));
    return HG_OK;
  }
  TemporalLayout L;
  carve_temporal(const_cast<void*>(saved), scratch, n, d, params->w, params->dtype, &L, nullptr, nullptr);
  if (temporal_tc_supported(params->dtype, d, params->w)) {
    const TemporalTcIn in{params, X, C, n, L.Ht, L.a};
    const TemporalTcScratch sc{L.dG, L.dhb, L.dHtb, L.part, L.sums, L.G, L.tmp};
    return temporal_bwd_tc(in, dH_out, dX, grads, sc, s);
  }
  HG_TEMPORAL_DISPATCH(params->dtype, d, bwd_simt, params, X, C, n, dH_out, dX, grads, L, s);
}
