// Attention layer (Heterogeneous Graph Transformer, Section 3.2, Eq. 6-11), forward and backward.
//
// With S heads of width d_h and c_r = mu[r] / sqrt(d_h), the layer is computed as
//   K, V = H W_K + b_K, H W_V + b_V (per source type; one N x 2d array, a node's K then V)
//   Q       = H W_Q + b_Q (per target type)
//   Q'_r(j) = c_r Q_j blockdiag(W_att[r])^T   (one row per (relation, target): the CSR row layout
//             of the mean layer; c_r applied in fp32)    so that score^s(e) = K^s(i) . Q'^s_r(j)
//   alpha   = softmax over every in-edge of j, per head (online: running maximum and sum)
//   S_r(j)  = sum over the r-edges into j of alpha V(i)    (per head; CSR row layout)
//   U       = sum_r S_r blockdiag(W_msg[r]) W_agg + b_agg, then activation, residual, LayerNorm:
//             the mean layer's projection with W_rel = blockdiag(W_msg[r]).
// Every product has a stored bf16 weight as one factor (W_K, W_Q, W_V, blockdiag(W_att[r]),
// blockdiag(W_msg[r]) paired with W_agg as the projection's hi / lo fused weights), so no product
// of two weights is ever rounded to bf16; the scalar c_r multiplies in the fp32 epilogue.
// The backward reuses that projection's backward (without the 1/deg scaling) for dS_r, then
//   target pass  D^s_j = sum_r <dS_r(j), S_r(j)>^s, de = alpha (<dS_r(j), V(i)>^s - D^s_j),
//                dQ'_r(j) = sum de K(i)
//   source pass  dK(i) = sum over out-edges de Q'_r(j), dV(i) = sum alpha dS_r(j)
//   and the dense products back to H (dQ = sum_r c_r dQ'_r blockdiag(W_att[r]), then dQ W_Q^T) and
//   to the weights.
// Edge work is warp per row (a lane holds d / 32 consecutive features, the 32 / S lanes of a head
// reduce by shuffles); rows above the hub degree are split into chunks whose partial results are
// merged in chunk order, so every reduction has a fixed order (deterministic, atomic-free).  The
// dense row products run on the tensor cores for bf16 (rows_gemm_tc.cu) and on CUDA cores for fp32.
#include <cuda_bf16.h>

#include <algorithm>

#include "hg_internal.cuh"
#include "layer_kernels.cuh"
#include "simt_tile.cuh"

namespace hg {

namespace {

// ---------------------------------------------------------------------------------------------
// per-lane slices: lane l owns features [l E, (l + 1) E), E = D / 32
// ---------------------------------------------------------------------------------------------
template <typename T, int E>
__device__ __forceinline__ void load_slice(const T* __restrict__ p, float (&f)[E]) {
  if constexpr (sizeof(T) == 4) {
    if constexpr (E == 2) {
      const float2 v = __ldg(reinterpret_cast<const float2*>(p));
      f[0] = v.x;
      f[1] = v.y;
    } else {
#pragma unroll
      for (int e = 0; e < E; e += 4) {
        const float4 v = __ldg(reinterpret_cast<const float4*>(p + e));
        f[e] = v.x;
        f[e + 1] = v.y;
        f[e + 2] = v.z;
        f[e + 3] = v.w;
      }
    }
  } else {
    if constexpr (E == 2) {
      const uint32_t u = __ldg(reinterpret_cast<const unsigned int*>(p));
      f[0] = __uint_as_float(u << 16);
      f[1] = __uint_as_float(u & 0xFFFF0000u);
    } else if constexpr (E == 4) {
      const uint2 u = __ldg(reinterpret_cast<const uint2*>(p));
      f[0] = __uint_as_float(u.x << 16);
      f[1] = __uint_as_float(u.x & 0xFFFF0000u);
      f[2] = __uint_as_float(u.y << 16);
      f[3] = __uint_as_float(u.y & 0xFFFF0000u);
    } else {
      unpack(ldg16(p), f, __nv_bfloat16());
    }
  }
}

template <typename T, int E>
__device__ __forceinline__ void store_slice(T* __restrict__ p, const float (&f)[E]) {
#pragma unroll
  for (int e = 0; e < E; ++e) p[e] = from_f32<T>(f[e]);
}

// Sum over the lanes of this lane's head (lpw = 32 / S consecutive lanes).
__device__ __forceinline__ float head_sum(float x, int lph) {
  for (int o = 1; o < lph; o <<= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

// ---------------------------------------------------------------------------------------------
// block-diagonal expansion of per-head weights (exact copies, no arithmetic)
// ---------------------------------------------------------------------------------------------
// out[r] = blockdiag(W[r]) (d x d, S blocks of d_h x d_h), or its transpose when transpose != 0.
template <typename T>
__global__ void hgt_blockdiag(const T* __restrict__ W, int R, int d, int S, int transpose, T* __restrict__ out) {
  const int dh = d / S;
  const int64_t total = (int64_t)R * d * d;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < total; q += (int64_t)gridDim.x * blockDim.x) {
    const int r = (int)(q / ((int64_t)d * d));
    int a = (int)((q / d) % d), b = (int)(q % d);
    if (transpose) {
      const int t = a;
      a = b;
      b = t;
    }
    const int s = a / dh;
    out[q] = b / dh == s ? W[((int64_t)r * S + s) * dh * dh + (a % dh) * dh + (b % dh)] : from_f32<T>(0.f);
  }
}

// out[i][j] = W[j][i] for one d x d matrix per block row.
template <typename T>
__global__ void hgt_transpose(const T* __restrict__ W, int count, int d, T* __restrict__ out) {
  const int64_t total = (int64_t)count * d * d;
  for (int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; q < total; q += (int64_t)gridDim.x * blockDim.x) {
    const int64_t m = q / ((int64_t)d * d);
    const int i = (int)((q / d) % d), j = (int)(q % d);
    out[q] = W[m * d * d + (int64_t)j * d + i];
  }
}

// ---------------------------------------------------------------------------------------------
// dense row products on CUDA cores: out[r][ocol0 + c] (=, or +=) scale sum_k A[r][k] B[k][c]
// (+ bias[c]), c < D, rows [0, n), K a multiple of 32; A row stride lda, out row stride ldo, B is
// K x D; scale = scale_mul * (*scale_ptr) (null scale_ptr: 1).
// ---------------------------------------------------------------------------------------------
template <typename T, int D>
__global__ void __launch_bounds__(256) hgt_gemm_simt(const T* __restrict__ A, int64_t lda, const T* __restrict__ B,
                                                     const T* __restrict__ bias, int K, int64_t n, T* __restrict__ out,
                                                     int64_t ldo, int ocol0, int accumulate,
                                                     const float* __restrict__ scale_ptr, float scale_mul) {
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
      Bs[k * D + c] = to_f32(B[(int64_t)(k0 + k) * D + c]);
    }
    __syncthreads();
    mma_chunk<D, RM, CN>(&As[0][0], kAPad, 0, Bs, acc);
    __syncthreads();
  }
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
  const float sc = scale_mul * (scale_ptr ? *scale_ptr : 1.f);
#pragma unroll
  for (int i = 0; i < RM; ++i) {
    const int64_t r = r0 + ty * RM + i;
    if (r >= n) continue;
    T* o = out + r * ldo + ocol0 + tx * CN;
#pragma unroll
    for (int j = 0; j < CN; ++j) {
      float v = sc * acc[i][j];
      if (bias) v += to_f32(bias[tx * CN + j]);
      if (accumulate) v += to_f32(o[j]);
      o[j] = from_f32<T>(v);
    }
  }
}

// part[block][c] = sum over the block's rows (in order) of X[row][c], rows [0, n), row stride ldx.
template <typename T>
__global__ void hgt_colsum(const T* __restrict__ X, int64_t ldx, int d, int64_t n, int64_t rows_per_block,
                           float* __restrict__ part) {
  const int64_t r0 = (int64_t)blockIdx.x * rows_per_block, r1 = min(n, r0 + rows_per_block);
  for (int c = threadIdx.x; c < d; c += blockDim.x) {
    float s = 0.f;
    for (int64_t r = r0; r < r1; ++r) s += to_f32(X[r * ldx + c]);
    part[(int64_t)blockIdx.x * d + c] = s;
  }
}

// ---------------------------------------------------------------------------------------------
// edge kernels
// ---------------------------------------------------------------------------------------------
struct HgtArgs {
  GraphMeta meta;
  int8_t rslot[kMaxTypes][kMaxRels];  // relations into each type in relation order, -1 past the last
  int64_t N, csr_rows;
  int S;
  // Edges as runs of parallel edges (column, multiplicity): a run's edges share their source, target
  // and relation, so their scores, weights and gradients are equal and the run is taken once times
  // its count.  Target side: each CSR row's runs by source (dptr / dcol / dcnt, hub chunks over
  // runs); source side: each node's out-runs (sptr / scol / scnt), scol naming the target's CSR row
  // through its compact index (the CSR row is mlist[scol]).
  const int32_t* dptr;
  const int32_t* dcol;
  const int32_t* dcnt;
  const int32_t* dchunk_ofs;
  const int32_t* dchunk_row;
  const int32_t* sptr;
  const int32_t* scol;
  const int32_t* scnt;
  const int32_t* schunk_ofs;
  const int32_t* schunk_row;
  const int32_t* mlist;
  const void* KV;    // N x 2d: K then V of each node
  const void* Qp;    // csr_rows x d: relation-scaled queries
  void* Srows;       // csr_rows x d: attention-weighted value sums (forward output, backward input)
  const void* dS;    // csr_rows x d
  float2* stats;     // N x S: running maximum and sum of each target's softmax
  float4* rstat;     // csr_rows x S: the target's (max, 1 / sum, D_j) on each of its rows, per head
  void* dQp;         // csr_rows x d
  void* dK;          // N x d
  void* dV;          // N x d
  float* part;       // chunk partials
};

constexpr int kBatch = 4;       // edges of a row in flight per warp (node kernels)
constexpr int kBatchChunk = 4;  // the same for the chunk kernels (eight was slower: registers)

// Online softmax step for one run of w parallel edges (per lane: its head's running maximum m and
// sum l; the value accumulators are rescaled when the maximum grows).
template <int E, int NACC>
__device__ __forceinline__ void online_step(float s, float w, const float (&v)[E], float& m, float& l,
                                            float (&acc)[NACC][E], int slot) {
  const float mn = fmaxf(m, s);
  if (mn > m) {
    const float so = expf(m - mn);
    l *= so;
#pragma unroll
    for (int k = 0; k < NACC; ++k)
#pragma unroll
      for (int e = 0; e < E; ++e) acc[k][e] *= so;
    m = mn;
  }
  const float p = w * expf(s - m);  // w edges with this score
  l += p;
#pragma unroll
  for (int k = 0; k < NACC; ++k)
    if (k == slot)
#pragma unroll
      for (int e = 0; e < E; ++e) acc[k][e] = fmaf(p, v[e], acc[k][e]);
}

// The edges [beg, end) of one CSR row against the query slice q, folded into (m, l, acc[slot]).
template <typename T, int D, int NACC, int NB = kBatch>
__device__ __forceinline__ void fwd_edges(const HgtArgs& a, int64_t beg, int64_t end, const float (&q)[D / 32], int lph,
                                          float& m, float& l, float (&acc)[NACC][D / 32], int slot) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31;
  const T* KV = (const T*)a.KV;
  for (int64_t e0 = beg; e0 < end; e0 += NB) {
    int src[NB];
    float w[NB];
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      src[u] = e0 + u < end ? __ldg(a.dcol + e0 + u) : -1;
      w[u] = e0 + u < end ? (float)__ldg(a.dcnt + e0 + u) : 0.f;
    }
    float k[NB][E], v[NB][E];
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      if (src[u] >= 0) {
        load_slice<T, E>(KV + (int64_t)src[u] * 2 * D + lane * E, k[u]);
        load_slice<T, E>(KV + (int64_t)src[u] * 2 * D + D + lane * E, v[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      if (src[u] < 0) break;
      float s = 0.f;
#pragma unroll
      for (int e = 0; e < E; ++e) s = fmaf(k[u][e], q[e], s);
      s = head_sum(s, lph);
      online_step<E, NACC>(s, w[u], v[u], m, l, acc, slot);
    }
  }
}

// One warp per chunk of a hub row: (m, l, unnormalised value sum) of the chunk's edges.
template <typename T, int D>
__global__ void __launch_bounds__(256) hgt_fwd_chunks(HgtArgs a) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, lph = 32 / a.S;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int nchunks = a.dchunk_ofs[a.csr_rows];
  const int stride = 2 * a.S + D;
  for (int64_t c = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; c < nchunks; c += nw) {
    const int row = a.dchunk_row[c];
    const int64_t beg = (int64_t)a.dptr[row] + (int64_t)(c - a.dchunk_ofs[row]) * kChunkEdges;
    const int64_t end = min((int64_t)a.dptr[row + 1], beg + kChunkEdges);
    float q[E];
    load_slice<T, E>((const T*)a.Qp + (int64_t)row * D + lane * E, q);
    float m = -INFINITY, l = 0.f, acc[1][E];
#pragma unroll
    for (int e = 0; e < E; ++e) acc[0][e] = 0.f;
    fwd_edges<T, D, 1, kBatchChunk>(a, beg, end, q, lph, m, l, acc, 0);
    float* p = a.part + c * stride;
    if (lane % lph == 0) {
      p[2 * (lane / lph)] = m;
      p[2 * (lane / lph) + 1] = l;
    }
#pragma unroll
    for (int e = 0; e < E; ++e) p[2 * a.S + lane * E + e] = acc[0][e];
  }
}

// One warp per node j: the softmax over all of j's in-edges (its rows of every relation into its
// type, hub rows through their chunk partials in order), S_r(j) = sum alpha V for each relation.
// The row bounds and query slices of all of j's rows are loaded before any edge.
template <typename T, int D, int KS>
__global__ void __launch_bounds__(256, (D <= 128 && KS <= 4) ? 3 : 1) hgt_fwd_nodes(HgtArgs a) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, lph = 32 / a.S;
  const int64_t j = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (j >= a.N) return;
  const int t = node_type_of(a.meta, j);
  const int64_t jl = j - a.meta.type_off[t];
  const int stride = 2 * a.S + D;
  int64_t row[KS];
  int c0[KS], c1[KS];
  int64_t e0[KS], e1[KS];
  float q[KS][E];
#pragma unroll
  for (int k = 0; k < KS; ++k) {
    const int r = a.rslot[t][k];
    row[k] = r >= 0 ? a.meta.row_base[r] + jl : -1;
    if (row[k] >= 0) {
      c0[k] = a.dchunk_ofs[row[k]];
      c1[k] = a.dchunk_ofs[row[k] + 1];
      e0[k] = a.dptr[row[k]];
      e1[k] = a.dptr[row[k] + 1];
      load_slice<T, E>((const T*)a.Qp + row[k] * D + lane * E, q[k]);
    }
  }
  float m = -INFINITY, l = 0.f, acc[KS][E];
#pragma unroll
  for (int k = 0; k < KS; ++k)
#pragma unroll
    for (int e = 0; e < E; ++e) acc[k][e] = 0.f;
#pragma unroll
  for (int k = 0; k < KS; ++k) {
    if (row[k] < 0) continue;
    if (c1[k] > c0[k]) {
      for (int c = c0[k]; c < c1[k]; ++c) {
        const float* p = a.part + (int64_t)c * stride;
        const float pm = p[2 * (lane / lph)], pl = p[2 * (lane / lph) + 1];
        const float mn = fmaxf(m, pm);
        if (mn > m) {
          const float so = expf(m - mn);
          l *= so;
#pragma unroll
          for (int kk = 0; kk < KS; ++kk)
#pragma unroll
            for (int e = 0; e < E; ++e) acc[kk][e] *= so;
          m = mn;
        }
        const float sp = expf(pm - m);
        l = fmaf(pl, sp, l);
#pragma unroll
        for (int e = 0; e < E; ++e) acc[k][e] = fmaf(sp, p[2 * a.S + lane * E + e], acc[k][e]);
      }
    } else {
      fwd_edges<T, D, KS>(a, e0[k], e1[k], q[k], lph, m, l, acc, k);
    }
  }
  const float inv = l > 0.f ? 1.f / l : 0.f;
#pragma unroll
  for (int k = 0; k < KS; ++k) {
    if (row[k] < 0) continue;
    float o[E];
#pragma unroll
    for (int e = 0; e < E; ++e) o[e] = acc[k][e] * inv;
    store_slice<T, E>((T*)a.Srows + row[k] * D + lane * E, o);
  }
  if (lane % lph == 0) a.stats[j * a.S + lane / lph] = make_float2(l > 0.f ? m : 0.f, l);
}

// D^s_j = sum over j's relation rows of <dS_r(j), S_r(j)> on head s, stored with the softmax statistics
// on every row of j (the source pass reads them by row).  One warp per node.
template <typename T, int D>
__global__ void __launch_bounds__(256) hgt_bwd_dstats(HgtArgs a) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, lph = 32 / a.S;
  const int64_t j = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (j >= a.N) return;
  const int t = node_type_of(a.meta, j);
  const int64_t jl = j - a.meta.type_off[t];
  float s = 0.f;
#pragma unroll
  for (int r = 0; r < kMaxRels; ++r) {
    if (r >= a.meta.num_rels || a.meta.rel_dst[r] != t) continue;
    const int64_t row = a.meta.row_base[r] + jl;
    float x[E], y[E];
    load_slice<T, E>((const T*)a.dS + row * D + lane * E, x);
    load_slice<T, E>((const T*)a.Srows + row * D + lane * E, y);
#pragma unroll
    for (int e = 0; e < E; ++e) s = fmaf(x[e], y[e], s);
  }
  s = head_sum(s, lph);
  if (lane % lph == 0) {
    const float2 st = a.stats[j * a.S + lane / lph];
    const float4 v = make_float4(st.x, st.y > 0.f ? 1.f / st.y : 0.f, s, 0.f);
#pragma unroll
    for (int r = 0; r < kMaxRels; ++r) {
      if (r >= a.meta.num_rels || a.meta.rel_dst[r] != t) continue;
      a.rstat[(a.meta.row_base[r] + jl) * a.S + lane / lph] = v;
    }
  }
}

// sum over the edges [beg, end) of one row (relation r, target j) of de K(i), with
// de = alpha (<dS_r(j), V(i)> - D_j) and alpha from the saved softmax statistics.
template <typename T, int D, int NB = kBatch>
__device__ __forceinline__ void dst_edges(const HgtArgs& a, int64_t beg, int64_t end, const float (&q)[D / 32],
                                          const float (&g)[D / 32], float m, float inv_l, float Dh, int lph,
                                          float (&acc)[D / 32]) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31;
  const T* KV = (const T*)a.KV;
  for (int64_t e0 = beg; e0 < end; e0 += NB) {
    int src[NB];
    float w[NB];
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      src[u] = e0 + u < end ? __ldg(a.dcol + e0 + u) : -1;
      w[u] = e0 + u < end ? (float)__ldg(a.dcnt + e0 + u) : 0.f;
    }
    float k[NB][E], v[NB][E];
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      if (src[u] >= 0) {
        load_slice<T, E>(KV + (int64_t)src[u] * 2 * D + lane * E, k[u]);
        load_slice<T, E>(KV + (int64_t)src[u] * 2 * D + D + lane * E, v[u]);
      }
    }
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      if (src[u] < 0) break;
      float s = 0.f, da = 0.f;
#pragma unroll
      for (int e = 0; e < E; ++e) {
        s = fmaf(k[u][e], q[e], s);
        da = fmaf(g[e], v[u][e], da);
      }
      s = head_sum(s, lph);
      da = head_sum(da, lph);
      const float alpha = expf(s - m) * inv_l;
      const float de = w[u] * alpha * (da - Dh);  // the run's w edges
#pragma unroll
      for (int e = 0; e < E; ++e) acc[e] = fmaf(de, k[u][e], acc[e]);
    }
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(256) hgt_bwd_dst_chunks(HgtArgs a) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, lph = 32 / a.S, h = lane / lph;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int nchunks = a.dchunk_ofs[a.csr_rows];
  for (int64_t c = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; c < nchunks; c += nw) {
    const int row = a.dchunk_row[c];
    const int64_t beg = (int64_t)a.dptr[row] + (int64_t)(c - a.dchunk_ofs[row]) * kChunkEdges;
    const int64_t end = min((int64_t)a.dptr[row + 1], beg + kChunkEdges);
    const float4 st = a.rstat[(int64_t)row * a.S + h];
    float q[E], g[E], acc[E];
    load_slice<T, E>((const T*)a.Qp + (int64_t)row * D + lane * E, q);
    load_slice<T, E>((const T*)a.dS + (int64_t)row * D + lane * E, g);
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = 0.f;
    dst_edges<T, D, kBatchChunk>(a, beg, end, q, g, st.x, st.y, st.z, lph, acc);
#pragma unroll
    for (int e = 0; e < E; ++e) a.part[c * D + lane * E + e] = acc[e];
  }
}

// dQ'_r(j) for every relation row of node j (hub rows: their chunk partials in order); the row
// bounds, query and gradient slices of all of j's rows are loaded before any edge.
template <typename T, int D, int KS>
__global__ void __launch_bounds__(256, (D <= 128 && KS <= 4) ? 3 : 1) hgt_bwd_dst_nodes(HgtArgs a) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, lph = 32 / a.S, h = lane / lph;
  const int64_t j = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (j >= a.N) return;
  const int t = node_type_of(a.meta, j);
  const int64_t jl = j - a.meta.type_off[t];
  int64_t row[KS];
  int c0[KS], c1[KS];
  int64_t e0[KS], e1[KS];
  float q[KS][E], g[KS][E];
#pragma unroll
  for (int k = 0; k < KS; ++k) {
    const int r = a.rslot[t][k];
    row[k] = r >= 0 ? a.meta.row_base[r] + jl : -1;
    if (row[k] >= 0) {
      c0[k] = a.dchunk_ofs[row[k]];
      c1[k] = a.dchunk_ofs[row[k] + 1];
      e0[k] = a.dptr[row[k]];
      e1[k] = a.dptr[row[k] + 1];
      load_slice<T, E>((const T*)a.Qp + row[k] * D + lane * E, q[k]);
      load_slice<T, E>((const T*)a.dS + row[k] * D + lane * E, g[k]);
    }
  }
  const float4 st = row[0] >= 0 ? a.rstat[row[0] * a.S + h] : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
  for (int k = 0; k < KS; ++k) {
    if (row[k] < 0) continue;
    float acc[E];
#pragma unroll
    for (int e = 0; e < E; ++e) acc[e] = 0.f;
    if (c1[k] > c0[k]) {
      for (int c = c0[k]; c < c1[k]; ++c)
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] += a.part[(int64_t)c * D + lane * E + e];
    } else {
      dst_edges<T, D>(a, e0[k], e1[k], q[k], g[k], st.x, st.y, st.z, lph, acc);
    }
    store_slice<T, E>((T*)a.dQp + row[k] * D + lane * E, acc);
  }
}

// Out-edges [beg, end) of source i (node-major list; each entry is the CSR row of the edge's
// target): dK(i) += de Q'_r(j), dV(i) += alpha dS_r(j).
template <typename T, int D, int NB = kBatch>
__device__ __forceinline__ void src_edges(const HgtArgs& a, int64_t beg, int64_t end, const float (&k)[D / 32],
                                          const float (&v)[D / 32], int lph, float (&ak)[D / 32],
                                          float (&av)[D / 32]) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, h = lane / lph;
  for (int64_t e0 = beg; e0 < end; e0 += NB) {
    int row[NB];
    float w[NB];
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      row[u] = e0 + u < end ? __ldg(a.mlist + __ldg(a.scol + e0 + u)) : -1;
      w[u] = e0 + u < end ? (float)__ldg(a.scnt + e0 + u) : 0.f;
    }
    float q[NB][E], g[NB][E];
    float4 st[NB];
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      if (row[u] >= 0) {
        load_slice<T, E>((const T*)a.Qp + (int64_t)row[u] * D + lane * E, q[u]);
        load_slice<T, E>((const T*)a.dS + (int64_t)row[u] * D + lane * E, g[u]);
        st[u] = a.rstat[(int64_t)row[u] * a.S + h];
      }
    }
#pragma unroll
    for (int u = 0; u < NB; ++u) {
      if (row[u] < 0) break;
      float s = 0.f, da = 0.f;
#pragma unroll
      for (int e = 0; e < E; ++e) {
        s = fmaf(k[e], q[u][e], s);
        da = fmaf(g[u][e], v[e], da);
      }
      s = head_sum(s, lph);
      da = head_sum(da, lph);
      const float alpha = w[u] * expf(s - st[u].x) * st[u].y;  // the run's w edges
      const float de = alpha * (da - st[u].z);
#pragma unroll
      for (int e = 0; e < E; ++e) {
        ak[e] = fmaf(de, q[u][e], ak[e]);
        av[e] = fmaf(alpha, g[u][e], av[e]);
      }
    }
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(256) hgt_bwd_src_chunks(HgtArgs a) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, lph = 32 / a.S;
  const int64_t nw = ((int64_t)gridDim.x * blockDim.x) >> 5;
  const int nchunks = a.schunk_ofs[a.N];
  const T* KV = (const T*)a.KV;
  for (int64_t c = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; c < nchunks; c += nw) {
    const int i = a.schunk_row[c];
    const int64_t beg = (int64_t)a.sptr[i] + (int64_t)(c - a.schunk_ofs[i]) * kChunkEdges;
    const int64_t end = min((int64_t)a.sptr[i + 1], beg + kChunkEdges);
    float k[E], v[E], ak[E], av[E];
    load_slice<T, E>(KV + (int64_t)i * 2 * D + lane * E, k);
    load_slice<T, E>(KV + (int64_t)i * 2 * D + D + lane * E, v);
#pragma unroll
    for (int e = 0; e < E; ++e) ak[e] = av[e] = 0.f;
    src_edges<T, D, kBatchChunk>(a, beg, end, k, v, lph, ak, av);
#pragma unroll
    for (int e = 0; e < E; ++e) {
      a.part[c * 2 * D + lane * E + e] = ak[e];
      a.part[c * 2 * D + D + lane * E + e] = av[e];
    }
  }
}

template <typename T, int D>
__global__ void __launch_bounds__(256) hgt_bwd_src_nodes(HgtArgs a) {
  constexpr int E = D / 32;
  const int lane = threadIdx.x & 31, lph = 32 / a.S;
  const int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (i >= a.N) return;
  float ak[E], av[E];
#pragma unroll
  for (int e = 0; e < E; ++e) ak[e] = av[e] = 0.f;
  const int c0 = a.schunk_ofs[i], c1 = a.schunk_ofs[i + 1];
  if (c1 > c0) {
    for (int c = c0; c < c1; ++c)
#pragma unroll
      for (int e = 0; e < E; ++e) {
        ak[e] += a.part[(int64_t)c * 2 * D + lane * E + e];
        av[e] += a.part[(int64_t)c * 2 * D + D + lane * E + e];
      }
  } else {
    float k[E], v[E];
    const T* KV = (const T*)a.KV;
    load_slice<T, E>(KV + i * 2 * D + lane * E, k);
    load_slice<T, E>(KV + i * 2 * D + D + lane * E, v);
    src_edges<T, D>(a, a.sptr[i], a.sptr[i + 1], k, v, lph, ak, av);
  }
  store_slice<T, E>((T*)a.dK + i * D + lane * E, ak);
  store_slice<T, E>((T*)a.dV + i * D + lane * E, av);
}

// dW_msg[r][s] = the diagonal blocks of the dense gradient G[r] (d x d); dW_att[r][s] = c_r times the
// blocks of Gq[r] = dQ'_r^T Q; dmu[r] = <blockdiag(W_att[r]), Gq[r]> / sqrt(d_h) (one block per relation,
// fixed-order reduction).
template <typename T>
__global__ void __launch_bounds__(256) hgt_finish(const float* __restrict__ G, const float* __restrict__ Gq,
                                                  const T* __restrict__ W_att, const float* __restrict__ mu, int d,
                                                  int S, float* __restrict__ dW_msg, float* __restrict__ dW_att,
                                                  float* __restrict__ dmu) {
  __shared__ float red[256];
  const int r = blockIdx.x, dh = d / S;
  const float rs = rsqrtf((float)dh);
  const float c = mu[r] * rs;
  float acc = 0.f;
  for (int q = threadIdx.x; q < S * dh * dh; q += blockDim.x) {
    const int s = q / (dh * dh), a = (q / dh) % dh, b = q % dh;
    const int64_t gi = (int64_t)r * d * d + (int64_t)(s * dh + a) * d + s * dh + b;
    dW_msg[(int64_t)r * S * dh * dh + q] = G[gi];
    dW_att[(int64_t)r * S * dh * dh + q] = c * Gq[gi];
    acc = fmaf(to_f32(W_att[(int64_t)r * S * dh * dh + q]), Gq[gi], acc);
  }
  red[threadIdx.x] = acc;
  __syncthreads();
  if (threadIdx.x == 0) {
    float t = 0.f;
    for (int k = 0; k < (int)blockDim.x; ++k) t += red[k];
    dmu[r] = t * rs;
  }
}

}  // namespace
}  // namespace hg

namespace hg {
namespace {

struct HgtLayout {
  LayerLayout L;
  // saved
  void* KV;       // N x 2d
  void* Qp;       // csr_rows x d
  float2* stats;  // N x S
  void* BDmsg;    // R x d x d  blockdiag(W_msg[r])
  // scratch
  void* BDattT;   // R x d x d  blockdiag(W_att[r])^T
  void* BDatt;    // R x d x d  blockdiag(W_att[r])
  void* WKt;      // T x d x d
  void* WVt;      // T x d x d
  void* WQt;      // T x d x d
  float4* rstat;  // csr_rows x S
  void* dQp;      // csr_rows x d
  void* dK;       // N x d
  void* dV;       // N x d
  void* Qbuf;     // N x d: Q (forward), recomputed in the backward
  void* dQ;       // N x d
  float* part;    // chunk partials
  float* cs;      // column-sum partials
  float* Gw;      // R x d x d
  float* Gq;      // R x d x d
};

constexpr int64_t kColRows = 128;  // rows per block of the bias sums (many blocks in flight)

int64_t max_type_rows(const GraphMeta& m) {
  int64_t r = 1;
  for (int t = 0; t < m.num_types; ++t) r = std::max(r, m.type_off[t + 1] - m.type_off[t]);
  return r;
}

void carve_hgt(const hg_graph* g, const hg_hgt_params* p, void* saved, void* scratch, HgtLayout* H,
               size_t* saved_bytes, size_t* scratch_bytes) {
  const GraphMeta& m = g->meta;
  const int d = p->d, S = p->heads;
  const size_t b = p->dtype == HG_F32 ? 4 : 2;
  const int64_t N = m.type_off[m.num_types];
  const size_t dd = (size_t)d * d;
  size_t ls = 0, lk = 0;
  carve_layer(g, d, p->dtype, saved, scratch, &H->L, &ls, &lk);
  Carve s(saved), k(scratch);
  s.used = align_up(ls);
  k.used = align_up(lk);
  H->KV = s.take<char>((size_t)std::max<int64_t>(N, 1) * 2 * d * b);
  H->Qp = s.take<char>((size_t)std::max<int64_t>(g->csr_rows, 1) * d * b);
  H->stats = s.take<float2>((size_t)std::max<int64_t>(N, 1) * S);
  H->BDmsg = s.take<char>(m.num_rels * dd * b);
  H->BDattT = k.take<char>(m.num_rels * dd * b);
  H->BDatt = k.take<char>(m.num_rels * dd * b);
  H->WKt = k.take<char>(m.num_types * dd * b);
  H->WVt = k.take<char>(m.num_types * dd * b);
  H->WQt = k.take<char>(m.num_types * dd * b);
  H->rstat = k.take<float4>((size_t)std::max<int64_t>(g->csr_rows, 1) * S);
  H->dQp = k.take<char>((size_t)std::max<int64_t>(g->csr_rows, 1) * d * b);
  H->dK = k.take<char>((size_t)std::max<int64_t>(N, 1) * d * b);
  H->dV = k.take<char>((size_t)std::max<int64_t>(N, 1) * d * b);
  H->Qbuf = k.take<char>((size_t)std::max<int64_t>(N, 1) * d * b);
  H->dQ = k.take<char>((size_t)std::max<int64_t>(N, 1) * d * b);
  const int64_t pc = std::max<int64_t>(g->chunk_cap_csr * (2 * S + d), g->chunk_cap_node * 2 * d);
  H->part = k.take<float>((size_t)std::max<int64_t>(pc, 1));
  H->cs = k.take<float>((size_t)ceil_div(max_type_rows(m), kColRows) * d);
  H->Gw = k.take<float>(m.num_rels * dd);
  H->Gq = k.take<float>(m.num_rels * dd);
  if (saved_bytes) *saved_bytes = s.used;
  if (scratch_bytes) *scratch_bytes = k.used;
}

hg_layer_params projection_params(const hg_hgt_params* p, const HgtLayout& H) {
  hg_layer_params lp{};
  lp.d = p->d;
  lp.dtype = p->dtype;
  lp.act = p->act;
  lp.layernorm = p->layernorm;
  lp.ln_eps = p->ln_eps;
  lp.W_rel = H.BDmsg;
  lp.W_agg = p->W_agg;
  lp.b_agg = p->b_agg;
  lp.ln_gamma = p->ln_gamma;
  lp.ln_beta = p->ln_beta;
  return lp;
}

HgtArgs edge_args(const hg_graph* g, const hg_hgt_params* p, const HgtLayout& H) {
  HgtArgs a{};
  a.meta = g->meta;
  for (int t = 0; t < kMaxTypes; ++t) {
    int k = 0;
    for (int r = 0; r < kMaxRels; ++r) a.rslot[t][r] = -1;
    for (int r = 0; r < g->meta.num_rels; ++r)
      if (t < g->meta.num_types && g->meta.rel_dst[r] == t) a.rslot[t][k++] = (int8_t)r;
  }
  a.N = g->meta.type_off[g->meta.num_types];
  a.csr_rows = g->csr_rows;
  a.S = p->heads;
  a.dptr = g->agg_ptr;
  a.dcol = g->agg_col;
  a.dcnt = g->agg_cnt;
  a.dchunk_ofs = g->agg_chunk_ofs;
  a.dchunk_row = g->agg_chunk_row;
  a.sptr = g->bagg_ptr;
  a.scol = g->bagg_col;
  a.scnt = g->bagg_cnt;
  a.schunk_ofs = g->bagg_chunk_ofs;
  a.schunk_row = g->bagg_chunk_row;
  a.mlist = g->mlist;
  a.KV = H.KV;
  a.Qp = H.Qp;
  a.Srows = H.L.M;
  a.dS = H.L.dMs;
  a.stats = H.stats;
  a.rstat = H.rstat;
  a.dQp = H.dQp;
  a.dK = H.dK;
  a.dV = H.dV;
  a.part = H.part;
  return a;
}

// Relations into the busiest type (the node kernels keep one slot per relation of a type).
int max_rels_per_type(const GraphMeta& m) {
  int best = 0;
  for (int t = 0; t < m.num_types; ++t) {
    int k = 0;
    for (int r = 0; r < m.num_rels; ++r) k += m.rel_dst[r] == t;
    best = std::max(best, k);
  }
  return best;
}

unsigned grid_of(int64_t threads) { return (unsigned)std::max<int64_t>(1, ceil_div(threads, 256)); }
unsigned chunk_blocks(int64_t cap) { return (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(cap, 8), 152 * 16)); }

template <typename T, int D>
hg_status gemm(const void* A, int64_t lda, const void* B, const void* bias, int K, int64_t n, void* out, int64_t ldo,
               int ocol0, int accumulate, cudaStream_t s, const float* scale_ptr = nullptr, float scale_mul = 1.f) {
  if (n <= 0) return HG_OK;
  if constexpr (sizeof(T) == 2) {  // bf16: tensor cores (every product here has K = lda = D)
    if (lda == D && K == D)
      return rows_gemm_tc(D, A, n, B, bias, out, ldo, ocol0, accumulate, scale_ptr, scale_mul, s);
  }
  return launch("hgt_gemm_simt", hgt_gemm_simt<T, D>, dim3((unsigned)ceil_div(n, kBM)), dim3(256),
                sizeof(float) * kKC * D, s, (const T*)A, lda, (const T*)B, (const T*)bias, K, n, (T*)out, ldo, ocol0,
                accumulate, scale_ptr, scale_mul);
}

template <typename T>
hg_status colsum(const void* X, int64_t ldx, int d, int64_t n, float* cs, float* out, float* tmp, cudaStream_t s) {
  if (n <= 0) {
    HG_CUDA(cudaMemsetAsync(out, 0, sizeof(float) * d, s));
    return HG_OK;
  }
  const int blocks = (int)ceil_div(n, kColRows);
  HG_TRY(launch("hgt_colsum", hgt_colsum<T>, dim3(blocks), dim3(std::min(d, 256)), 0, s, (const T*)X, ldx, d, n,
                kColRows, cs));
  return reduce_partials(cs, d, blocks, d, out, tmp, s);
}

hg_status wgrad(hg_dtype dt, int d, const void* X, int64_t x0, const void* Y, int64_t y0, int64_t n, float* out,
                const LayerLayout& L, cudaStream_t s) {
  if (n <= 0) {
    HG_CUDA(cudaMemsetAsync(out, 0, sizeof(float) * d * d, s));
    return HG_OK;
  }
  if (dt == HG_BF16) {
    float* outs[1] = {out};
    return tc_weight_grad(d, X, &x0, 1, Y, y0, n, L.wpart, outs, L.rtmp, s);
  }
  return weight_grad(dt, d, X, x0, Y, y0, n, L.wpart, out, L.rtmp, s);
}

template <typename T, int D>
hg_status hgt_fwd_t(const hg_graph* g, const hg_hgt_params* p, const void* H_in, void* H_out, const HgtLayout& H,
                    cudaStream_t s) {
  const GraphMeta& m = g->meta;
  const int S = p->heads;
  const int64_t N = m.type_off[m.num_types];
  const size_t dd = (size_t)D * D;
  const T* Hin = (const T*)H_in;
  const float rs = (float)(1.0 / std::sqrt((double)(D / S)));
  // block-diagonal attention (transposed) and message matrices
  HG_TRY(launch("hgt_blockdiag", hgt_blockdiag<T>, dim3(grid_of((int64_t)m.num_rels * dd)), dim3(256), 0, s,
                (const T*)p->W_att, m.num_rels, D, S, 1, (T*)H.BDattT));
  HG_TRY(launch("hgt_blockdiag", hgt_blockdiag<T>, dim3(grid_of((int64_t)m.num_rels * dd)), dim3(256), 0, s,
                (const T*)p->W_msg, m.num_rels, D, S, 0, (T*)H.BDmsg));
  // K, V and Q of every node, Q' of every (relation, target) row
  for (int t = 0; t < m.num_types; ++t) {
    const int64_t off = m.type_off[t], n = m.type_off[t + 1] - off;
    HG_TRY((gemm<T, D>(Hin + off * D, D, (const T*)p->W_K + t * dd, (const T*)p->b_K + (size_t)t * D, D, n,
                       (T*)H.KV + off * 2 * D, 2 * D, 0, 0, s)));
    HG_TRY((gemm<T, D>(Hin + off * D, D, (const T*)p->W_V + t * dd, (const T*)p->b_V + (size_t)t * D, D, n,
                       (T*)H.KV + off * 2 * D, 2 * D, D, 0, s)));
    HG_TRY((gemm<T, D>(Hin + off * D, D, (const T*)p->W_Q + t * dd, (const T*)p->b_Q + (size_t)t * D, D, n,
                       (T*)H.Qbuf + off * D, D, 0, 0, s)));
  }
  for (int r = 0; r < m.num_rels; ++r) {  // Q'_r = c_r Q blockdiag(W_att[r])^T, c_r = mu[r] / sqrt(d_h)
    const int t = m.rel_dst[r];
    const int64_t off = m.type_off[t], n = m.type_off[t + 1] - off;
    HG_TRY((gemm<T, D>((const T*)H.Qbuf + off * D, D, (const T*)H.BDattT + r * dd, nullptr, D, n,
                       (T*)H.Qp + m.row_base[r] * D, D, 0, 0, s, p->mu + r, rs)));
  }
  // Eq. 6-10: softmax over the in-edges, weighted value sums per relation row
  const HgtArgs a = edge_args(g, p, H);
  HG_TRY(launch("hgt_fwd_chunks", hgt_fwd_chunks<T, D>, dim3(chunk_blocks(g->chunk_cap_csr)), dim3(256), 0, s, a));
  if (max_rels_per_type(m) <= 4)
    HG_TRY(launch("hgt_fwd_nodes", hgt_fwd_nodes<T, D, 4>, dim3(grid_of(N * 32)), dim3(256), 0, s, a));
  else
    HG_TRY(launch("hgt_fwd_nodes", hgt_fwd_nodes<T, D, kMaxRels>, dim3(grid_of(N * 32)), dim3(256), 0, s, a));
  // Eq. 11 on S_r with W_rel = blockdiag(W_msg[r])
  const hg_layer_params lp = projection_params(p, H);
  return project_forward(g, &lp, H_in, H_out, H.L, false, s);
}

template <typename T, int D>
hg_status hgt_bwd_t(const hg_graph* g, const hg_hgt_params* p, const void* H_in, const void* dH_out, void* dH_in,
                    const hg_hgt_grads* gr, const HgtLayout& H, cudaStream_t s) {
  constexpr hg_dtype kDt = sizeof(T) == 2 ? HG_BF16 : HG_F32;
  const GraphMeta& m = g->meta;
  const int S = p->heads;
  const int64_t N = m.type_off[m.num_types];
  const size_t dd = (size_t)D * D;
  const T* Hin = (const T*)H_in;
  const float rs = (float)(1.0 / std::sqrt((double)(D / S)));
  // Eq. 11 backward: dY (residual), dS_r (no degree scaling), dW of blockdiag(W_msg), dW_agg, db, LN
  const hg_layer_params lp = projection_params(p, H);
  hg_layer_grads lg{};
  lg.dW_rel = H.Gw;
  lg.dW_agg = gr->dW_agg;
  lg.db_agg = gr->db_agg;
  lg.dln_gamma = gr->dln_gamma;
  lg.dln_beta = gr->dln_beta;
  HG_TRY(project_backward(g, &lp, H_in, dH_out, &lg, H.L, false, false, s));
  // attention backward: target pass (dQ'), source pass (dK, dV)
  const HgtArgs a = edge_args(g, p, H);
  HG_TRY(launch("hgt_bwd_dstats", hgt_bwd_dstats<T, D>, dim3(grid_of(N * 32)), dim3(256), 0, s, a));
  HG_TRY(launch("hgt_bwd_dst_chunks", hgt_bwd_dst_chunks<T, D>, dim3(chunk_blocks(g->chunk_cap_csr)), dim3(256), 0, s,
                a));
  if (max_rels_per_type(m) <= 4)
    HG_TRY(launch("hgt_bwd_dst_nodes", hgt_bwd_dst_nodes<T, D, 4>, dim3(grid_of(N * 32)), dim3(256), 0, s, a));
  else
    HG_TRY(launch("hgt_bwd_dst_nodes", hgt_bwd_dst_nodes<T, D, kMaxRels>, dim3(grid_of(N * 32)), dim3(256), 0, s,
                  a));
  HG_TRY(launch("hgt_bwd_src_chunks", hgt_bwd_src_chunks<T, D>, dim3(chunk_blocks(g->chunk_cap_node)), dim3(256), 0,
                s, a));
  HG_TRY(launch("hgt_bwd_src_nodes", hgt_bwd_src_nodes<T, D>, dim3(grid_of(N * 32)), dim3(256), 0, s, a));
  // weights of the backward products (exact copies and transposes)
  HG_TRY(launch("hgt_blockdiag", hgt_blockdiag<T>, dim3(grid_of((int64_t)m.num_rels * dd)), dim3(256), 0, s,
                (const T*)p->W_att, m.num_rels, D, S, 0, (T*)H.BDatt));
  HG_TRY(launch("hgt_transpose", hgt_transpose<T>, dim3(grid_of((int64_t)m.num_types * dd)), dim3(256), 0, s,
                (const T*)p->W_K, m.num_types, D, (T*)H.WKt));
  HG_TRY(launch("hgt_transpose", hgt_transpose<T>, dim3(grid_of((int64_t)m.num_types * dd)), dim3(256), 0, s,
                (const T*)p->W_V, m.num_types, D, (T*)H.WVt));
  HG_TRY(launch("hgt_transpose", hgt_transpose<T>, dim3(grid_of((int64_t)m.num_types * dd)), dim3(256), 0, s,
                (const T*)p->W_Q, m.num_types, D, (T*)H.WQt));
  // dQ = sum_r c_r dQ'_r blockdiag(W_att[r]) per target type
  for (int t = 0; t < m.num_types; ++t) {
    const int64_t off = m.type_off[t], n = m.type_off[t + 1] - off;
    int k = 0;
    for (int r = 0; r < m.num_rels; ++r) {
      if (m.rel_dst[r] != t) continue;
      HG_TRY((gemm<T, D>((const T*)H.dQp + m.row_base[r] * D, D, (const T*)H.BDatt + r * dd, nullptr, D, n,
                         (T*)H.dQ + off * D, D, 0, k > 0, s, p->mu + r, rs)));
      ++k;
    }
    if (k == 0 && n > 0) HG_CUDA(cudaMemsetAsync((T*)H.dQ + off * D, 0, (size_t)n * D * sizeof(T), s));
  }
  // dH_in = dY + dK W_K^T + dV W_V^T + dQ W_Q^T
  if (dH_in) {
    HG_CUDA(cudaMemcpyAsync(dH_in, H.L.dY, (size_t)N * D * sizeof(T), cudaMemcpyDeviceToDevice, s));
    T* dH = (T*)dH_in;
    for (int t = 0; t < m.num_types; ++t) {
      const int64_t off = m.type_off[t], n = m.type_off[t + 1] - off;
      HG_TRY((gemm<T, D>((const T*)H.dK + off * D, D, (const T*)H.WKt + t * dd, nullptr, D, n, dH + off * D, D, 0, 1,
                         s)));
      HG_TRY((gemm<T, D>((const T*)H.dV + off * D, D, (const T*)H.WVt + t * dd, nullptr, D, n, dH + off * D, D, 0, 1,
                         s)));
      HG_TRY((gemm<T, D>((const T*)H.dQ + off * D, D, (const T*)H.WQt + t * dd, nullptr, D, n, dH + off * D, D, 0, 1,
                         s)));
    }
  }
  // weight gradients of the three typed maps: dW = H^T dZ, db = column sums of dZ; Q recomputed for
  // the attention matrices' gradients
  for (int t = 0; t < m.num_types; ++t) {
    const int64_t off = m.type_off[t], n = m.type_off[t + 1] - off;
    HG_TRY(wgrad(kDt, D, H_in, off, H.dK, off, n, gr->dW_K + t * dd, H.L, s));
    HG_TRY(wgrad(kDt, D, H_in, off, H.dV, off, n, gr->dW_V + t * dd, H.L, s));
    HG_TRY(colsum<T>((const T*)H.dK + off * D, D, D, n, H.cs, gr->db_K + (size_t)t * D, H.L.rtmp, s));
    HG_TRY(colsum<T>((const T*)H.dV + off * D, D, D, n, H.cs, gr->db_V + (size_t)t * D, H.L.rtmp, s));
    HG_TRY(wgrad(kDt, D, H_in, off, H.dQ, off, n, gr->dW_Q + t * dd, H.L, s));
    HG_TRY(colsum<T>((const T*)H.dQ + off * D, D, D, n, H.cs, gr->db_Q + (size_t)t * D, H.L.rtmp, s));
    HG_TRY((gemm<T, D>(Hin + off * D, D, (const T*)p->W_Q + t * dd, (const T*)p->b_Q + (size_t)t * D, D, n,
                       (T*)H.Qbuf + off * D, D, 0, 0, s)));
  }
  for (int r = 0; r < m.num_rels; ++r) {  // Gq[r] = dQ'_r^T Q
    const int t = m.rel_dst[r];
    const int64_t off = m.type_off[t], n = m.type_off[t + 1] - off;
    HG_TRY(wgrad(kDt, D, H.dQp, m.row_base[r], H.Qbuf, off, n, H.Gq + r * dd, H.L, s));
  }
  return launch("hgt_finish", hgt_finish<T>, dim3(m.num_rels), dim3(256), 0, s, (const float*)H.Gw,
                (const float*)H.Gq, (const T*)p->W_att, p->mu, D, S, gr->dW_msg, gr->dW_att, gr->dmu);
}

#define HG_HGT_DISPATCH(dtype, d, FN, ...)                                                  \
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

hg_status check_hgt(const hg_graph* g, const hg_hgt_params* p) {
  HG_REQUIRE(g && p, "graph and params must be non-null");
  if (!(p->d == 64 || p->d == 128 || p->d == 256) || !(p->dtype == HG_F32 || p->dtype == HG_BF16)) {
    set_error("unsupported d=%d / dtype=%d", p->d, (int)p->dtype);
    return HG_ERR_UNSUPPORTED;
  }
  HG_REQUIRE(p->heads >= 1 && p->heads <= 32 && (p->heads & (p->heads - 1)) == 0,
             "heads must be a power of two in [1, 32]");
  HG_REQUIRE(p->act == HG_ACT_RELU || p->act == HG_ACT_GELU_TANH || p->act == HG_ACT_NONE, "unknown activation");
  HG_REQUIRE(p->W_K && p->W_Q && p->W_V && p->b_K && p->b_Q && p->b_V && p->W_att && p->W_msg && p->mu && p->W_agg &&
                 p->b_agg,
             "every parameter pointer must be non-null");
  HG_REQUIRE(!p->layernorm || (p->ln_gamma && p->ln_beta && p->ln_eps > 0.f), "layernorm needs gamma, beta, eps > 0");
  return HG_OK;
}

hg_status check_buf256(const void* q, const char* name) {
  HG_REQUIRE(q != nullptr, "%s must be non-null", name);
  HG_REQUIRE(((uintptr_t)q & 255) == 0, "%s must be 256-byte aligned", name);
  return HG_OK;
}

}  // namespace
}  // namespace hg

using namespace hg;

extern "C" hg_status hg_hgt_workspace_size(const hg_graph* graph, const hg_hgt_params* params, size_t* saved_bytes,
                                          size_t* scratch_bytes) {
  clear_error();
  HG_TRY(check_hgt(graph, params));
  HG_REQUIRE(saved_bytes && scratch_bytes, "saved_bytes and scratch_bytes must be non-null");
  HgtLayout H;
  carve_hgt(graph, params, nullptr, nullptr, &H, saved_bytes, scratch_bytes);
  return HG_OK;
}

extern "C" hg_status hg_hgt_fwd(const hg_graph* graph, const hg_hgt_params* params, const void* H_in, void* H_out,
                               void* saved, void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_hgt(graph, params));
  HG_TRY(check_buf256(H_in, "H_in"));
  HG_TRY(check_buf256(H_out, "H_out"));
  HG_TRY(check_buf256(saved, "saved"));
  HG_TRY(check_buf256(scratch, "scratch"));
  HG_REQUIRE(H_in != H_out, "H_in and H_out must not alias");
  HgtLayout H;
  carve_hgt(graph, params, saved, scratch, &H, nullptr, nullptr);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  HG_HGT_DISPATCH(params->dtype, params->d, hgt_fwd_t, graph, params, H_in, H_out, H, s);
}

extern "C" hg_status hg_hgt_bwd(const hg_graph* graph, const hg_hgt_params* params, const void* H_in,
                               const void* saved, const void* dH_out, void* dH_in, const hg_hgt_grads* grads,
                               void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  HG_TRY(check_hgt(graph, params));
  HG_TRY(check_buf256(H_in, "H_in"));
  HG_TRY(check_buf256(saved, "saved"));
  HG_TRY(check_buf256(dH_out, "dH_out"));
  HG_TRY(check_buf256(scratch, "scratch"));
  HG_REQUIRE(dH_in == nullptr || ((uintptr_t)dH_in & 255) == 0, "dH_in must be 256-byte aligned");
  HG_REQUIRE(dH_in != dH_out, "dH_in and dH_out must not alias");
  HG_REQUIRE(grads && grads->dW_K && grads->dW_Q && grads->dW_V && grads->db_K && grads->db_Q && grads->db_V &&
                 grads->dW_att && grads->dW_msg && grads->dmu && grads->dW_agg && grads->db_agg,
             "every gradient pointer must be non-null");
  HG_REQUIRE(!params->layernorm || (grads->dln_gamma && grads->dln_beta), "layernorm needs dln_gamma and dln_beta");
  HgtLayout H;
  carve_hgt(graph, params, const_cast<void*>(saved), scratch, &H, nullptr, nullptr);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  HG_HGT_DISPATCH(params->dtype, params->d, hgt_bwd_t, graph, params, H_in, dH_out, dH_in, grads, H, s);
}
