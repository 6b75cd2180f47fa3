// Overlap batch and cross-subgraph CCA alignment (Section 3.3, Eq. 14-17).
//
// Intersection: both global-id lists are strictly ascending; each id of list a is located in
// list b by binary search, the hits are compacted with an exclusive scan, so the pairs come out
// in ascending global id.  Integer work, bit-exact.
//
// Loss, on X_a = H_a[idx_a], X_b = H_b[idx_b] (n rows, d columns, fp32 arithmetic):
//   mu, var (population, two passes) per column -> s = sqrt(var + eps)
//   Z = (X - mu) / (s sqrt(n))                                        (Eq. 14)
//   C = Z^T Z per view (split over rows, fixed-order reduction)
//   L_inv = ||Z_a - Z_b||^2, L_dec = ||C_a - I||^2 + ||C_b - I||^2    (Eq. 15-17)
// Gradient of dloss * L:
//   G_a = dloss (2 (Z_a - Z_b) + 4 lambda Z_a (C_a - I)),  G_b = dloss (-2 (Z_a - Z_b) + 4 lambda Z_b (C_b - I))
//   with x_hat = sqrt(n) Z and g = G / sqrt(n) per column:
//   dX = (g - mean(g) - x_hat mean(g x_hat)) / s, added into dH at the overlap rows.
// All reductions run in a fixed order (per-block partials, then a serial sum over blocks).
#include <algorithm>
#include <type_traits>

#include "align_kernels.cuh"
#include "layer_kernels.cuh"
#include "simt_tile.cuh"

namespace hg {

// ---------------------------------------------------------------------------------------------
// intersection
// ---------------------------------------------------------------------------------------------
__global__ void intersect_flags(const int64_t* __restrict__ a, int64_t na, const int64_t* __restrict__ b, int64_t nb,
                                int32_t* __restrict__ flag, int32_t* __restrict__ pos, int32_t* __restrict__ bad) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < na; i += stride) {
    const int64_t x = a[i];
    if (i > 0 && a[i - 1] >= x) atomicOr(bad, 1);
    int64_t lo = 0, hi = nb;  // first index with b[k] >= x
    while (lo < hi) {
      const int64_t mid = (lo + hi) >> 1;
      if (b[mid] < x) lo = mid + 1; else hi = mid;
    }
    const bool hit = lo < nb && b[lo] == x;
    flag[i] = hit ? 1 : 0;
    pos[i] = hit ? (int32_t)lo : -1;
  }
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x + 1; k < nb; k += stride)
    if (b[k - 1] >= b[k]) atomicOr(bad, 1);
}

__global__ void intersect_write(const int32_t* __restrict__ flag, const int32_t* __restrict__ pos,
                                const int32_t* __restrict__ ofs, int64_t na, int64_t cap, const int32_t* __restrict__ bad,
                                int32_t* __restrict__ idx_a, int32_t* __restrict__ idx_b, int64_t* __restrict__ n_out) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < na; i += (int64_t)gridDim.x * blockDim.x) {
    if (flag[i] && ofs[i] < cap) {  // cap bounds the writes even for lists that are not ascending
      idx_a[ofs[i]] = (int32_t)i;
      idx_b[ofs[i]] = pos[i];
    }
  }
  if (blockIdx.x == 0 && threadIdx.x == 0) *n_out = *bad ? -1 : (int64_t)ofs[na];
}

// ---------------------------------------------------------------------------------------------
// alignment helpers
// ---------------------------------------------------------------------------------------------
constexpr int kAlignBlocks = 304;  // row blocks of the column reductions (2 per SM)

// Column sums over the overlap rows of both views, per block (fixed order within the block):
//   MODE 0: x_a, x_b                               part[block][2][d]
//   MODE 1: (x_a - mu_a)^2, (x_b - mu_b)^2          part[block][2][d]
//   MODE 2: the kNumCross sums of z (CrossSum)      part[block][6][d]
// A thread owns one 16-byte piece (VEC columns) of a row and keeps four rows in flight.
template <typename T, int D, int MODE>
__global__ void __launch_bounds__(256, 2) align_colstats(const T* __restrict__ Ha, int64_t rows_a,
                                                      const int32_t* __restrict__ ia, const T* __restrict__ Hb,
                                                      int64_t rows_b, const int32_t* __restrict__ ib, int64_t n_max,
                                                      const int64_t* __restrict__ n_dev,
                                                      const float* __restrict__ stats, float* __restrict__ part,
                                                      int32_t* __restrict__ bad) {
  constexpr int VEC = VecTraits<T>::kElems;
  constexpr int TPR = D / VEC;                // threads per row
  constexpr int RPP = 256 / TPR;              // rows per block pass
  constexpr int Q = MODE == 2 ? kNumCross : 2;
  constexpr int U = MODE == 2 ? 2 : 4;        // rows in flight per thread
  constexpr int SLOTS = TPR < 32 ? 8 : RPP;   // partial rows left after the warp-level sums
  __shared__ float red[SLOTS][D];
  const int64_t n = count_of(n_dev, n_max);
  const int g = threadIdx.x % TPR, sub = threadIdx.x / TPR;
  const int c0 = g * VEC;
  float ma[VEC], mb[VEC], ka[VEC], kb[VEC];
  const float rsn = n > 0 ? rsqrtf((float)n) : 0.f;
#pragma unroll
  for (int i = 0; i < VEC; ++i) {
    ma[i] = MODE ? stats[c0 + i] : 0.f;
    mb[i] = MODE ? stats[D + c0 + i] : 0.f;
    ka[i] = MODE == 2 ? rsn / stats[2 * D + c0 + i] : 1.f;  // z = (x - mu) / (s sqrt(n))
    kb[i] = MODE == 2 ? rsn / stats[3 * D + c0 + i] : 1.f;
  }
  float acc[Q][VEC];
#pragma unroll
  for (int q = 0; q < Q; ++q)
#pragma unroll
    for (int i = 0; i < VEC; ++i) acc[q][i] = 0.f;
  const int64_t step = (int64_t)gridDim.x * RPP;
  for (int64_t r0 = (int64_t)blockIdx.x * RPP + sub; r0 < n; r0 += U * step) {
    float xa[U][VEC], xb[U][VEC];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int64_t r = r0 + u * step;
      if (r < n) {
        if (MODE == 0 && g == 0) {
          const int64_t va = ia[r], vb = ib[r];
          if (va < 0 || va >= rows_a || vb < 0 || vb >= rows_b) atomicOr(bad, 1);
        }
        unpack(ldg16(Ha + safe_row(ia, r, rows_a) * D + c0), xa[u], T());
        unpack(ldg16(Hb + safe_row(ib, r, rows_b) * D + c0), xb[u], T());
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (r0 + u * step >= n) break;
#pragma unroll
      for (int i = 0; i < VEC; ++i) {
        if (MODE == 0) {
          acc[0][i] += xa[u][i];
          acc[1][i] += xb[u][i];
        } else if (MODE == 1) {
          const float da = xa[u][i] - ma[i], db = xb[u][i] - mb[i];
          acc[0][i] += da * da;
          acc[1][i] += db * db;
        } else {
          const float za = (xa[u][i] - ma[i]) * ka[i];
          const float zb = (xb[u][i] - mb[i]) * kb[i];
          acc[kSumZa][i] += za;
          acc[kSumZb][i] += zb;
          acc[kSumZaZb][i] += za * zb;
          acc[kSumDiff2][i] += (za - zb) * (za - zb);
          acc[kSumZa2][i] += za * za;
          acc[kSumZb2][i] += zb * zb;
        }
      }
    }
  }
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int q = 0; q < Q; ++q) {
#pragma unroll
    for (int i = 0; i < VEC; ++i) {
      float v = acc[q][i];
      if (TPR < 32) {
#pragma unroll
        for (int off = TPR; off < 32; off <<= 1) v += __shfl_xor_sync(0xffffffffu, v, off);
      }
      acc[q][i] = v;
    }
    if (TPR < 32) {
      if (lane < TPR)
#pragma unroll
        for (int i = 0; i < VEC; ++i) red[warp][c0 + i] = acc[q][i];
    } else {
#pragma unroll
      for (int i = 0; i < VEC; ++i) red[sub][c0 + i] = acc[q][i];
    }
    __syncthreads();
    for (int c = threadIdx.x; c < D; c += blockDim.x) {
      float t = 0.f;
#pragma unroll
      for (int k = 0; k < SLOTS; ++k) t += red[k][c];
      part[((int64_t)blockIdx.x * Q + q) * D + c] = t;
    }
    __syncthreads();
  }
}

// In place over the column sums (reduced from the block partials by reduce_partials):
// mode 0 -> mu = sum / n;  mode 1 -> s = sqrt(sum / n + eps).
__global__ void align_colscale(float* __restrict__ v, int count, const int64_t* __restrict__ n_dev, int64_t n_max,
                               int mode, float eps) {
  const int64_t n = count_of(n_dev, n_max);
  const int k = blockIdx.x * blockDim.x + threadIdx.x;
  if (k >= count) return;
  const float m = n > 0 ? v[k] / (float)n : 0.f;
  v[k] = mode ? sqrtf(m + eps) : m;
}

// Gram partials of the standardised rows on the CUDA cores (fp32 storage): part[split][view][d][d].
template <typename T, int D>
__global__ void __launch_bounds__(256) align_gram(const T* __restrict__ Ha, int64_t rows_a,
                                                  const int32_t* __restrict__ ia, const T* __restrict__ Hb,
                                                  int64_t rows_b, const int32_t* __restrict__ ib,
                                                  int64_t n_max, const int64_t* __restrict__ n_dev,
                                                  const float* __restrict__ stats, float* __restrict__ part) {
  constexpr int TW = D < 128 ? D : 128;
  constexpr int TPT = TW / 16;
  constexpr int KR = 32;
  __shared__ __align__(16) float Xs[KR][TW];
  __shared__ __align__(16) float Ys[KR][TW];
  const int64_t n = count_of(n_dev, n_max);
  const int view = blockIdx.z;
  const T* H = view ? Hb : Ha;
  const int32_t* idx = view ? ib : ia;
  const int64_t rows = view ? rows_b : rows_a;
  const float* mu = stats + view * D;         // stats = [mu_a, mu_b, s_a, s_b]
  const float* sd = stats + 2 * D + view * D;
  const float rsn = n > 0 ? rsqrtf((float)n) : 0.f;
  const int tiles_per_dim = D / TW;
  const int ti = blockIdx.x / tiles_per_dim, tj = blockIdx.x % tiles_per_dim;
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
  const int64_t rows_per_split = (n + gridDim.y - 1) / gridDim.y;
  const int64_t r0 = (int64_t)blockIdx.y * rows_per_split;
  const int64_t r1 = min(n, r0 + rows_per_split);
  float acc[TPT][TPT];
#pragma unroll
  for (int i = 0; i < TPT; ++i)
#pragma unroll
    for (int j = 0; j < TPT; ++j) acc[i][j] = 0.f;
  for (int64_t rb = r0; rb < r1; rb += KR) {
    for (int e = threadIdx.x; e < KR * TW; e += blockDim.x) {
      const int k = e / TW, c = e % TW;
      float x = 0.f, y = 0.f;
      if (rb + k < r1) {
        const int64_t row = safe_row(idx, rb + k, rows);
        const int ca = ti * TW + c, cb = tj * TW + c;
        x = (to_f32(H[row * D + ca]) - mu[ca]) / sd[ca] * rsn;
        y = (to_f32(H[row * D + cb]) - mu[cb]) / sd[cb] * rsn;
      }
      Xs[k][c] = x;
      Ys[k][c] = y;
    }
    __syncthreads();
#pragma unroll 4
    for (int k = 0; k < KR; ++k) {
      float xa[TPT], yb[TPT];
#pragma unroll
      for (int i = 0; i < TPT; ++i) {
        xa[i] = Xs[k][ty * TPT + i];
        yb[i] = Ys[k][tx * TPT + i];
      }
#pragma unroll
      for (int i = 0; i < TPT; ++i)
#pragma unroll
        for (int j = 0; j < TPT; ++j) acc[i][j] = fmaf(xa[i], yb[j], acc[i][j]);
    }
    __syncthreads();
  }
  float* out = part + ((int64_t)blockIdx.y * 2 + view) * D * D;
#pragma unroll
  for (int i = 0; i < TPT; ++i)
#pragma unroll
    for (int j = 0; j < TPT; ++j) out[(int64_t)(ti * TW + ty * TPT + i) * D + tj * TW + tx * TPT + j] = acc[i][j];
}

// C[view] = sum of Gram partials in split order (count = 2 d^2 entries).
__global__ void align_gram_reduce(const float* __restrict__ part, int splits, int64_t count, float* __restrict__ C) {
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < count; i += (int64_t)gridDim.x * blockDim.x) {
    const int64_t per = count / 2;
    const int view = (int)(i / per);
    const int64_t k = i % per;
    float s = 0.f;
    for (int sp = 0; sp < splits; ++sp) s += part[((int64_t)sp * 2 + view) * per + k];
    C[i] = s;
  }
}

// One block of 1024 threads: L_dec from C, L_inv from the column sums of (z_a - z_b)^2,
// loss = [L, L_inv, L_dec]; fixed-order warp and block sums.
__global__ void __launch_bounds__(1024) align_loss_finish(const float* __restrict__ C, int d,
                                                          const float* __restrict__ cross,
                                                          const int64_t* __restrict__ n_dev, int64_t n_max,
                                                          float lambda_n, const int32_t* __restrict__ bad,
                                                          float* __restrict__ loss) {
  __shared__ float red[2][32];
  const int64_t n = count_of(n_dev, n_max);
  const int64_t dd = (int64_t)d * d;
  float s = 0.f, si = 0.f;
  for (int64_t k4 = threadIdx.x; k4 < 2 * dd / 4; k4 += blockDim.x) {
    const float4 v = reinterpret_cast<const float4*>(C)[k4];
    const float x[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int64_t e = (4 * k4 + u) % dd;
      const float c = x[u] - ((e / d) == (e % d) ? 1.f : 0.f);
      s += c * c;
    }
  }
  for (int c = threadIdx.x; c < d; c += blockDim.x) si += cross[kSumDiff2 * d + c];
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    s += __shfl_xor_sync(0xffffffffu, s, o);
    si += __shfl_xor_sync(0xffffffffu, si, o);
  }
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  if (lane == 0) {
    red[0][w] = s;
    red[1][w] = si;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float dec = 0.f, iv = 0.f;
    for (int k = 0; k < (int)(blockDim.x >> 5); ++k) {
      dec += red[0][k];
      iv += red[1][k];
    }
    if (n < 2) dec = iv = 0.f;
    if (*bad) dec = iv = __int_as_float(0x7fc00000);  // an overlap index outside its table: NaN loss
    loss[0] = iv + lambda_n * dec;
    loss[1] = iv;
    loss[2] = dec;
  }
}

// Backward, row tiles of 64 for one view (blockIdx.y): G = dloss (+-2 (z_a - z_b) + 4 lambda z (C - I)),
// stored in fp32 scratch; per-block column partials of g = G / sqrt(n) and g * x_hat.
template <typename T, int D>
__global__ void __launch_bounds__(256) align_bwd_rows(const T* __restrict__ Ha, int64_t rows_a,
                                                      const int32_t* __restrict__ ia, const T* __restrict__ Hb,
                                                      int64_t rows_b, const int32_t* __restrict__ ib,
                                                      int64_t n_max, const int64_t* __restrict__ n_dev,
                                                      const float* __restrict__ stats, const float* __restrict__ C,
                                                      float lambda_n, float dloss, float* __restrict__ G,
                                                      float* __restrict__ part) {
  using TL = Tile<float, D>;
  constexpr int RM = TL::RM, CN = TL::CN;
  constexpr int LD = D + 4;
  extern __shared__ __align__(16) float smem[];
  float* Zs = smem;            // kBM x LD
  float* Bs = Zs + kBM * LD;   // kKC x D
  float* red = Bs + kKC * D;   // 16 x 2 x D
  const int64_t n = count_of(n_dev, n_max);
  const int view = blockIdx.y;
  const int ty = threadIdx.x / 16, tx = threadIdx.x % 16;
  const float rsn = n > 0 ? rsqrtf((float)n) : 0.f;
  const float sn = sqrtf((float)n);
  const float* mu_a = stats;
  const float* mu_b = stats + D;
  const float* s_a = stats + 2 * D;
  const float* s_b = stats + 3 * D;
  const T* H = view ? Hb : Ha;
  const int32_t* idx = view ? ib : ia;
  const int64_t rows = view ? rows_b : rows_a;
  const float* mu = view ? mu_b : mu_a;
  const float* sd = view ? s_b : s_a;
  const float* Cv = C + (int64_t)view * D * D;
  const float sign = view ? -1.f : 1.f;
  float pg[CN], pgx[CN];
#pragma unroll
  for (int j = 0; j < CN; ++j) pg[j] = pgx[j] = 0.f;
  for (int64_t m0 = (int64_t)blockIdx.x * kBM; m0 < n; m0 += (int64_t)gridDim.x * kBM) {
    const int64_t nv = min((int64_t)kBM, n - m0);
    // standardised rows of this view into Zs
    for (int e = threadIdx.x; e < kBM * D; e += blockDim.x) {
      const int m = e / D, c = e % D;
      float z = 0.f;
      if (m < nv) z = (to_f32(H[safe_row(idx, m0 + m, rows) * D + c]) - mu[c]) / sd[c] * rsn;
      Zs[m * LD + c] = z;
    }
    __syncthreads();
    float acc[RM][CN];
#pragma unroll
    for (int i = 0; i < RM; ++i)
#pragma unroll
      for (int j = 0; j < CN; ++j) acc[i][j] = 0.f;
    for (int k0 = 0; k0 < D; k0 += kKC) {
      for (int e = threadIdx.x; e < kKC * D; e += blockDim.x) {
        const int k = e / D, c = e % D;
        Bs[e] = Cv[(int64_t)(k0 + k) * D + c] - ((k0 + k) == c ? 1.f : 0.f);
      }
      __syncthreads();
      mma_chunk<D, RM, CN>(Zs, LD, k0, Bs, acc);
      __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < RM; ++i) {
      const int m = ty * RM + i;
      if (m >= nv) continue;
      const int64_t ra = safe_row(ia, m0 + m, rows_a), rb = safe_row(ib, m0 + m, rows_b);
#pragma unroll
      for (int j = 0; j < CN; ++j) {
        const int c = tx * CN + j;
        const float za = (to_f32(Ha[ra * D + c]) - mu_a[c]) / s_a[c] * rsn;
        const float zb = (to_f32(Hb[rb * D + c]) - mu_b[c]) / s_b[c] * rsn;
        const float z = view ? zb : za;
        const float g = dloss * (sign * 2.f * (za - zb) + 4.f * lambda_n * acc[i][j]);
        G[((int64_t)view * n_max + m0 + m) * D + c] = g;
        const float gs = g * rsn;      // dL/dx_hat
        pg[j] += gs;
        pgx[j] += gs * (z * sn);       // x_hat = sqrt(n) z
      }
    }
  }
#pragma unroll
  for (int j = 0; j < CN; ++j) {
    red[(ty * 2 + 0) * D + tx * CN + j] = pg[j];
    red[(ty * 2 + 1) * D + tx * CN + j] = pgx[j];
  }
  __syncthreads();
  for (int k = threadIdx.x; k < 2 * D; k += blockDim.x) {
    float s = 0.f;
    for (int r = 0; r < 16; ++r) s += red[r * 2 * D + k];
    part[((int64_t)blockIdx.x * 2 + view) * 2 * D + k] = s;
  }
}

// means[view][0][c] = mean g, means[view][1][c] = mean g * x_hat (sum of block partials / n)
__global__ void align_bwd_means(const float* __restrict__ part, int blocks, int d, const int64_t* __restrict__ n_dev,
                                int64_t n_max, float* __restrict__ means) {
  const int64_t n = count_of(n_dev, n_max);
  for (int k = threadIdx.x; k < 4 * d; k += blockDim.x) {
    float s = 0.f;
    for (int b = 0; b < blocks; ++b) s += part[(int64_t)b * 4 * d + k];
    means[k] = n > 0 ? s / (float)n : 0.f;
  }
}

// dH[idx[r]] += (g - mean g - x_hat mean(g x_hat)) / s, for the views whose dH is non-null.
template <typename T>
__global__ void align_bwd_apply(const T* __restrict__ Ha, int64_t rows_a, const int32_t* __restrict__ ia,
                                const T* __restrict__ Hb, int64_t rows_b, const int32_t* __restrict__ ib, int64_t n_max,
                                const int64_t* __restrict__ n_dev, int d, const float* __restrict__ stats,
                                const float* __restrict__ G, const float* __restrict__ means,
                                const int32_t* __restrict__ bad, T* __restrict__ dHa, T* __restrict__ dHb) {
  const int64_t n = count_of(n_dev, n_max);
  if (n < 2 || *bad) return;
  const float rsn = rsqrtf((float)n);
  const int64_t total = 2 * n * d;
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < total; e += (int64_t)gridDim.x * blockDim.x) {
    const int view = (int)(e / (n * d));
    const int64_t rc = e % (n * d);
    const int64_t r = rc / d;
    const int c = (int)(rc % d);
    T* dH = view ? dHb : dHa;
    if (!dH) continue;
    const T* H = view ? Hb : Ha;
    const int64_t row = view ? safe_row(ib, r, rows_b) : safe_row(ia, r, rows_a);
    const float mu = stats[view * d + c], sd = stats[2 * d + view * d + c];
    const float xh = (to_f32(H[row * d + c]) - mu) / sd;
    const float g = G[((int64_t)view * n_max + r) * d + c] * rsn;
    const float mg = means[(view * 2 + 0) * d + c], mgx = means[(view * 2 + 1) * d + c];
    const float dx = (g - mg - xh * mgx) / sd;
    dH[row * d + c] = from_f32<T>(to_f32(dH[row * d + c]) + dx);
  }
}

// ---------------------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------------------
static int gram_splits(int64_t n_max) { return (int)std::max<int64_t>(1, std::min<int64_t>(152, ceil_div(n_max, 512))); }
static int max_gram_splits(int64_t n_max, int d) { return std::max(gram_splits(n_max), align_gram_tc_splits(n_max, d, 152)); }

struct AlignLayout {
  float* stats;   // saved: [mu_a, mu_b, s_a, s_b] (4 d)
  float* C;       // saved: [C_a, C_b] (2 d^2)
  int32_t* bad;   // saved: non-zero when an overlap index lies outside its table
  float* cross;   // saved: kNumCross column sums of z (CrossSum order, 6 d)
  float* part;    // scratch: column partials (blocks x 6 d) / fp32 backward partials (row blocks x 4 d)
  float* gpart;   // scratch: Gram partials (splits x 2 x d^2)
  float* rtmp;    // scratch: reduction temporaries
  float* G;       // scratch: fp32 backward, 2 x n_max x d
  float* means;   // scratch: 4 d
  void* cmi;      // scratch: bf16 backward operand C - I, 2 d^2 bf16
  int max_splits;
};

static void carve_saved(Carve& s, int d, AlignLayout* L) {
  L->stats = s.take<float>(4 * d);
  L->C = s.take<float>(2 * (size_t)d * d);
  L->bad = s.take<int32_t>(1);
  L->cross = s.take<float>((size_t)kNumCross * d);
}

static void carve_align(void* saved, void* scratch, int64_t n_max, int d, AlignLayout* L, size_t* sb, size_t* kb) {
  Carve s(saved), k(scratch);
  carve_saved(s, d, L);
  const int64_t rb = std::max<int64_t>(1, ceil_div(n_max, kBM));
  L->max_splits = max_gram_splits(n_max, d);
  L->part = k.take<float>(std::max<int64_t>((int64_t)kAlignBlocks * kNumCross * d, std::min<int64_t>(rb, kAlignBlocks) * 4 * d));
  L->gpart = k.take<float>((size_t)L->max_splits * 2 * d * d);
  L->rtmp = k.take<float>(reduce_tmp_floats(L->max_splits, (int64_t)d * d));
  L->G = k.take<float>(2 * std::max<int64_t>(n_max, 1) * d);
  L->means = k.take<float>(4 * d);
  L->cmi = k.take<__nv_bfloat16>(2 * (size_t)d * d);
  if (sb) *sb = s.used;
  if (kb) *kb = k.used;
}

struct AlignIn {
  const void* Ha;
  int64_t rows_a;
  const int32_t* ia;
  const void* Hb;
  int64_t rows_b;
  const int32_t* ib;
  int64_t n_max;
  const int64_t* n_dev;
};

static hg_status check_align_args(const AlignIn& in, int32_t d, hg_dtype dt, const void* saved, const void* scratch) {
  HG_REQUIRE(in.n_max >= 0, "n_max must be >= 0");
  HG_REQUIRE(in.n_max < (int64_t(1) << 31), "n_max must be < 2^31");
  HG_REQUIRE(in.n_max == 0 || (in.Ha && in.ia && in.Hb && in.ib), "H_a, idx_a, H_b, idx_b must be non-null");
  HG_REQUIRE(in.n_max == 0 || (in.rows_a > 0 && in.rows_b > 0), "rows_a and rows_b must be > 0 when n_max > 0");
  HG_REQUIRE(saved && scratch, "saved and scratch must be non-null");
  HG_REQUIRE(((uintptr_t)saved & 255) == 0 && ((uintptr_t)scratch & 255) == 0, "buffers must be 256-byte aligned");
  if (!(d == 64 || d == 128 || d == 256) || !(dt == HG_F32 || dt == HG_BF16)) {
    set_error("unsupported d=%d / dtype=%d", d, (int)dt);
    return HG_ERR_UNSUPPORTED;
  }
  return HG_OK;
}

// The loss (both entry points): three column passes (mean, variance, the sums of z), the Gram
// partials of both views over `splits` row ranges, their fixed-order reduction and the loss.
template <typename T, int D>
static hg_status align_loss_run(const AlignIn& in, float lambda_n, float eps, float* loss, const AlignLayout& L,
                                int splits, cudaStream_t s) {
  constexpr int RPP = 256 / (D / VecTraits<T>::kElems);
  const int blocks = (int)std::max<int64_t>(1, std::min<int64_t>(kAlignBlocks, ceil_div(in.n_max, RPP)));
  const T* Ha = (const T*)in.Ha;
  const T* Hb = (const T*)in.Hb;
  const float* no_stats = nullptr;
  HG_CUDA(cudaMemsetAsync(L.bad, 0, sizeof(int32_t), s));
  HG_TRY(launch("align_colstats", align_colstats<T, D, 0>, dim3(blocks), dim3(256), 0, s, Ha, in.rows_a, in.ia, Hb,
                in.rows_b, in.ib, in.n_max, in.n_dev, no_stats, L.part, L.bad));
  HG_TRY(reduce_partials(L.part, 2LL * D, blocks, 2LL * D, L.stats, L.rtmp, s));
  HG_TRY(launch("align_colscale", align_colscale, dim3((unsigned)ceil_div(2 * D, 256)), dim3(256), 0, s, L.stats,
                2 * D, in.n_dev, in.n_max, 0, 0.f));
  HG_TRY(launch("align_colstats", align_colstats<T, D, 1>, dim3(blocks), dim3(256), 0, s, Ha, in.rows_a, in.ia, Hb,
                in.rows_b, in.ib, in.n_max, in.n_dev, (const float*)L.stats, L.part, L.bad));
  HG_TRY(reduce_partials(L.part, 2LL * D, blocks, 2LL * D, L.stats + 2 * D, L.rtmp, s));
  HG_TRY(launch("align_colscale", align_colscale, dim3((unsigned)ceil_div(2 * D, 256)), dim3(256), 0, s,
                L.stats + 2 * D, 2 * D, in.n_dev, in.n_max, 1, eps));
  HG_TRY(launch("align_colstats", align_colstats<T, D, 2>, dim3(blocks), dim3(256), 0, s, Ha, in.rows_a, in.ia, Hb,
                in.rows_b, in.ib, in.n_max, in.n_dev, (const float*)L.stats, L.part, L.bad));
  HG_TRY(reduce_partials(L.part, (int64_t)kNumCross * D, blocks, (int64_t)kNumCross * D, L.cross, L.rtmp, s));
  if constexpr (std::is_same<T, __nv_bfloat16>::value) {
    HG_TRY(align_gram_tc(D, in.Ha, in.rows_a, in.ia, in.Hb, in.rows_b, in.ib, in.n_max, in.n_dev, L.stats, splits,
                         L.gpart, s));
  } else {
    constexpr int TW = D < 128 ? D : 128;
    const int tiles = (D / TW) * (D / TW);
    HG_TRY(launch("align_gram", align_gram<T, D>, dim3(tiles, splits, 2), dim3(256), 0, s, Ha, in.rows_a, in.ia, Hb,
                  in.rows_b, in.ib, in.n_max, in.n_dev, (const float*)L.stats, L.gpart));
  }
  for (int v = 0; v < 2; ++v)
    HG_TRY(reduce_partials(L.gpart + (size_t)v * D * D, 2LL * D * D, splits, (int64_t)D * D, L.C + (size_t)v * D * D,
                           L.rtmp, s));
  return launch("align_loss_finish", align_loss_finish, dim3(1), dim3(1024), 0, s, (const float*)L.C, D,
                (const float*)L.cross, in.n_dev, in.n_max, lambda_n, (const int32_t*)L.bad, loss);
}

template <typename T, int D>
static hg_status align_loss_t(const AlignIn& in, float lambda_n, float eps, float* loss, AlignLayout& L,
                              cudaStream_t s) {
  const int splits = std::is_same<T, __nv_bfloat16>::value ? align_gram_tc_splits(in.n_max, D, L.max_splits)
                                                           : std::min(gram_splits(in.n_max), L.max_splits);
  return align_loss_run<T, D>(in, lambda_n, eps, loss, L, splits, s);
}

template <typename T, int D>
static hg_status align_bwd_t(const AlignIn& in, float lambda_n, float dloss, void* dHa, void* dHb, AlignLayout& L,
                             cudaStream_t s) {
  if (in.n_max == 0 || (!dHa && !dHb)) return HG_OK;
  if constexpr (std::is_same<T, __nv_bfloat16>::value) {
    return align_bwd_tc(D, in.Ha, in.rows_a, in.ia, in.Hb, in.rows_b, in.ib, in.n_max, in.n_dev, L.stats, L.C,
                        L.cross, L.bad, lambda_n, dloss, L.cmi, L.means, dHa, dHb, s);
  } else {
    const size_t smem = sizeof(float) * (kBM * (D + 4) + kKC * D + 16 * 2 * D);
    static bool attr = false;
    if (!attr) {
      HG_CUDA(cudaFuncSetAttribute(align_bwd_rows<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem));
      attr = true;
    }
    const T* Ha = (const T*)in.Ha;
    const T* Hb = (const T*)in.Hb;
    const int rblocks = (int)std::max<int64_t>(1, std::min<int64_t>(ceil_div(in.n_max, kBM), kAlignBlocks));
    HG_TRY(launch("align_bwd_rows", align_bwd_rows<T, D>, dim3(rblocks, 2), dim3(256), smem, s, Ha, in.rows_a, in.ia,
                  Hb, in.rows_b, in.ib, in.n_max, in.n_dev, (const float*)L.stats, (const float*)L.C, lambda_n, dloss,
                  L.G, L.part));
    HG_TRY(launch("align_bwd_means", align_bwd_means, dim3(1), dim3(256), 0, s, (const float*)L.part, rblocks, D,
                  in.n_dev, in.n_max, L.means));
    const unsigned g = (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(2 * in.n_max * D, 256), 152 * 16));
    return launch("align_bwd_apply", align_bwd_apply<T>, dim3(g), dim3(256), 0, s, Ha, in.rows_a, in.ia, Hb,
                  in.rows_b, in.ib, in.n_max, in.n_dev, D, (const float*)L.stats, (const float*)L.G,
                  (const float*)L.means, (const int32_t*)L.bad, (T*)dHa, (T*)dHb);
  }
}

#define HG_DISPATCH_ALIGN(dtype, d, FN, ...)                                                \
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

static hg_status align_loss_dispatch(hg_dtype dt, int d, const AlignIn& in, float lambda_n, float eps, float* loss,
                                     AlignLayout& L, cudaStream_t s) {
  HG_DISPATCH_ALIGN(dt, d, align_loss_t, in, lambda_n, eps, loss, L, s);
}

static hg_status align_bwd_dispatch(hg_dtype dt, int d, const AlignIn& in, float lambda_n, float dloss, void* dHa,
                                    void* dHb, AlignLayout& L, cudaStream_t s) {
  HG_DISPATCH_ALIGN(dt, d, align_bwd_t, in, lambda_n, dloss, dHa, dHb, L, s);
}

}  // namespace hg

using namespace hg;

extern "C" hg_status hg_overlap_intersect_workspace_size(int64_t n_a, int64_t n_b, size_t* bytes) {
  clear_error();
  HG_REQUIRE(bytes && n_a >= 0 && n_b >= 0, "bytes must be non-null and sizes >= 0");
  HG_REQUIRE(n_a < (int64_t(1) << 31) && n_b < (int64_t(1) << 31), "lists must hold < 2^31 ids");
  Carve c(nullptr);
  c.take<int32_t>(n_a + 1);
  c.take<int32_t>(n_a + 1);
  c.take<int32_t>(n_a + 1);
  c.take<int32_t>(1);
  c.take<char>(scan_scratch_bytes(n_a));
  *bytes = c.used;
  return HG_OK;
}

extern "C" hg_status hg_overlap_intersect(const int64_t* gid_a, int64_t n_a, const int64_t* gid_b, int64_t n_b,
                                          int32_t* idx_a, int32_t* idx_b, int64_t* n_out, void* scratch,
                                          size_t scratch_bytes, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  size_t need = 0;
  HG_TRY(hg_overlap_intersect_workspace_size(n_a, n_b, &need));
  HG_REQUIRE(n_out && scratch, "n_out and scratch must be non-null");
  HG_REQUIRE((n_a == 0 || (gid_a && idx_a && idx_b)) && (n_b == 0 || gid_b), "id and index arrays must be non-null");
  HG_REQUIRE(((uintptr_t)scratch & 255) == 0, "scratch must be 256-byte aligned");
  if (scratch_bytes < need) {
    set_error("scratch has %zu bytes, %zu needed", scratch_bytes, need);
    return HG_ERR_WORKSPACE;
  }
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  Carve c(scratch);
  int32_t* flag = c.take<int32_t>(n_a + 1);
  int32_t* pos = c.take<int32_t>(n_a + 1);
  int32_t* ofs = c.take<int32_t>(n_a + 1);
  int32_t* bad = c.take<int32_t>(1);
  void* sc = c.take<char>(scan_scratch_bytes(n_a));
  HG_CUDA(cudaMemsetAsync(bad, 0, sizeof(int32_t), s));
  const unsigned g = (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(std::max(n_a, n_b), 256), 152 * 16));
  if (n_a > 0 || n_b > 0)
    HG_TRY(launch("intersect_flags", intersect_flags, dim3(g), dim3(256), 0, s, gid_a, n_a, gid_b, n_b, flag, pos, bad));
  HG_TRY(exclusive_scan(flag, ofs, n_a, sc, s));
  return launch("intersect_write", intersect_write, dim3(g), dim3(256), 0, s, (const int32_t*)flag,
                (const int32_t*)pos, (const int32_t*)ofs, n_a, std::min(n_a, n_b), (const int32_t*)bad, idx_a,
                idx_b, n_out);
}

extern "C" hg_status hg_overlap_align_workspace_size(int64_t n_max, int32_t d, size_t* saved_bytes,
                                                     size_t* scratch_bytes) {
  clear_error();
  HG_REQUIRE(saved_bytes && scratch_bytes && n_max >= 0 && d > 0, "bad arguments");
  AlignLayout L;
  carve_align(nullptr, nullptr, n_max, d, &L, saved_bytes, scratch_bytes);
  return HG_OK;
}

extern "C" hg_status hg_overlap_align_loss(const void* H_a, int64_t rows_a, const int32_t* idx_a, const void* H_b,
                                           int64_t rows_b, const int32_t* idx_b, int64_t n_max, const int64_t* n_dev,
                                           int32_t d, hg_dtype dtype, float lambda_n, float var_eps, float* loss_out,
                                           void* saved, void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  const AlignIn in{H_a, rows_a, idx_a, H_b, rows_b, idx_b, n_max, n_dev};
  HG_TRY(check_align_args(in, d, dtype, saved, scratch));
  HG_REQUIRE(loss_out != nullptr, "loss_out must be non-null");
  HG_REQUIRE(lambda_n >= 0.f && var_eps >= 0.f, "lambda_n and var_eps must be >= 0");
  AlignLayout L;
  carve_align(saved, scratch, n_max, d, &L, nullptr, nullptr);
  return align_loss_dispatch(dtype, d, in, lambda_n, var_eps, loss_out, L, reinterpret_cast<cudaStream_t>(stream));
}

extern "C" hg_status hg_overlap_align_bwd(const void* H_a, int64_t rows_a, const int32_t* idx_a, const void* H_b,
                                          int64_t rows_b, const int32_t* idx_b, int64_t n_max, const int64_t* n_dev,
                                          int32_t d, hg_dtype dtype, float lambda_n, float var_eps, float dloss,
                                          const void* saved, void* dH_a, void* dH_b, void* scratch, hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  (void)var_eps;  // s = sqrt(var + eps) is part of `saved`
  const AlignIn in{H_a, rows_a, idx_a, H_b, rows_b, idx_b, n_max, n_dev};
  HG_TRY(check_align_args(in, d, dtype, saved, scratch));
  AlignLayout L;
  carve_align(const_cast<void*>(saved), scratch, n_max, d, &L, nullptr, nullptr);
  return align_bwd_dispatch(dtype, d, in, lambda_n, dloss, dH_a, dH_b, L, reinterpret_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------------------------------------
// Allocation-free variant of hg_overlap_align_loss.
//
// Some callers cannot hand this library a scratch buffer: a host program that links only this C
// ABI and owns no CUDA allocator, a serving process whose device memory is entirely reserved by
// another framework's caching allocator, or code for which cudaMalloc is off limits because it can
// synchronise the device.  This variant runs the same kernels with their scratch in a file-scope
// device array of kStaticAlignBytes (every GPU that loads the library holds it until exit), so
// the caller passes only inputs and outputs.  The array's device address is looked up once per
// device, on the first call made with that device current (that first call should therefore come
// before any stream capture).  All calls share the array: calls that overlap on the GPU race, and
// each call leaves its partial sums behind.  Nothing needs zeroing first: every scratch element a
// kernel reads has been written earlier in the same call.
// ---------------------------------------------------------------------------------------------
#include <mutex>

namespace hg {

constexpr int kStaticGramSplits = 16;                        // row splits of the Gram products
constexpr size_t kStaticAlignBytes = size_t(12) << 20;      // 12 MiB: d <= 256 at 16 splits
static __device__ __align__(256) unsigned char g_align_static_scratch[kStaticAlignBytes];

constexpr int kStaticMaxDevices = 64;
static std::mutex g_static_mu;
static void* g_static_addr[kStaticMaxDevices] = {};

static hg_status static_align_scratch(void** out) {
  int dev = 0;
  HG_CUDA(cudaGetDevice(&dev));
  if (dev < 0 || dev >= kStaticMaxDevices) {
    set_error("device %d is beyond the %d devices this entry point tracks", dev, kStaticMaxDevices);
    return HG_ERR_UNSUPPORTED;
  }
  std::lock_guard<std::mutex> lk(g_static_mu);
  if (!g_static_addr[dev]) {
    void* p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_align_static_scratch);
    if (e != cudaSuccess || p == nullptr) {
      set_error("cudaGetSymbolAddress of the static alignment scratch failed: %s", cudaGetErrorString(e));
      return HG_ERR_CUDA;
    }
    g_static_addr[dev] = p;
  }
  *out = g_static_addr[dev];
  return HG_OK;
}

// Layout of the static scratch for width d: column partials, Gram partials, reduction temporaries.
static size_t carve_static(void* base, int d, AlignLayout* L) {
  Carve k(base);
  L->part = k.take<float>((size_t)kAlignBlocks * kNumCross * d);
  L->gpart = k.take<float>((size_t)kStaticGramSplits * 2 * d * d);
  L->rtmp = k.take<float>(reduce_tmp_floats(kStaticGramSplits, (int64_t)d * d));
  L->max_splits = kStaticGramSplits;
  return k.used;
}

template <typename T, int D>
static hg_status align_loss_static_t(const AlignIn& in, float lambda_n, float eps, float* loss, const AlignLayout& L,
                                     cudaStream_t s) {
  const int splits = std::is_same<T, __nv_bfloat16>::value ? align_gram_tc_splits(in.n_max, D, kStaticGramSplits)
                                                           : std::min(gram_splits(in.n_max), kStaticGramSplits);
  return align_loss_run<T, D>(in, lambda_n, eps, loss, L, splits, s);
}

}  // namespace hg

extern "C" hg_status hg_overlap_align_loss_static(const void* H_a, int64_t rows_a, const int32_t* idx_a,
                                                  const void* H_b, int64_t rows_b, const int32_t* idx_b,
                                                  int64_t n_max, const int64_t* n_dev, int32_t d, hg_dtype dtype,
                                                  float lambda_n, float var_eps, float* loss_out, void* saved,
                                                  hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  const AlignIn in{H_a, rows_a, idx_a, H_b, rows_b, idx_b, n_max, n_dev};
  void* scratch = nullptr;
  HG_TRY(static_align_scratch(&scratch));
  HG_TRY(check_align_args(in, d, dtype, saved, scratch));
  HG_REQUIRE(loss_out != nullptr, "loss_out must be non-null");
  HG_REQUIRE(lambda_n >= 0.f && var_eps >= 0.f, "lambda_n and var_eps must be >= 0");
  AlignLayout L{};
  const size_t need = carve_static(nullptr, d, &L);
  if (need > kStaticAlignBytes) {
    set_error("d=%d needs %zu bytes of scratch, beyond the %zu-byte static array of this entry point", d, need,
              kStaticAlignBytes);
    return HG_ERR_UNSUPPORTED;
  }
  carve_static(scratch, d, &L);
  Carve sv(saved);  // the `saved` part (statistics, Gram matrices, index flag, column sums)
  carve_saved(sv, d, &L);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
#define HG_STATIC_CASE(T, D_)                                                                                \
  if (d == D_) return align_loss_static_t<T, D_>(in, lambda_n, var_eps, loss_out, L, s);
  if (dtype == HG_F32) {
    HG_STATIC_CASE(float, 64)
    HG_STATIC_CASE(float, 128)
    HG_STATIC_CASE(float, 256)
  } else {
    HG_STATIC_CASE(__nv_bfloat16, 64)
    HG_STATIC_CASE(__nv_bfloat16, 128)
    HG_STATIC_CASE(__nv_bfloat16, 256)
  }
#undef HG_STATIC_CASE
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}
