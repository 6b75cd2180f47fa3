// Tensor-core kernels of the bf16 alignment path (Section 3.3, Eq. 14-17).
//
// Gram matrices C_v = Z_v^T Z_v (Eq. 16): the standardised overlap rows never exist in global
// memory.  The 128 threads of a CTA gather 64 overlap rows of H_v at a time (coalesced 16-byte
// pieces), standardise them, round them to bf16 and write them into a 128-byte-swizzled stage in
// shared memory, which is both MN-major operands of one tcgen05.mma chain (A = Z^T, B = Z, K = the
// 64 rows); the fp32 accumulator stays in tensor memory across all the row chunks of the CTA's
// split, and the split's partial Gram matrix is written once at the end.
//
// Gradient (Eq. 15-17): with P_v = Z_v (C_v - I),
//   G_a = dloss (2 (Z_a - Z_b) + 4 lambda P_a),   G_b = dloss (-2 (Z_a - Z_b) + 4 lambda P_b)
// and the standardisation's backward dX = (g - mean g - x_hat mean(g x_hat)) / s, g = G / sqrt(n).
// The two column means need no pass over the rows:
//   sum_r P_v[r,c]         = sum_k (sum_r z_v[r,k]) (C_v - I)[k,c]
//   sum_r P_v[r,c] z_v[r,c] = sum_k (C_v - I)[k,c] C_v[k,c]
// and the rest are the column sums kept by the loss (align_bwd_coef).  align_bwd_tc then makes one
// pass: per 128 rows it builds the bf16 Z_v tile in shared memory, multiplies it by (C_v - I)
// (bf16, TMA) on the tensor cores, stages P through shared memory and applies dX to dH_v with
// coalesced loads and stores; Z_a - Z_b is formed in fp32 from H.
#include <algorithm>

#include "align_kernels.cuh"
#include "layer_kernels.cuh"
#include "tc_util.cuh"

namespace hg {

using namespace tc;

namespace {

constexpr int kThreads = 128;
constexpr int kBlk = 64 * 128;  // 64 rows x 64 bf16, 128B-swizzled

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

// z = (x - mu) * k for eight columns, k = 1 / (s sqrt(n)).
__device__ __forceinline__ uint4 standardise8(uint4 raw, const float* mu, const float* k) {
  float x[8];
  unpack(raw, x, __nv_bfloat16());
#pragma unroll
  for (int i = 0; i < 8; ++i) x[i] = (x[i] - mu[i]) * k[i];
  return pack(x, __nv_bfloat16());
}

template <int D>
struct GramCfg {
  static constexpr int NB = D / 64;                // 64-column blocks of a stage
  static constexpr int kBlocks = NB < 2 ? 2 : NB;  // d = 64: a zero block lets A span M = 128
  static constexpr int kStage = kBlocks * kBlk;
  static constexpr int kStages = 4;
  static constexpr int kSmem = kStages * kStage + 256 + 1024;
  static constexpr int kTmemCols = D;
};

// grid (M tiles of 128 Gram rows, splits, 2 views); 128 threads.
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    align_gram_tc_kernel(const __nv_bfloat16* __restrict__ Ha, int64_t rows_a, const int32_t* __restrict__ ia,
                         const __nv_bfloat16* __restrict__ Hb, int64_t rows_b, const int32_t* __restrict__ ib,
                         int64_t n_max, const int64_t* __restrict__ n_dev, const float* __restrict__ stats,
                         float* __restrict__ part, int* __restrict__ status) {
  using C = GramCfg<D>;
  constexpr int S = C::kStages;
  constexpr int TPR = D / 8;             // 16-byte pieces per row
  constexpr int RPP = kThreads / TPR;    // rows per producer pass
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * C::kStage);
  uint64_t* empty = full + S;
  uint64_t* accb = empty + S;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x, view = blockIdx.z;
  const int64_t n = count_of(n_dev, n_max);
  const int64_t nchunks = (n + 63) / 64;  // the splits share the rows in use, not n_max
  const int64_t chunks_per_split = (nchunks + gridDim.y - 1) / gridDim.y;
  const int64_t c0 = (int64_t)blockIdx.y * chunks_per_split;
  const int CT = (int)max((int64_t)0, min(nchunks, c0 + chunks_per_split) - c0);
  const __nv_bfloat16* H = view ? Hb : Ha;
  const int32_t* idx = view ? ib : ia;
  const int64_t rows = view ? rows_b : rows_a;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], kThreads);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accb, 1);
    fence_mbar_init();
  }
  if (C::NB < 2) {  // the zero block of every stage
    for (int s = 0; s < S; ++s)
      for (int e = threadIdx.x; e < kBlk / 16; e += kThreads)
        st16(smem + s * C::kStage + kBlk + e * 16, make_uint4(0, 0, 0, 0));
  }
  if (warp == 0) tmem_alloc(tslot, C::kTmemCols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;

  const int g = threadIdx.x % TPR, sub = threadIdx.x / TPR;
  float mu[8], k[8];
  {
    const float rsn = n > 0 ? rsqrtf((float)n) : 0.f;
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      mu[i] = stats[view * D + g * 8 + i];
      k[i] = rsn / stats[2 * D + view * D + g * 8 + i];
    }
  }
  const uint32_t idesc = idesc_bf16(128, D, true, true);
  bool ok = true;
  for (int it = 0; it < CT && ok; ++it) {
    const int s = it % S;
    if (it >= S) ok = mbar_wait(&empty[s], ((it / S) - 1) & 1);
    if (!ok) break;
    uint8_t* stage = smem + s * C::kStage;
    const int64_t rb = (c0 + it) * 64;
    constexpr int RT = 64 / RPP;  // rows of this thread in the chunk, all loads in flight together
    uint4 v[RT];
#pragma unroll
    for (int p = 0; p < RT; ++p) {
      const int64_t r = rb + sub + p * RPP;
      v[p] = r < n ? ldg16(H + safe_row(idx, r, rows) * D + g * 8) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int p = 0; p < RT; ++p) {
      const int rl = sub + p * RPP;
      st16(stage + (g >> 3) * kBlk + sw128_offset(rl, (g & 7) * 16),
           rb + rl < n ? standardise8(v[p], mu, k) : make_uint4(0, 0, 0, 0));
    }
    fence_async_smem();
    mbar_arrive(&full[s]);
    if (threadIdx.x == 0) {
      ok = mbar_wait(&full[s], (it / S) & 1);
      if (ok) {
        fence_after_sync();
        const uint32_t B = smem_u32(stage);
        const uint32_t A = B + 2 * mt * kBlk;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
          mma_bf16(tmem, desc_sw128(A + ks * 2048, kBlk, 1024), desc_sw128(B + ks * 2048, kBlk, 1024), idesc,
                   (it > 0 || ks > 0) ? 1u : 0u);
        mma_commit(&empty[s]);
      }
    }
  }
  if (!ok) atomicOr(status, kErrTimeout);
  if (threadIdx.x == 0) mma_commit(accb);
  if (!mbar_wait(accb, 0)) atomicOr(status, kErrTimeout);
  fence_after_sync();
  const int orow = mt * 128 + warp * 32 + lane;  // Gram row (column of Z)
  float* out = part + ((int64_t)blockIdx.y * 2 + view) * D * D;
#pragma unroll 1
  for (int c = 0; c < D; c += 16) {
    float v[16];
    if (CT > 0) {
      tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + c, v);
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = 0.f;
    }
    if (orow < D) {
#pragma unroll
      for (int i = 0; i < 16; i += 4)
        *reinterpret_cast<float4*>(out + (int64_t)orow * D + c + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

// Grid (2 views, D / 32 column slices), 256 threads: per column c the means of g and g x_hat (the
// sums over k split over the eight warps, k = w, w + 8, ..., then added in warp order), and the
// slice's rows of the bf16 operand cmi[v][c][k] = C_v[k][c] - [k == c] of the gradient's product.
template <int D>
__global__ void __launch_bounds__(256) align_bwd_coef(const float* __restrict__ Cm, const float* __restrict__ cross,
                                                      const int64_t* __restrict__ n_dev, int64_t n_max,
                                                      float lambda_n, float dloss, __nv_bfloat16* __restrict__ cmi,
                                                      float* __restrict__ means) {
  __shared__ float red[2][8][33];
  const int view = blockIdx.x, lane = threadIdx.x & 31, w = threadIdx.x >> 5;
  const int c = blockIdx.y * 32 + lane;
  const int64_t n = count_of(n_dev, n_max);
  const float* Cv = Cm + (int64_t)view * D * D;
  const float* Sv = cross + (view ? kSumZb : kSumZa) * D;
  float sp = 0.f, spz = 0.f;
  for (int kk = w; kk < D; kk += 8) {
    const float cv = Cv[(int64_t)kk * D + c];
    const float cm = cv - (kk == c ? 1.f : 0.f);
    sp += Sv[kk] * cm;
    spz += cm * cv;
  }
  red[0][w][lane] = sp;
  red[1][w][lane] = spz;
  __syncthreads();
  if (w == 0) {
    sp = spz = 0.f;
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      sp += red[0][k][lane];
      spz += red[1][k][lane];
    }
    const float sign = view ? -1.f : 1.f;
    const float dz = cross[kSumZa * D + c] - cross[kSumZb * D + c];
    const float dzz = view ? cross[kSumZaZb * D + c] - cross[kSumZb2 * D + c]
                           : cross[kSumZa2 * D + c] - cross[kSumZaZb * D + c];
    const float sum_g = dloss * (sign * 2.f * dz + 4.f * lambda_n * sp);
    const float sum_gz = dloss * (sign * 2.f * dzz + 4.f * lambda_n * spz);
    const float rn = n > 0 ? 1.f / (float)n : 0.f;
    means[(view * 2 + 0) * D + c] = (n > 0 ? rsqrtf((float)n) : 0.f) * sum_g * rn;
    means[(view * 2 + 1) * D + c] = sum_gz * rn;
  }
  for (int e = threadIdx.x; e < 32 * D; e += blockDim.x) {  // rows c0 .. c0+31 of cmi[view]
    const int cl = e / D, kk = e % D;
    const int cc = blockIdx.y * 32 + cl;
    cmi[((int64_t)view * D + cc) * D + kk] = __float2bfloat16_rn(Cv[(int64_t)kk * D + cc] - (kk == cc ? 1.f : 0.f));
  }
}

template <int D>
struct ABwdCfg {
  static constexpr int KC = D / 64;
  static constexpr int kB = KC * D * 128;    // C - I: D rows (N) x D (K), 64-column blocks of D x 128 B, resident
  static constexpr int kA = KC * 128 * 128;  // Z tile: 128 rows x D, K-major, 64-column blocks of 16 KB
  static constexpr int kPCols = 32;          // P staged through shared memory 32 columns at a time
  static constexpr int kPLd = kPCols + 4;    // padded fp32 rows (conflict-free 16-byte accesses)
  static constexpr int kP = 128 * kPLd * 4;  // reuses the Z tile once the product is in TMEM
  static constexpr int kAP = kA > kP ? kA : kP;
  static constexpr int kRows = 2 * 128 * 8;  // table rows of the tile's overlap rows, both views (int64)
  static constexpr int kSmem = kB + kAP + kRows + 256 + 1024;
  static constexpr int kTmemCols = D;
};

// grid (row tiles of 128 over n_max, 2 views); 128 threads.  Tiles past the device count exit at
// once, so the grid may be sized by a capacity far above the rows in use.
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    align_bwd_tc_kernel(const __grid_constant__ CUtensorMap tm_cmi, const __nv_bfloat16* __restrict__ Ha,
                        int64_t rows_a, const int32_t* __restrict__ ia, const __nv_bfloat16* __restrict__ Hb,
                        int64_t rows_b, const int32_t* __restrict__ ib, int64_t n_max,
                        const int64_t* __restrict__ n_dev, const float* __restrict__ stats,
                        const int32_t* __restrict__ bad, const float* __restrict__ means, float lambda_n, float dloss,
                        __nv_bfloat16* __restrict__ dHa, __nv_bfloat16* __restrict__ dHb, int* __restrict__ status) {
  using C = ABwdCfg<D>;
  constexpr int KC = C::KC;
  constexpr int TPR = D / 8;
  constexpr int RPP = kThreads / TPR;
  constexpr int PPR = C::kPCols / 8;       // 16-byte pieces per row in a P pass
  constexpr int PRP = kThreads / PPR;      // rows per P-pass step
  const int view = blockIdx.y;
  const int64_t n = count_of(n_dev, n_max);
  const int64_t m0 = (int64_t)blockIdx.x * 128;
  __nv_bfloat16* dH = view ? dHb : dHa;
  if (m0 >= n || n < 2 || *bad || dH == nullptr) return;  // uniform over the CTA
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Bt = smem;
  uint8_t* At = smem + C::kB;
  float* Ps = reinterpret_cast<float*>(At);
  int64_t* rowa = reinterpret_cast<int64_t*>(At + C::kAP);
  int64_t* rowb = rowa + 128;
  uint64_t* bbar = reinterpret_cast<uint64_t*>(rowb + 128);
  uint64_t* accb = bbar + 1;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  const int warp = threadIdx.x >> 5;
  const __nv_bfloat16* H = view ? Hb : Ha;
  const float rsn = rsqrtf((float)n);

  if (threadIdx.x == 0) {
    mbar_init(bbar, 1);
    mbar_init(accb, 1);
    fence_mbar_init();
    prefetch_tmap(&tm_cmi);
    mbar_expect_tx(bbar, C::kB);
    for (int kc = 0; kc < KC; ++kc) tma_load_2d(Bt + kc * D * 128, &tm_cmi, kc * 64, view * D, bbar);
  }
  if (warp == 0) tmem_alloc(tslot, C::kTmemCols);
  {  // table rows of the tile (clamped)
    const int64_t r = m0 + threadIdx.x;
    rowa[threadIdx.x] = r < n ? safe_row(ia, r, rows_a) : 0;
    rowb[threadIdx.x] = r < n ? safe_row(ib, r, rows_b) : 0;
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);

  // the bf16 Z_v tile (K-major, 128B-swizzled), rows past n zero
  {
    const int64_t* rowv = view ? rowb : rowa;
    const int g = threadIdx.x % TPR, sub = threadIdx.x / TPR;
    float zmu[8], zk[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      zmu[i] = stats[view * D + g * 8 + i];
      zk[i] = rsn / stats[2 * D + view * D + g * 8 + i];
    }
    constexpr int RT = 128 / RPP;
    constexpr int RB = RT < 8 ? RT : 8;  // loads in flight per batch
#pragma unroll 1
    for (int p0 = 0; p0 < RT; p0 += RB) {
      uint4 v[RB];
#pragma unroll
      for (int q = 0; q < RB; ++q) {
        const int rl = sub + (p0 + q) * RPP;
        v[q] = m0 + rl < n ? ldg16(H + rowv[rl] * D + g * 8) : make_uint4(0, 0, 0, 0);
      }
#pragma unroll
      for (int q = 0; q < RB; ++q) {
        const int rl = sub + (p0 + q) * RPP;
        st16(At + (g >> 3) * (128 * 128) + sw128_offset(rl, (g & 7) * 16),
             m0 + rl < n ? standardise8(v[q], zmu, zk) : make_uint4(0, 0, 0, 0));
      }
    }
  }
  fence_async_smem();
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  if (threadIdx.x == 0) {
    if (mbar_wait(bbar, 0)) {
      const uint32_t idesc = idesc_bf16(128, D, false, false);
      const uint32_t A = smem_u32(At), B = smem_u32(Bt);
#pragma unroll
      for (int kc = 0; kc < KC; ++kc)
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
          mma_bf16(tmem, desc_sw128(A + kc * (128 * 128) + ks * 32, 16, 1024),
                   desc_sw128(B + kc * (D * 128) + ks * 32, 16, 1024), idesc, (kc > 0 || ks > 0) ? 1u : 0u);
    } else {
      atomicOr(status, kErrTimeout);
      mbar_wait(bbar, 0);  // give-up path: the weight load still lands before the CTA moves on
    }
    mma_commit(accb);
  }
  if (!mbar_wait(accb, 0)) atomicOr(status, kErrTimeout);
  fence_after_sync();

  // dX = (g / sqrt(n) - mean g - x_hat mean(g x_hat)) / s, g = dloss (+-2 (z_a - z_b) + 4 lambda P)
  const float* mu_a = stats;
  const float* mu_b = stats + D;
  const float* s_a = stats + 2 * D;
  const float* s_b = stats + 3 * D;
  const float* mg_v = means + (view * 2 + 0) * D;
  const float* mgx_v = means + (view * 2 + 1) * D;
  const float two_sign_dloss = (view ? -2.f : 2.f) * dloss;
  const float p_scale = 4.f * lambda_n * dloss;
  const int pg = threadIdx.x % PPR, psub = threadIdx.x / PPR;
#pragma unroll 1
  for (int c0p = 0; c0p < D; c0p += C::kPCols) {
    __syncthreads();  // the Z tile (first pass) or the previous staging is no longer read
#pragma unroll
    for (int c = 0; c < C::kPCols; c += 16) {
      float v[16];
      tmem_ld16(trow + c0p + c, v);
      float* dst = Ps + threadIdx.x * C::kPLd + c;
#pragma unroll
      for (int i = 0; i < 16; i += 4) *reinterpret_cast<float4*>(dst + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
    __syncthreads();
    const int c0 = c0p + pg * 8;
    float ma[8], mb[8], ka[8], kb[8], iv[8], mg[8], mgx[8];  // ka, kb = 1 / (s sqrt n); iv = 1 / s_v
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      ma[i] = mu_a[c0 + i];
      mb[i] = mu_b[c0 + i];
      const float ra = 1.f / s_a[c0 + i], rb = 1.f / s_b[c0 + i];
      ka[i] = ra * rsn;
      kb[i] = rb * rsn;
      iv[i] = view ? rb : ra;
      mg[i] = mg_v[c0 + i];
      mgx[i] = mgx_v[c0 + i];
    }
    constexpr int RT = 128 / PRP;  // rows per thread in this pass
    uint4 xa4[RT], xb4[RT], d4[RT];
#pragma unroll
    for (int q = 0; q < RT; ++q) {
      const int rl = psub + q * PRP;
      if (m0 + rl < n) {
        xa4[q] = ldg16(Ha + rowa[rl] * D + c0);
        xb4[q] = ldg16(Hb + rowb[rl] * D + c0);
        d4[q] = ld16(dH + (view ? rowb[rl] : rowa[rl]) * D + c0);
      }
    }
#pragma unroll
    for (int q = 0; q < RT; ++q) {
      const int rl = psub + q * PRP;
      if (m0 + rl >= n) continue;
      float xa[8], xb[8], d[8];
      unpack(xa4[q], xa, __nv_bfloat16());
      unpack(xb4[q], xb, __nv_bfloat16());
      unpack(d4[q], d, __nv_bfloat16());
      const float* ps = Ps + rl * C::kPLd + pg * 8;
      const float4 lo = *reinterpret_cast<const float4*>(ps);
      const float4 hi = *reinterpret_cast<const float4*>(ps + 4);
      const float P[8] = {lo.x, lo.y, lo.z, lo.w, hi.x, hi.y, hi.z, hi.w};
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float za = (xa[i] - ma[i]) * ka[i];
        const float zb = (xb[i] - mb[i]) * kb[i];
        const float gv = two_sign_dloss * (za - zb) + p_scale * P[i];
        const float xh = view ? (xb[i] - mb[i]) * iv[i] : (xa[i] - ma[i]) * iv[i];
        d[i] += (gv * rsn - mg[i] - xh * mgx[i]) * iv[i];
      }
      st16(dH + (view ? rowb[rl] : rowa[rl]) * D + c0, pack(d, __nv_bfloat16()));
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

template <int D>
hg_status gram_t(const void* Ha, int64_t rows_a, const int32_t* ia, const void* Hb, int64_t rows_b, const int32_t* ib,
                 int64_t n_max, const int64_t* n_dev, const float* stats, int splits, float* part, cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    HG_CUDA(cudaFuncSetAttribute(align_gram_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 GramCfg<D>::kSmem));
    attr = true;
  }
  const int mtiles = D > 128 ? D / 128 : 1;
  return launch("align_gram_tc", align_gram_tc_kernel<D>, dim3(mtiles, splits, 2), dim3(kThreads), GramCfg<D>::kSmem,
                s, (const __nv_bfloat16*)Ha, rows_a, ia, (const __nv_bfloat16*)Hb, rows_b, ib, n_max, n_dev, stats,
                part, device_status_ptr());
}

template <int D>
hg_status bwd_t(const void* Ha, int64_t rows_a, const int32_t* ia, const void* Hb, int64_t rows_b, const int32_t* ib,
                int64_t n_max, const int64_t* n_dev, const float* stats, const float* Cm, const float* cross,
                const int32_t* bad, float lambda_n, float dloss, void* cmi, float* means, void* dHa, void* dHb,
                cudaStream_t s) {
  static bool attr = false;
  if (!attr) {
    HG_CUDA(cudaFuncSetAttribute(align_bwd_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 ABwdCfg<D>::kSmem));
    attr = true;
  }
  HG_TRY(launch("align_bwd_coef", align_bwd_coef<D>, dim3(2, D / 32), dim3(256), 0, s, Cm, cross, n_dev, n_max, lambda_n,
                dloss, (__nv_bfloat16*)cmi, means));
  CUtensorMap tm;
  HG_TRY(make_tmap_bf16(&tm, cmi, (uint64_t)2 * D, D, D));
  return launch("align_bwd_tc", align_bwd_tc_kernel<D>, dim3((unsigned)ceil_div(n_max, 128), 2), dim3(kThreads),
                ABwdCfg<D>::kSmem, s, tm, (const __nv_bfloat16*)Ha, rows_a, ia, (const __nv_bfloat16*)Hb, rows_b, ib,
                n_max, n_dev, stats, bad, (const float*)means, lambda_n, dloss, (__nv_bfloat16*)dHa,
                (__nv_bfloat16*)dHb, device_status_ptr());
}

}  // namespace

int align_gram_tc_splits(int64_t n_max, int d, int max_splits) {
  const int mtiles = d > 128 ? d / 128 : 1;
  const int64_t chunks = std::max<int64_t>(1, ceil_div(n_max, 64));
  // about 152 CTAs per view, each with at least four row chunks
  const int64_t want = std::min<int64_t>(152 / mtiles, ceil_div(chunks, 4));
  return (int)std::max<int64_t>(1, std::min<int64_t>(want, max_splits));
}

hg_status align_gram_tc(int d, const void* Ha, int64_t rows_a, const int32_t* ia, const void* Hb, int64_t rows_b,
                        const int32_t* ib, int64_t n_max, const int64_t* n_dev, const float* stats, int splits,
                        float* part, cudaStream_t s) {
  if (d == 64) return gram_t<64>(Ha, rows_a, ia, Hb, rows_b, ib, n_max, n_dev, stats, splits, part, s);
  if (d == 128) return gram_t<128>(Ha, rows_a, ia, Hb, rows_b, ib, n_max, n_dev, stats, splits, part, s);
  if (d == 256) return gram_t<256>(Ha, rows_a, ia, Hb, rows_b, ib, n_max, n_dev, stats, splits, part, s);
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}

hg_status align_bwd_tc(int d, const void* Ha, int64_t rows_a, const int32_t* ia, const void* Hb, int64_t rows_b,
                       const int32_t* ib, int64_t n_max, const int64_t* n_dev, const float* stats, const float* C,
                       const float* cross, const int32_t* bad, float lambda_n, float dloss, void* cmi, float* means,
                       void* dHa, void* dHb, cudaStream_t s) {
#define HG_ALIGN_BWD_CASE(D_)                                                                                   \
  if (d == D_)                                                                                                  \
    return bwd_t<D_>(Ha, rows_a, ia, Hb, rows_b, ib, n_max, n_dev, stats, C, cross, bad, lambda_n, dloss, cmi, \
                     means, dHa, dHb, s);
  HG_ALIGN_BWD_CASE(64)
  HG_ALIGN_BWD_CASE(128)
  HG_ALIGN_BWD_CASE(256)
#undef HG_ALIGN_BWD_CASE
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}

}  // namespace hg
