// Dense projections of the layer on the 5th-generation tensor cores (tcgen05, bf16 operands,
// fp32 accumulation in tensor memory).  Used for bf16 storage; fp32 storage stays on CUDA cores.
//
// Forward, one CTA per 128 destination rows of type t (Eq. 7 with one W_r per relation, Eq. 11):
//   phase 1  Z = sum_{r -> t} M_r W_r      A = relation means (TMA, 128 x 64 tiles), B = W_r^T chunks
//   phase 2  U = Z W_agg[t]                A = Z (written to shared memory by the epilogue), B = W_agg^T
//   epilogue U += b, stored; Y = act(U) + H_in; H_out = LayerNorm(Y); row statistics saved.
// Backward, one CTA per 128 rows of type t:
//   prologue dY = LayerNorm backward, dU = dY act'(U) -> shared memory; column partials of the
//            bias / gain / shift gradients
//   dZ = dU W_agg^T  (B = W_agg as stored: rows d_in, K = d_out)
//   dMs_r = (dZ W_r^T) / deg_r per relation r into t (B = W_r as stored)
// Weight gradients, split over rows (K = rows): dW = X^T Y with MN-major operands loaded by TMA,
// fp32 partials per split, reduced in a fixed order afterwards.
//
// Thread layout: 128 threads; thread (warp w, lane l) owns accumulator row 32 w + l (its TMEM
// lane).  Thread 0 issues every TMA load and MMA.  All waits are bounded (tc::kSpinLimit).
#include <algorithm>

#include "layer_kernels.cuh"
#include "simt_tile.cuh"
#include "tc_util.cuh"

namespace hg {

using namespace tc;

namespace {

constexpr int kThreads = 128;
constexpr int kTileRows = 128;
constexpr int kATile = kTileRows * 128;  // 128 rows x 64 bf16

template <int D>
struct FwdCfg {
  static constexpr int kStages = D == 64 ? 4 : (D == 128 ? 2 : 3);
  static constexpr int kB = D * 128;  // D rows x 64 bf16
  static constexpr int kStage = kATile + kB;
  static constexpr int kZ = kTileRows * D * 2;
  static constexpr int kSmem = kStages * kStage + kZ + 256 + 1024;
  static constexpr int kTmemCols = D < 32 ? 32 : D;
};

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

// 16 fp32 values -> bf16, stored as two 16-byte pieces into a K-major swizzled tile row.
__device__ __forceinline__ void put_tile16(uint8_t* tile, int row, int col, const float* v) {
  // col is a multiple of 16 elements; chunk of 64 columns -> separate 16 KB tile
  uint8_t* t = tile + (col >> 6) * kATile;
  const uint32_t cb = (uint32_t)(col & 63) * 2;
  uint4 lo = make_uint4(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]), pack_bf16x2(v[4], v[5]), pack_bf16x2(v[6], v[7]));
  uint4 hi = make_uint4(pack_bf16x2(v[8], v[9]), pack_bf16x2(v[10], v[11]), pack_bf16x2(v[12], v[13]),
                        pack_bf16x2(v[14], v[15]));
  *reinterpret_cast<uint4*>(t + sw128_offset(row, cb)) = lo;
  *reinterpret_cast<uint4*>(t + sw128_offset(row, cb + 16)) = hi;
}

__device__ __forceinline__ void round16(float* v) {
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] = __bfloat162float(__float2bfloat16_rn(v[i]));
}

__device__ __forceinline__ void load16_bf16(const __nv_bfloat16* p, float* v) {
  unpack(ld16(p), v, __nv_bfloat16());
  unpack(ld16(p + 8), v + 8, __nv_bfloat16());
}
__device__ __forceinline__ void store16_bf16(__nv_bfloat16* p, const float* v) {
  st16(p, pack(v, __nv_bfloat16()));
  st16(p + 8, pack(v + 8, __nv_bfloat16()));
}

// Butterfly reduction of 32 per-lane values: afterwards lane l holds the warp-wide sum of v[l]
// (fixed order, deterministic).
__device__ __forceinline__ float warp_transpose_sum(float* v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int w = 16; w >= 1; w >>= 1) {
    const bool upper = (lane & w) != 0;
#pragma unroll
    for (int i = 0; i < w; ++i) {
      const float send = upper ? v[i] : v[i + w];
      const float keep = upper ? v[i + w] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, w);
    }
  }
  return v[0];
}

}  // namespace

// ---------------------------------------------------------------------------------------------
// forward projection
// ---------------------------------------------------------------------------------------------

template <int D>
__global__ void __launch_bounds__(kThreads, 1) proj_fwd_tc(const __grid_constant__ CUtensorMap tm_M,
                                                          const __grid_constant__ CUtensorMap tm_WrelT,
                                                          const __grid_constant__ CUtensorMap tm_WaggT, TcFwdArgs a) {
  using C = FwdCfg<D>;
  constexpr int S = C::kStages;
  constexpr int KC = D / 64;  // 64-wide K chunks per D
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* stage = smem;                               // S x (A | B)
  uint8_t* ztile = smem + S * C::kStage;               // KC x 16 KB
  uint64_t* full = reinterpret_cast<uint64_t*>(ztile + C::kZ);
  uint64_t* empty = full + S;
  uint64_t* accb = empty + S;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  int* abort_flag = reinterpret_cast<int*>(tslot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t m0 = (int64_t)blockIdx.x * kTileRows;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accb, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_M);
    prefetch_tmap(&tm_WrelT);
    prefetch_tmap(&tm_WaggT);
  }
  if (warp == 0) tmem_alloc(tslot, C::kTmemCols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  const int C1 = a.nrel * KC, CT = C1 + KC;
  const uint32_t idesc = idesc_bf16(128, D, false, false);

  auto issue_load = [&](int g) {
    const int s = g % S;
    uint8_t* A = stage + s * C::kStage;
    uint8_t* B = A + kATile;
    if (g < C1) {
      const int r = g / KC, kc = g % KC;
      mbar_expect_tx(&full[s], kATile + C::kB);
      tma_load_2d(A, &tm_M, kc * 64, (int)(a.mrow0[r] + m0), &full[s]);
      tma_load_2d(B, &tm_WrelT, kc * 64, a.rel[r] * D, &full[s]);
    } else {
      mbar_expect_tx(&full[s], C::kB);
      tma_load_2d(B, &tm_WaggT, (g - C1) * 64, a.type * D, &full[s]);
    }
  };
  // consumes chunks [g0, g1): MMAs into the accumulator, refills freed stages
  auto run_chunks = [&](int g0, int g1) {
    bool ok = *abort_flag == 0;
    for (int g = g0; g < g1 && ok; ++g) {
      const int s = g % S;
      ok = mbar_wait(&full[s], (g / S) & 1);
      if (!ok) break;
      fence_after_sync();
      const uint8_t* A = g < C1 ? stage + s * C::kStage : ztile + (g - C1) * kATile;
      const uint8_t* B = stage + s * C::kStage + kATile;
#pragma unroll
      for (int ks = 0; ks < 4; ++ks) {
        const uint64_t ad = desc_sw128(smem_u32(A) + ks * 32, 16, 1024);
        const uint64_t bd = desc_sw128(smem_u32(B) + ks * 32, 16, 1024);
        mma_bf16(tmem, ad, bd, idesc, (g > g0 || ks > 0) ? 1u : 0u);
      }
      mma_commit(&empty[s]);
      if (g + S < CT) {
        ok = mbar_wait(&empty[s], (g / S) & 1);
        if (ok) issue_load(g + S);
      }
    }
    if (!ok) {
      *abort_flag = 1;
      atomicOr(a.status, kErrTimeout);
    }
    mma_commit(accb);
  };

  // ---- phase 1: Z = sum_r M_r W_r
  if (warp == 0) {
    if (lane == 0) {
      for (int g = 0; g < S && g < CT; ++g) issue_load(g);
      if (C1 > 0) run_chunks(0, C1);
      else mma_commit(accb);
    }
    __syncwarp();
  }
  const int row = warp * 32 + lane;
  const int64_t m = m0 + row;
  const bool live = m < a.n;
  const int64_t node = a.off + (live ? m : 0);
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  if (!mbar_wait(accb, 0)) atomicOr(a.status, kErrTimeout);
  fence_after_sync();
  // ---- epilogue 1: Z -> bf16 -> saved + shared-memory operand (zero when no relation)
#pragma unroll 1
  for (int c = 0; c < D; c += 16) {
    float v[16];
    if (C1 > 0) {
      tmem_ld16(trow + c, v);
      round16(v);
    } else {
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] = 0.f;
    }
    if (live) store16_bf16(a.Z + node * D + c, v);
    put_tile16(ztile, row, c, v);
  }
  fence_async_smem();
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  // ---- phase 2: U = Z W_agg
  if (warp == 0) {
    if (lane == 0) run_chunks(C1, CT);
    __syncwarp();
  }
  if (!mbar_wait(accb, 1)) atomicOr(a.status, kErrTimeout);
  fence_after_sync();
  // ---- epilogue 2: bias, activation, residual, LayerNorm
  const __nv_bfloat16* hrow = a.H_in + node * D;
  float sum = 0.f;
  if constexpr (D <= 128) {
    float y[D];
#pragma unroll
    for (int c = 0; c < D; c += 16) {
      float u[16], h[16], bb[16];
      tmem_ld16(trow + c, u);
      load16_bf16(a.b + c, bb);
      load16_bf16(hrow + c, h);
#pragma unroll
      for (int i = 0; i < 16; ++i) u[i] = __bfloat162float(__float2bfloat16_rn(u[i] + bb[i]));
      if (live) store16_bf16(a.U + node * D + c, u);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        y[c + i] = act_apply(u[i], a.act) + h[i];
        sum += y[c + i];
      }
    }
    if (a.ln) {
      const float mean = sum * (1.f / D);
      float q = 0.f;
#pragma unroll
      for (int i = 0; i < D; ++i) q += (y[i] - mean) * (y[i] - mean);
      const float rstd = rsqrtf(q * (1.f / D) + a.eps);
#pragma unroll
      for (int c = 0; c < D; c += 16) {
        float g[16], be[16], o[16];
        load16_bf16(a.gamma + c, g);
        load16_bf16(a.beta + c, be);
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i] = (y[c + i] - mean) * rstd * g[i] + be[i];
        if (live) store16_bf16(a.H_out + node * D + c, o);
      }
      if (live) a.stats[node] = make_float2(mean, rstd);
    } else if (live) {
#pragma unroll
      for (int c = 0; c < D; c += 16) store16_bf16(a.H_out + node * D + c, y + c);
    }
  } else {
    // wide rows: three passes over TMEM / H_in instead of holding the row in registers
    auto y16 = [&](int c, float* y) {
      float u[16], h[16], bb[16];
      tmem_ld16(trow + c, u);
      load16_bf16(a.b + c, bb);
      load16_bf16(hrow + c, h);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        u[i] = __bfloat162float(__float2bfloat16_rn(u[i] + bb[i]));
        y[i] = act_apply(u[i], a.act) + h[i];
      }
      return;
    };
#pragma unroll 1
    for (int c = 0; c < D; c += 16) {
      float u[16], h[16], bb[16], y[16];
      tmem_ld16(trow + c, u);
      load16_bf16(a.b + c, bb);
      load16_bf16(hrow + c, h);
#pragma unroll
      for (int i = 0; i < 16; ++i) {
        u[i] = __bfloat162float(__float2bfloat16_rn(u[i] + bb[i]));
        y[i] = act_apply(u[i], a.act) + h[i];
        sum += y[i];
      }
      if (live) store16_bf16(a.U + node * D + c, u);
      if (!a.ln && live) store16_bf16(a.H_out + node * D + c, y);
    }
    if (a.ln) {
      const float mean = sum * (1.f / D);
      float q = 0.f;
#pragma unroll 1
      for (int c = 0; c < D; c += 16) {
        float y[16];
        y16(c, y);
#pragma unroll
        for (int i = 0; i < 16; ++i) q += (y[i] - mean) * (y[i] - mean);
      }
      const float rstd = rsqrtf(q * (1.f / D) + a.eps);
#pragma unroll 1
      for (int c = 0; c < D; c += 16) {
        float y[16], g[16], be[16], o[16];
        y16(c, y);
        load16_bf16(a.gamma + c, g);
        load16_bf16(a.beta + c, be);
#pragma unroll
        for (int i = 0; i < 16; ++i) o[i] = (y[i] - mean) * rstd * g[i] + be[i];
        if (live) store16_bf16(a.H_out + node * D + c, o);
      }
      if (live) a.stats[node] = make_float2(mean, rstd);
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

// ---------------------------------------------------------------------------------------------
// backward, row side
// ---------------------------------------------------------------------------------------------
template <int D>
struct BwdCfg {
  static constexpr int kStages = D == 256 ? 3 : 2;
  static constexpr int kB = D * 128;
  static constexpr int kT = kTileRows * D * 2;  // dU / dZ operand tile
  static constexpr int kRed = 4 * 3 * D * 4;    // per-warp column partials
  static constexpr int kSmem = kStages * kB + kT + kRed + 256 + 1024;
  static constexpr int kTmemCols = D < 32 ? 32 : D;
};


template <int D>
__global__ void __launch_bounds__(kThreads, 1) proj_bwd_tc(const __grid_constant__ CUtensorMap tm_Wagg,
                                                          const __grid_constant__ CUtensorMap tm_Wrel, TcBwdArgs a) {
  using C = BwdCfg<D>;
  constexpr int S = C::kStages;
  constexpr int KC = D / 64;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* bstage = smem;                       // S x B chunk
  uint8_t* tile = smem + S * C::kB;             // KC x 16 KB
  float* red = reinterpret_cast<float*>(tile + C::kT);
  uint64_t* full = reinterpret_cast<uint64_t*>(reinterpret_cast<uint8_t*>(red) + C::kRed);
  uint64_t* empty = full + S;
  uint64_t* accb = empty + S;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  int* abort_flag = reinterpret_cast<int*>(tslot + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t m0 = (int64_t)blockIdx.x * kTileRows;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accb, 1);
    *abort_flag = 0;
    fence_mbar_init();
    prefetch_tmap(&tm_Wagg);
    prefetch_tmap(&tm_Wrel);
  }
  if (warp == 0) tmem_alloc(tslot, C::kTmemCols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  // B chunks: [0, KC) = W_agg[t], then KC per relation
  const int CT = KC * (1 + a.nrel);
  auto issue_load = [&](int g) {
    const int s = g % S;
    mbar_expect_tx(&full[s], C::kB);
    if (g < KC)
      tma_load_2d(bstage + s * C::kB, &tm_Wagg, g * 64, a.type * D, &full[s]);
    else
      tma_load_2d(bstage + s * C::kB, &tm_Wrel, (g % KC) * 64, a.rel[g / KC - 1] * D, &full[s]);
  };
  if (threadIdx.x == 0)
    for (int g = 0; g < S && g < CT; ++g) issue_load(g);
  const uint32_t idesc = idesc_bf16(128, D, false, false);
  // one product: accumulator = tile (128 x D) x chunks [g0, g0 + KC)
  auto product = [&](int g0) {
    bool ok = *abort_flag == 0;
    for (int g = g0; g < g0 + KC && ok; ++g) {
      const int s = g % S;
      ok = mbar_wait(&full[s], (g / S) & 1);
      if (!ok) break;
      fence_after_sync();
      const uint8_t* A = tile + (g - g0) * kATile;
      const uint8_t* B = bstage + s * C::kB;
#pragma unroll
      for (int ks = 0; ks < 4; ++ks)
        mma_bf16(tmem, desc_sw128(smem_u32(A) + ks * 32, 16, 1024), desc_sw128(smem_u32(B) + ks * 32, 16, 1024), idesc,
                 (g > g0 || ks > 0) ? 1u : 0u);
      mma_commit(&empty[s]);
      if (g + S < CT) {
        ok = mbar_wait(&empty[s], (g / S) & 1);
        if (ok) issue_load(g + S);
      }
    }
    if (!ok) {
      *abort_flag = 1;
      atomicOr(a.status, kErrTimeout);
    }
    mma_commit(accb);
  };

  const int row = warp * 32 + lane;
  const int64_t m = m0 + row;
  const bool live = m < a.n;
  const int64_t node = a.off + (live ? m : 0);
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  // ---- prologue: LayerNorm / activation backward, dU -> tile; column partials
  {
    const __nv_bfloat16* dor = a.dH_out + node * D;
    const __nv_bfloat16* ur = a.U + node * D;
    const __nv_bfloat16* hr = a.H_in + node * D;
    const float2 st = (live && a.ln) ? a.stats[node] : make_float2(0.f, 1.f);
    float s1 = 0.f, s2 = 0.f;
    if (a.ln) {
#pragma unroll 1
      for (int c = 0; c < D; c += 16) {
        float dv[16], uv[16], hv[16], g[16];
        load16_bf16(dor + c, dv);
        load16_bf16(ur + c, uv);
        load16_bf16(hr + c, hv);
        load16_bf16(a.gamma + c, g);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          const float xh = (act_apply(uv[i], a.act) + hv[i] - st.x) * st.y;
          const float dxh = dv[i] * g[i];
          s1 += dxh;
          s2 += dxh * xh;
        }
      }
    }
    const float mean1 = s1 * (1.f / D), mean2 = s2 * (1.f / D);
#pragma unroll 1
    for (int c = 0; c < D; c += 32) {
      float pdb[32], pdg[32], pdb2[32];
#pragma unroll
      for (int h = 0; h < 32; h += 16) {
        float dv[16], uv[16], hv[16], g[16], dy[16], du[16];
        load16_bf16(dor + c + h, dv);
        load16_bf16(ur + c + h, uv);
        load16_bf16(hr + c + h, hv);
        if (a.ln) load16_bf16(a.gamma + c + h, g);
#pragma unroll
        for (int i = 0; i < 16; ++i) {
          float xh = 0.f;
          if (a.ln) {
            xh = (act_apply(uv[i], a.act) + hv[i] - st.x) * st.y;
            dy[i] = st.y * (dv[i] * g[i] - mean1 - xh * mean2);
          } else {
            dy[i] = dv[i];
          }
          du[i] = __bfloat162float(__float2bfloat16_rn(dy[i] * act_grad(uv[i], a.act)));
          if (!live) du[i] = dy[i] = dv[i] = xh = 0.f;
          pdb[h + i] = du[i];
          pdg[h + i] = dv[i] * xh;
          pdb2[h + i] = dv[i];
        }
        if (live) {
          store16_bf16(a.dY + node * D + c + h, dy);
          store16_bf16(a.dU + node * D + c + h, du);
        }
        put_tile16(tile, row, c + h, du);
      }
      const float vdb = warp_transpose_sum(pdb);
      const float vdg = warp_transpose_sum(pdg);
      const float vdb2 = warp_transpose_sum(pdb2);
      red[(warp * 3 + 0) * D + c + lane] = vdb;
      red[(warp * 3 + 1) * D + c + lane] = vdg;
      red[(warp * 3 + 2) * D + c + lane] = vdb2;
    }
  }
  fence_async_smem();
  __syncthreads();
  for (int k = threadIdx.x; k < 3 * D; k += kThreads) {
    const int q = k / D, c = k % D;
    a.part[((int64_t)blockIdx.x * 3 + q) * D + c] =
        ((red[(0 * 3 + q) * D + c] + red[(1 * 3 + q) * D + c]) + red[(2 * 3 + q) * D + c]) + red[(3 * 3 + q) * D + c];
  }
  fence_after_sync();
  // ---- dZ = dU W_agg^T
  if (warp == 0) {
    if (lane == 0) product(0);
    __syncwarp();
  }
  uint32_t phase = 0;
  if (!mbar_wait(accb, phase)) atomicOr(a.status, kErrTimeout);
  phase ^= 1;
  fence_after_sync();
#pragma unroll 1
  for (int c = 0; c < D; c += 16) {
    float v[16];
    tmem_ld16(trow + c, v);
    round16(v);
    if (live) store16_bf16(a.dZ + node * D + c, v);
    put_tile16(tile, row, c, v);
  }
  fence_async_smem();
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  // ---- dMs_r = (dZ W_r^T) / deg_r
  for (int r = 0; r < a.nrel; ++r) {
    if (warp == 0) {
      if (lane == 0) product(KC * (1 + r));
      __syncwarp();
    }
    if (!mbar_wait(accb, phase)) atomicOr(a.status, kErrTimeout);
    phase ^= 1;
    fence_after_sync();
    const int64_t crow = a.mrow0[r] + (live ? m : 0);
    const int deg = live ? a.csr_ptr[crow + 1] - a.csr_ptr[crow] : 0;
    const float sc = deg > 0 ? __fdiv_rn(1.0f, (float)deg) : 0.f;
#pragma unroll 1
    for (int c = 0; c < D; c += 16) {
      float v[16];
      tmem_ld16(trow + c, v);
#pragma unroll
      for (int i = 0; i < 16; ++i) v[i] *= sc;
      if (live) store16_bf16(a.dMs + crow * D + c, v);
    }
    fence_before_sync();
    __syncthreads();
    fence_after_sync();
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, C::kTmemCols);
}

// ---------------------------------------------------------------------------------------------
// weight gradients: part[split][i][j] = sum over the split's rows k of X[k][i] Y[k][j]
// ---------------------------------------------------------------------------------------------
template <int D>
struct WgCfg {
  static constexpr int kStages = 4;
  static constexpr int kA = 2 * 8192;                  // 64 rows x 128 columns (two 64-wide blocks)
  static constexpr int kB = (D < 64 ? 64 : D) * 128;   // 64 rows x D columns
  static constexpr int kStage = kA + kB;
  static constexpr int kSmem = kStages * kStage + 256 + 1024;
  static constexpr int kTmemCols = D < 32 ? 32 : D;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1) wgrad_tc(const __grid_constant__ CUtensorMap tm_X,
                                                       const __grid_constant__ CUtensorMap tm_Y, int64_t n,
                                                       int chunks_per_split, float* __restrict__ part,
                                                       int* __restrict__ status) {
  using C = WgCfg<D>;
  constexpr int S = C::kStages;
  constexpr int NB = D / 64;  // 64-wide column blocks of Y
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * C::kStage);
  uint64_t* empty = full + S;
  uint64_t* accb = empty + S;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x;  // 128-wide block of X's columns (output rows)
  const int64_t nchunks = (n + 63) / 64;
  const int64_t c0 = (int64_t)blockIdx.y * chunks_per_split;
  const int64_t c1 = min(nchunks, c0 + chunks_per_split);
  const int CT = (int)max((int64_t)0, c1 - c0);
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(accb, 1);
    fence_mbar_init();
    prefetch_tmap(&tm_X);
    prefetch_tmap(&tm_Y);
  }
  if (warp == 0) tmem_alloc(tslot, C::kTmemCols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  if (warp == 0) {
    if (lane == 0) {
      auto issue_load = [&](int g) {
        const int s = g % S;
        uint8_t* A = smem + s * C::kStage;
        uint8_t* B = A + C::kA;
        const int y = (int)((c0 + g) * 64);
        mbar_expect_tx(&full[s], C::kA + NB * 8192);
        tma_load_2d(A, &tm_X, mt * 128, y, &full[s]);
        tma_load_2d(A + 8192, &tm_X, mt * 128 + 64, y, &full[s]);
        for (int j = 0; j < NB; ++j) tma_load_2d(B + j * 8192, &tm_Y, j * 64, y, &full[s]);
      };
      const uint32_t idesc = idesc_bf16(128, D, true, true);
      bool ok = true;
      for (int g = 0; g < S && g < CT; ++g) issue_load(g);
      for (int g = 0; g < CT && ok; ++g) {
        const int s = g % S;
        ok = mbar_wait(&full[s], (g / S) & 1);
        if (!ok) break;
        fence_after_sync();
        const uint32_t A = smem_u32(smem + s * C::kStage);
        const uint32_t B = A + C::kA;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks)
          mma_bf16(tmem, desc_sw128(A + ks * 2048, 8192, 1024), desc_sw128(B + ks * 2048, 8192, 1024), idesc,
                   (g > 0 || ks > 0) ? 1u : 0u);
        mma_commit(&empty[s]);
        if (g + S < CT) {
          ok = mbar_wait(&empty[s], (g / S) & 1);
          if (ok) issue_load(g + S);
        }
      }
      if (!ok) atomicOr(status, kErrTimeout);
      mma_commit(accb);
    }
    __syncwarp();
  }
  if (!mbar_wait(accb, 0)) atomicOr(status, kErrTimeout);
  fence_after_sync();
  const int orow = mt * 128 + warp * 32 + lane;  // output row i (column of X)
  float* out = part + (int64_t)blockIdx.y * D * D;
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

// ---------------------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------------------
template <int D>
static hg_status smem_attr_once() {
  static bool done = false;
  if (!done) {
    HG_CUDA(cudaFuncSetAttribute(proj_fwd_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, FwdCfg<D>::kSmem));
    HG_CUDA(cudaFuncSetAttribute(proj_bwd_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, BwdCfg<D>::kSmem));
    HG_CUDA(cudaFuncSetAttribute(wgrad_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, WgCfg<D>::kSmem));
    done = true;
  }
  return HG_OK;
}

template <int D>
static hg_status tc_fwd_t(const TcFwdArgs& a, const void* M, int64_t m_rows, const void* WrelT, int num_rels,
                          const void* WaggT, int num_types, cudaStream_t s) {
  HG_TRY(smem_attr_once<D>());
  CUtensorMap tm_M, tm_W, tm_A;
  HG_TRY(make_tmap_bf16(&tm_M, M, (uint64_t)std::max<int64_t>(m_rows, 1), D, kTileRows));
  HG_TRY(make_tmap_bf16(&tm_W, WrelT, (uint64_t)num_rels * D, D, D));
  HG_TRY(make_tmap_bf16(&tm_A, WaggT, (uint64_t)num_types * D, D, D));
  return launch("proj_fwd_tc", proj_fwd_tc<D>, dim3((unsigned)ceil_div(a.n, kTileRows)), dim3(kThreads),
                FwdCfg<D>::kSmem, s, tm_M, tm_W, tm_A, a);
}

template <int D>
static hg_status tc_bwd_t(const TcBwdArgs& a, const void* Wagg, int num_types, const void* Wrel, int num_rels,
                          cudaStream_t s) {
  HG_TRY(smem_attr_once<D>());
  CUtensorMap tm_A, tm_W;
  HG_TRY(make_tmap_bf16(&tm_A, Wagg, (uint64_t)num_types * D, D, D));
  HG_TRY(make_tmap_bf16(&tm_W, Wrel, (uint64_t)num_rels * D, D, D));
  return launch("proj_bwd_tc", proj_bwd_tc<D>, dim3((unsigned)ceil_div(a.n, kTileRows)), dim3(kThreads),
                BwdCfg<D>::kSmem, s, tm_A, tm_W, a);
}

int wgrad_tc_splits(int64_t n, int d) {
  const int mtiles = d > 128 ? d / 128 : 1;
  const int64_t chunks = std::max<int64_t>(1, ceil_div(n, 64));
  return (int)std::max<int64_t>(1, std::min<int64_t>(chunks, (2 * 152) / mtiles));
}

template <int D>
static hg_status tc_wgrad_t(const void* X, int64_t x0, const void* Y, int64_t y0, int64_t n, float* part, float* out,
                            float* tmp, cudaStream_t s) {
  HG_TRY(smem_attr_once<D>());
  const int mtiles = D > 128 ? D / 128 : 1;
  const int splits = wgrad_tc_splits(n, D);
  const int64_t chunks = std::max<int64_t>(1, ceil_div(n, 64));
  const int cps = (int)ceil_div(chunks, splits);
  if (n == 0) {
    HG_CUDA(cudaMemsetAsync(out, 0, (size_t)D * D * sizeof(float), s));
    return HG_OK;
  }
  CUtensorMap tm_X, tm_Y;
  HG_TRY(make_tmap_bf16(&tm_X, (const __nv_bfloat16*)X + x0 * D, (uint64_t)n, D, 64));
  HG_TRY(make_tmap_bf16(&tm_Y, (const __nv_bfloat16*)Y + y0 * D, (uint64_t)n, D, 64));
  HG_TRY(launch("wgrad_tc", wgrad_tc<D>, dim3(mtiles, splits), dim3(kThreads), WgCfg<D>::kSmem, s, tm_X, tm_Y, n, cps,
                part, device_status_ptr()));
  return reduce_partials(part, (int64_t)D * D, splits, (int64_t)D * D, out, tmp, s);
}

hg_status tc_proj_forward(int d, const TcFwdArgs& a, const void* M, int64_t m_rows, const void* WrelT, int num_rels,
                          const void* WaggT, int num_types, cudaStream_t s) {
  if (d == 64) return tc_fwd_t<64>(a, M, m_rows, WrelT, num_rels, WaggT, num_types, s);
  if (d == 128) return tc_fwd_t<128>(a, M, m_rows, WrelT, num_rels, WaggT, num_types, s);
  if (d == 256) return tc_fwd_t<256>(a, M, m_rows, WrelT, num_rels, WaggT, num_types, s);
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}

hg_status tc_proj_backward(int d, const TcBwdArgs& a, const void* Wagg, int num_types, const void* Wrel, int num_rels,
                           cudaStream_t s) {
  if (d == 64) return tc_bwd_t<64>(a, Wagg, num_types, Wrel, num_rels, s);
  if (d == 128) return tc_bwd_t<128>(a, Wagg, num_types, Wrel, num_rels, s);
  if (d == 256) return tc_bwd_t<256>(a, Wagg, num_types, Wrel, num_rels, s);
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}

hg_status tc_weight_grad(int d, const void* X, int64_t x0, const void* Y, int64_t y0, int64_t n, float* part,
                         float* out, float* tmp, cudaStream_t s) {
  if (d == 64) return tc_wgrad_t<64>(X, x0, Y, y0, n, part, out, tmp, s);
  if (d == 128) return tc_wgrad_t<128>(X, x0, Y, y0, n, part, out, tmp, s);
  if (d == 256) return tc_wgrad_t<256>(X, x0, Y, y0, n, part, out, tmp, s);
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}

}  // namespace hg
