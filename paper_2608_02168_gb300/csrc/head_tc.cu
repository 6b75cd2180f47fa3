// Tensor-core kernels of the bf16 prediction head (Section 3.4, Eq. 18-19).
//
// Forward, one CTA of 128 threads per 128 labelled rows: the threads gather the labelled rows of H
// into a 128-byte-swizzled K-major tile in shared memory (and the rows' MeanAgg embedding, the
// mean with the replica in H_rep rounded to bf16, into the saved Hm for the weight gradient); W1
// arrives by TMA as an MN-major operand (its rows are the K dimension, 64-column blocks along the
// hidden units); one chain of tcgen05.mma puts H W1 (fp32, 128 x d) in tensor memory.  When rows
// of the tile have a replica, the tile is refilled with the replica rows (zero elsewhere) once the
// first chain has read it, and a second chain adds H_rep W1; the epilogue halves those rows.  So
// the pre-activation a = ((h + h_rep) / 2) W1 is formed from the stored bf16 rows without rounding
// their mean.  Thread t then owns row t:
// it adds b1, forms the logit z = relu(a) . w2 + b2, the loss term and the unit gradient
// dA = (sigmoid(z) - y)/n * w2 * [a > 0], stores dA (bf16), and the CTA writes its partial sums
// (loss, dz, column sums of dA and of dz relu(a)) in a fixed order.
//
// Input gradient, one CTA per 128 rows: dA (TMA, K-major) times W1 as a K-major operand (W1[i][h]
// with h contiguous is exactly B[n = i][k = h]) gives dh = dA W1^T in tensor memory; thread t adds
// dloss * dh (halved for a row with a replica) to its row of dH and of dH_rep.
#include <algorithm>

#include "head_kernels.cuh"
#include "layer_kernels.cuh"
#include "tc_util.cuh"

namespace hg {

using namespace tc;

namespace {

constexpr int kThreads = 128;
constexpr int kRows = kHeadTcRows;
constexpr int kABlk = kRows * 128;  // one 64-column block of the 128-row K-major tile

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

template <int D>
struct HeadTcCfg {
  static constexpr int NB = D / 64;
  static constexpr int kWBlk = D * 128;  // one 64-column block of W1: D rows x 128 bytes
  static constexpr int kW = NB * kWBlk;
  static constexpr int kA = NB * kABlk;
  // forward tail: 2 barriers + TMEM slot (32 B), b1 / w2 (fp32), column partials [4][2D], row
  // partials [4][2], row table [2][128]
  static constexpr int kFwdTail = 32 + 2 * D * 4 + 4 * 2 * D * 4 + 4 * 2 * 4 + 2 * kRows * 4;
  static constexpr int kFwdSmem = kW + kA + kFwdTail + 1024;
  static constexpr int kDxSmem = kW + kA + 32 + 1024;
};

__device__ __forceinline__ float softplus_f(float x) { return fmaxf(x, 0.f) + log1pf(expf(-fabsf(x))); }

__device__ __forceinline__ float sigmoid_f(float z) {
  const float e = expf(-fabsf(z));
  return z >= 0.f ? 1.f / (1.f + e) : e / (1.f + e);
}

// v[0..31] per lane -> lane L returns the sum over the warp of v[L] (fixed butterfly order).
__device__ __forceinline__ float transpose_sum32(float (&v)[32]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int s = 16; s >= 1; s >>= 1) {
    const bool hi = (lane & s) != 0;
#pragma unroll
    for (int i = 0; i < s; ++i) {
      const float send = hi ? v[i] : v[i + s];
      const float keep = hi ? v[i + s] : v[i];
      v[i] = keep + __shfl_xor_sync(0xffffffffu, send, s);
    }
  }
  return v[0];
}

__device__ __forceinline__ float warp_sum(float x) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) x += __shfl_xor_sync(0xffffffffu, x, o);
  return x;
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    head_fwd_tc_kernel(const __grid_constant__ CUtensorMap tm_W, HeadFwdArgs a) {
  using C = HeadTcCfg<D>;
  constexpr int TPR = D / 8;           // 16-byte pieces per row
  constexpr int RPP = kThreads / TPR;  // rows per gather pass
  constexpr int PASSES = kRows / RPP;
  constexpr int BATCH = PASSES < 8 ? PASSES : 8;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Wimg = smem;
  uint8_t* Aimg = smem + C::kW;
  uint64_t* bars = reinterpret_cast<uint64_t*>(Aimg + C::kA);  // [0] W1 loaded, [1] MMA done
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
  float* b1f = reinterpret_cast<float*>(bars + 4);
  float* w2f = b1f + D;
  float* colred = w2f + D;          // [4][2D]
  float* rowred = colred + 8 * D;   // [4][2]
  int32_t* rowi = reinterpret_cast<int32_t*>(rowred + 8);
  int32_t* repi = rowi + kRows;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t r0 = (int64_t)blockIdx.x * kRows;
  const __nv_bfloat16* H = (const __nv_bfloat16*)a.H;
  const __nv_bfloat16* Hr = (const __nv_bfloat16*)a.H_rep;

  if (tid == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, D);
  {  // row table: labelled row and replica row of each tile row
    const int64_t r = r0 + tid;
    int32_t i = -1, j = -1;
    if (r < a.n) {
      const int32_t li = a.lab[r];
      if (li >= 0 && li < a.rows) {
        i = li;
        j = a.map[li];
      }
      a.rep_row[r] = i >= 0 ? j : -2;
    }
    rowi[tid] = i;
    repi[tid] = j;
  }
  for (int c = tid; c < D; c += kThreads) {
    b1f[c] = __bfloat162float(((const __nv_bfloat16*)a.b1)[c]);
    w2f[c] = __bfloat162float(((const __nv_bfloat16*)a.w2)[c]);
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  if (tid == 0) {
    mbar_expect_tx(&bars[0], (uint32_t)C::kW);
#pragma unroll
    for (int b = 0; b < C::NB; ++b) tma_load_2d(Wimg + b * C::kWBlk, &tm_W, b * 64, 0, &bars[0]);
  }
  // gather the MeanAgg rows (coalesced 16-byte pieces), BATCH passes of loads in flight
  const int g = tid % TPR, sub = tid / TPR;
#pragma unroll 1
  for (int p0 = 0; p0 < PASSES; p0 += BATCH) {
    uint4 v[BATCH], u[BATCH];
#pragma unroll
    for (int q = 0; q < BATCH; ++q) {
      const int rl = sub + (p0 + q) * RPP;
      const int32_t i = rowi[rl], j = repi[rl];
      v[q] = i >= 0 ? ldg16(H + (int64_t)i * D + g * 8) : make_uint4(0, 0, 0, 0);
      u[q] = (i >= 0 && j >= 0) ? ldg16(Hr + (int64_t)j * D + g * 8) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int q = 0; q < BATCH; ++q) {
      const int rl = sub + (p0 + q) * RPP;
      const int64_t r = r0 + rl;
      uint4 h = v[q];
      if (rowi[rl] >= 0 && repi[rl] >= 0) {
        float x[8], y[8];
        unpack(v[q], x, __nv_bfloat16());
        unpack(u[q], y, __nv_bfloat16());
#pragma unroll
        for (int e = 0; e < 8; ++e) x[e] = 0.5f * (x[e] + y[e]);
        h = pack(x, __nv_bfloat16());
      }
      if (r < a.n) st16((__nv_bfloat16*)a.Hm + r * D + g * 8, h);
      st16(Aimg + (g >> 3) * kABlk + sw128_offset(rl, (g & 7) * 16), v[q]);
    }
  }
  fence_async_smem();
  const bool two = __syncthreads_or(rowi[tid] >= 0 && repi[tid] >= 0) != 0;  // any replica in the tile
  int chains = 0;  // MMA chains issued (thread 0)
  auto issue_chain = [&](bool accumulate) {
    ++chains;
    fence_after_sync();
    const uint32_t A = smem_u32(Aimg), W = smem_u32(Wimg);
    const uint32_t idesc = idesc_bf16(128, D, false, true);
#pragma unroll
    for (int j = 0; j < D / 16; ++j)
      mma_bf16(tmem, desc_sw128(A + (j >> 2) * kABlk + (j & 3) * 32, 16, 1024),
               desc_sw128(W + j * 2048, C::kWBlk, 1024), idesc, (accumulate || j > 0) ? 1u : 0u);
    mma_commit(&bars[1]);
  };
  bool ok = true;
  if (tid == 0) {
    ok = mbar_wait(&bars[0], 0);
    if (ok)
      issue_chain(false);
    else
      record_device_error(a.status, kErrTimeout);
  }
  ok = __syncthreads_and(ok);
  if (ok && two) {
    // the first chain has read the tile: refill it with the replica rows (zero for rows without)
    if (!mbar_wait(&bars[1], 0)) {
      record_device_error(a.status, kErrTimeout);
      ok = false;
    }
    ok = __syncthreads_and(ok);
    if (ok) {
      fence_after_sync();
#pragma unroll 1
      for (int p0 = 0; p0 < PASSES; p0 += BATCH) {
        uint4 u[BATCH];
#pragma unroll
        for (int q = 0; q < BATCH; ++q) {
          const int rl = sub + (p0 + q) * RPP;
          const int32_t i = rowi[rl], j = repi[rl];
          u[q] = (i >= 0 && j >= 0) ? ldg16(Hr + (int64_t)j * D + g * 8) : make_uint4(0, 0, 0, 0);
        }
#pragma unroll
        for (int q = 0; q < BATCH; ++q)
          st16(Aimg + (g >> 3) * kABlk + sw128_offset(sub + (p0 + q) * RPP, (g & 7) * 16), u[q]);
      }
      fence_async_smem();
      __syncthreads();
      if (tid == 0) issue_chain(true);
    }
  }
  if (ok && !mbar_wait(&bars[1], two ? 1 : 0)) {
    record_device_error(a.status, kErrTimeout);
    ok = false;
  }
  fence_after_sync();
  // epilogue: thread tid owns tile row tid (TMEM lane tid)
  const int rl = tid;
  const int64_t r = r0 + rl;
  const bool live = r < a.n;
  const bool valid = live && rowi[rl] >= 0;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
  const float b2 = __bfloat162float(((const __nv_bfloat16*)a.b2)[0]);
  const float half = (rowi[rl] >= 0 && repi[rl] >= 0) ? 0.5f : 1.f;  // (h + h_rep) W1 / 2
  float zpart = 0.f;
#pragma unroll 1
  for (int c = 0; c < D; c += 32) {
    float acc[32];
    tmem_ld32(trow + c, acc);
#pragma unroll
    for (int e = 0; e < 32; ++e) zpart = fmaf(fmaxf(fmaf(half, acc[e], b1f[c + e]), 0.f), w2f[c + e], zpart);
  }
  const float z = zpart + b2;
  float term = 0.f, dz = 0.f;
  if (live) {
    const float y = a.y[r];
    if (valid) {
      term = y * softplus_f(-z) + (1.f - y) * softplus_f(z);
      dz = (sigmoid_f(z) - y) * a.inv_n;
    } else {
      term = __int_as_float(0x7fc00000);  // an out-of-range row makes the loss NaN
    }
    if (a.logits) a.logits[r] = z;
  }
  if (!ok) dz = 0.f;
#pragma unroll 1
  for (int c = 0; c < D; c += 32) {
    float acc[32], da[32], dw[32];
    tmem_ld32(trow + c, acc);
#pragma unroll
    for (int e = 0; e < 32; ++e) {
      const float h = fmaf(half, acc[e], b1f[c + e]);
      da[e] = h > 0.f ? dz * w2f[c + e] : 0.f;
      dw[e] = dz * fmaxf(h, 0.f);
    }
    if (live) {
      __nv_bfloat16* dst = (__nv_bfloat16*)a.dA + r * D + c;
#pragma unroll
      for (int e = 0; e < 32; e += 8) st16(dst + e, pack(da + e, __nv_bfloat16()));
    }
    colred[warp * 2 * D + c + lane] = transpose_sum32(da);
    colred[warp * 2 * D + D + c + lane] = transpose_sum32(dw);
  }
  const float tsum = warp_sum(term), dsum = warp_sum(dz);
  if (lane == 0) {
    rowred[warp * 2] = tsum;
    rowred[warp * 2 + 1] = dsum;
  }
  fence_before_sync();
  __syncthreads();
  float* out = a.part + (int64_t)blockIdx.x * (2 + 2 * D);
  for (int c = tid; c < 2 * D; c += kThreads)
    out[2 + c] = ((colred[c] + colred[2 * D + c]) + colred[4 * D + c]) + colred[6 * D + c];
  if (tid == 0) {
    out[0] = ((rowred[0] + rowred[2]) + rowred[4]) + rowred[6];
    out[1] = ((rowred[1] + rowred[3]) + rowred[5]) + rowred[7];
  }
  if (!ok && tid == 0) {  // give-up path: the weight load and the MMAs issued complete first
    mbar_wait(&bars[0], 0);
    if (chains > 0) mbar_wait(&bars[1], (uint32_t)(chains - 1) & 1u);
  }
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, D);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    head_dx_tc_kernel(const __grid_constant__ CUtensorMap tm_W, const __grid_constant__ CUtensorMap tm_dA,
                      HeadBwdArgs a) {
  using C = HeadTcCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Wimg = smem;
  uint8_t* Aimg = smem + C::kW;
  uint64_t* bars = reinterpret_cast<uint64_t*>(Aimg + C::kA);  // [0] operands loaded, [1] MMA done
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int64_t r0 = (int64_t)blockIdx.x * kRows;
  if (tid == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, D);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  bool ok = true;
  if (tid == 0) {
    mbar_expect_tx(&bars[0], (uint32_t)(C::kW + C::kA));
#pragma unroll
    for (int b = 0; b < C::NB; ++b) {
      tma_load_2d(Wimg + b * C::kWBlk, &tm_W, b * 64, 0, &bars[0]);
      tma_load_2d(Aimg + b * kABlk, &tm_dA, b * 64, (int)r0, &bars[0]);
    }
    ok = mbar_wait(&bars[0], 0);
    if (ok) {
      fence_after_sync();
      const uint32_t A = smem_u32(Aimg), W = smem_u32(Wimg);
      const uint32_t idesc = idesc_bf16(128, D, false, false);
#pragma unroll
      for (int j = 0; j < D / 16; ++j)
        mma_bf16(tmem, desc_sw128(A + (j >> 2) * kABlk + (j & 3) * 32, 16, 1024),
                 desc_sw128(W + (j >> 2) * C::kWBlk + (j & 3) * 32, 16, 1024), idesc, j > 0 ? 1u : 0u);
      mma_commit(&bars[1]);
    } else {
      record_device_error(a.status, kErrTimeout);
      mbar_wait(&bars[0], 0);  // give-up path: the loads land before the CTA moves on
    }
  }
  ok = __syncthreads_and(ok);
  if (ok && !mbar_wait(&bars[1], 0)) {
    record_device_error(a.status, kErrTimeout);
    ok = false;
    if (tid == 0) mbar_wait(&bars[1], 0);  // the MMAs issued complete before TMEM is released
  }
  fence_after_sync();
  const int64_t r = r0 + tid;
  int32_t rep = -2;
  int64_t li = 0;
  if (ok && r < a.n) {
    rep = a.rep_row[r];
    if (rep != -2) li = a.lab[r];
  }
  const float scale = rep >= 0 ? 0.5f * a.dloss : a.dloss;
  __nv_bfloat16* dst_h = (rep != -2 && a.dH) ? (__nv_bfloat16*)a.dH + li * D : nullptr;
  __nv_bfloat16* dst_r = (rep >= 0 && a.dH_rep) ? (__nv_bfloat16*)a.dH_rep + (int64_t)rep * D : nullptr;
  const uint32_t trow = tmem + ((uint32_t)(warp * 32) << 16);
#pragma unroll 1
  for (int c = 0; c < D; c += 32) {
    float acc[32];
    tmem_ld32(trow + c, acc);
#pragma unroll
    for (int e = 0; e < 32; ++e) acc[e] *= scale;
#pragma unroll
    for (int k = 0; k < 2; ++k) {
      __nv_bfloat16* dst = k == 0 ? dst_h : dst_r;
      if (!dst) continue;
#pragma unroll
      for (int e = 0; e < 32; e += 8) {
        float x[8];
        unpack(ld16(dst + c + e), x, __nv_bfloat16());
#pragma unroll
        for (int q = 0; q < 8; ++q) x[q] += acc[e + q];
        st16(dst + c + e, pack(x, __nv_bfloat16()));
      }
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, D);
}

template <int D>
hg_status smem_once() {
  static bool done = false;
  if (!done) {
    HG_CUDA(cudaFuncSetAttribute(head_fwd_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 HeadTcCfg<D>::kFwdSmem));
    HG_CUDA(cudaFuncSetAttribute(head_dx_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 HeadTcCfg<D>::kDxSmem));
    done = true;
  }
  return HG_OK;
}

template <int D>
hg_status fwd_t(const HeadFwdArgs& a, cudaStream_t s) {
  HG_TRY(smem_once<D>());
  CUtensorMap tm_W;
  HG_TRY(make_tmap_bf16(&tm_W, a.W1, D, D, D));
  return launch("head_fwd_tc", head_fwd_tc_kernel<D>, dim3((unsigned)ceil_div(a.n, kRows)), dim3(kThreads),
                (size_t)HeadTcCfg<D>::kFwdSmem, s, tm_W, a);
}

template <int D>
hg_status dx_t(const HeadBwdArgs& a, cudaStream_t s) {
  HG_TRY(smem_once<D>());
  CUtensorMap tm_W, tm_dA;
  HG_TRY(make_tmap_bf16(&tm_W, a.W1, D, D, D));
  HG_TRY(make_tmap_bf16(&tm_dA, a.dA, (uint64_t)a.n, D, kRows));
  return launch("head_dx_tc", head_dx_tc_kernel<D>, dim3((unsigned)ceil_div(a.n, kRows)), dim3(kThreads),
                (size_t)HeadTcCfg<D>::kDxSmem, s, tm_W, tm_dA, a);
}

}  // namespace

hg_status head_fwd_tc(int d, const HeadFwdArgs& a, cudaStream_t s) {
  if (a.n <= 0) return HG_OK;
  if (d == 64) return fwd_t<64>(a, s);
  if (d == 128) return fwd_t<128>(a, s);
  if (d == 256) return fwd_t<256>(a, s);
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}

hg_status head_dx_tc(int d, const HeadBwdArgs& a, cudaStream_t s) {
  if (a.n <= 0) return HG_OK;
  if (d == 64) return dx_t<64>(a, s);
  if (d == 128) return dx_t<128>(a, s);
  if (d == 256) return dx_t<256>(a, s);
  set_error("unsupported feature width %d", d);
  return HG_ERR_UNSUPPORTED;
}

}  // namespace hg
