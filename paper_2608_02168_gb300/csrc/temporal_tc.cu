// Tensor-core kernels of the bf16 temporal module (Section 3.2, Eq. 12-13), d in {64, 128}.
//
// All operands are 128-byte-swizzled shared-memory tiles loaded by TMA; every product runs on
// tcgen05 with fp32 accumulators in tensor memory, and thread t of the 128-thread CTA owns row t of
// the 128-node tile in the epilogues.
//
//   temporal_attn_tc   Eq. 12 forward: U_k = C_k W_a for the w context tiles (W_a MN-major), then
//                      per row e_k = r . tanh(U_k), a = softmax(e), H~ = sum_k a_k c_k (c_k read back
//                      from the swizzled tiles), H~ rounded to bf16 and saved with a.
//   temporal_gru_tc    Eq. 13: the gate products x W_i (phase 1) and H~ W_h (phase 2, W_h loaded into
//                      the buffer W_i used) into four accumulators (r and z summed over both phases,
//                      the two parts of n apart); the forward epilogue writes H^t, the backward one
//                      the gate gradients dpre_r, dpre_z, dpre_n, dhn, the direct gradient z dH^t and
//                      the column partials of the first four.
//   temporal_dx_tc     dX = [dpre_r | dpre_z | dpre_n] W_i^T and dH~ = z dH^t + [dpre_r | dpre_z | dhn] W_h^T
//                      with W_i, W_h read as K-major operands as stored (no transpose).
//   temporal_attn_bwd_tc  persistent: U_k recomputed, per row da_k = <dH~, c_k>, de = a (da - sum a da),
//                      P_k = de_k r (1 - tanh(U_k)^2) written as a bf16 tile, and dW_a += C_k^T P_k
//                      accumulated in tensor memory over all of the CTA's tiles; dr = sum de_k tanh(U_k)
//                      by warp transposed sums.
#include <algorithm>

#include "layer_kernels.cuh"
#include "tc_util.cuh"
#include "temporal_kernels.cuh"

namespace hg {

using namespace tc;

namespace {

constexpr int kRows = 128;
constexpr int kABlk = kRows * 128;  // one 64-column block of a 128-row tile
// Four warps per 32-lane quarter of tensor memory: warp w reads lanes 32 (w % 4) .. + 31 (rows of the
// tile) and the column group w / 4, so sixteen warps share each epilogue.
constexpr int kGroups = 4;
constexpr int kThreads = 128 * kGroups;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

template <int D>
struct TCfg {
  static constexpr int NB = D / 64;
  static constexpr int kWBlk = D * 128;  // a 64-column block of a D-row weight
  static constexpr int kW = NB * kWBlk;  // D x D bf16
  static constexpr int kA = NB * kABlk;  // 128 x D bf16
};

__device__ __forceinline__ float sigm(float x) {
  const float e = expf(-fabsf(x));
  return x >= 0.f ? 1.f / (1.f + e) : e / (1.f + e);
}

// Sum over the warp of v[L], returned to lane L (fixed butterfly order).
__device__ __forceinline__ float tsum32(float (&v)[32]) {
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

// Sum over the warp of v[L & 15], returned to lanes L and L + 16.
__device__ __forceinline__ float tsum16(float (&v)[16]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < 16; ++i) v[i] += __shfl_xor_sync(0xffffffffu, v[i], 16);
#pragma unroll
  for (int s = 8; s >= 1; s >>= 1) {
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

// Sum over the warp of v[L & 7], returned to lanes L, L + 8, L + 16 and L + 24.
__device__ __forceinline__ float tsum8(float (&v)[8]) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    v[i] += __shfl_xor_sync(0xffffffffu, v[i], 16);
    v[i] += __shfl_xor_sync(0xffffffffu, v[i], 8);
  }
#pragma unroll
  for (int s = 4; s >= 1; s >>= 1) {
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

// 8 bf16 of row `row` starting at column c (a multiple of 8) of a swizzled K-major tile.
__device__ __forceinline__ void tile_row8(const uint8_t* tile, int row, int c, float* f) {
  unpack(ld16(tile + (c >> 6) * kABlk + sw128_offset(row, (c & 63) * 2)), f, __nv_bfloat16());
}
__device__ __forceinline__ void tile_put8(uint8_t* tile, int row, int c, const float* f) {
  st16(tile + (c >> 6) * kABlk + sw128_offset(row, (c & 63) * 2), pack(f, __nv_bfloat16()));
}

// K-major A (rows x 64-column blocks) times MN-major B (K rows x N in 64-column blocks), K = D:
// D / 16 instructions into `acc`.
template <int D>
__device__ __forceinline__ void mma_kmaj_mn(uint32_t acc, uint32_t A, uint32_t B, uint32_t idesc, bool accumulate) {
#pragma unroll
  for (int j = 0; j < D / 16; ++j)
    mma_bf16(acc, desc_sw128(A + (j >> 2) * kABlk + (j & 3) * 32, 16, 1024),
             desc_sw128(B + j * 2048, TCfg<D>::kWBlk, 1024), idesc, (accumulate || j > 0) ? 1u : 0u);
}

struct TAttnArgs {
  int64_t n;
  int w;
  const __nv_bfloat16* r;
  __nv_bfloat16* Ht;
  float* a;
  int* status;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    temporal_attn_tc(const __grid_constant__ CUtensorMap tm_C, const __grid_constant__ CUtensorMap tm_Wa, TAttnArgs p) {
  using C = TCfg<D>;
  constexpr int CW = D / kGroups;  // columns of a warp's group
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Wimg = smem;
  uint8_t* Cimg = smem + C::kW;
  uint64_t* bars = reinterpret_cast<uint64_t*>(Cimg + p.w * C::kA);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
  float* rf = reinterpret_cast<float*>(bars + 4);
  float* epart = rf + D;  // [kGroups][w][128]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q = warp & 3, cg = warp >> 2;
  const int row = q * 32 + lane;
  const int64_t r0 = (int64_t)blockIdx.x * kRows;
  uint32_t tcols = 32;
  while (tcols < (uint32_t)(p.w * D)) tcols <<= 1;
  if (tid == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, tcols);
  for (int c = tid; c < D; c += kThreads) rf[c] = __bfloat162float(p.r[c]);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  bool ok = true;
  IssueLog<3> lg;  // thread 0's copies and MMAs, for the give-up path
  if (tid == 0) {
    mbar_expect_tx(&bars[0], (uint32_t)(C::kW + p.w * C::kA));
    lg.begin(0);
    for (int b = 0; b < C::NB; ++b) tma_load_2d(Wimg + b * C::kWBlk, &tm_Wa, b * 64, 0, &bars[0]);
    for (int k = 0; k < p.w; ++k)
      for (int b = 0; b < C::NB; ++b)
        tma_load_2d(Cimg + k * C::kA + b * kABlk, &tm_C, b * 64, (int)(k * p.n + r0), &bars[0]);
    ok = mbar_wait(&bars[0], 0);
    if (ok) {
      fence_after_sync();
      const uint32_t idesc = idesc_bf16(128, D, false, true);
      for (int k = 0; k < p.w; ++k)
        mma_kmaj_mn<D>(tmem + k * D, smem_u32(Cimg + k * C::kA), smem_u32(Wimg), idesc, false);
      mma_commit(&bars[1]);
      lg.begin(1);
    } else {
      record_device_error(p.status, kErrTimeout);
    }
  }
  ok = __syncthreads_and(ok);
  if (ok && !mbar_wait(&bars[1], 0)) {
    record_device_error(p.status, kErrTimeout);
    ok = false;
  }
  fence_after_sync();
  const int64_t r = r0 + row;
  const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + cg * CW;
  // partial scores over this warp's columns, combined over the groups in order
  for (int k = 0; k < p.w; ++k) {
    float s = 0.f;
#pragma unroll
    for (int c = 0; c < CW; c += 8) {
      float u[8];
      tmem_ld8(trow + k * D + c, u);
#pragma unroll
      for (int e = 0; e < 8; ++e) s = fmaf(rf[cg * CW + c + e], tanhf(u[e]), s);
    }
    epart[(cg * p.w + k) * kRows + row] = s;
  }
  __syncthreads();
  float e[kTemporalMaxW];
  float m = -INFINITY;
#pragma unroll
  for (int k = 0; k < kTemporalMaxW; ++k) {
    if (k >= p.w) break;
    float s = 0.f;
#pragma unroll
    for (int g = 0; g < kGroups; ++g) s += epart[(g * p.w + k) * kRows + row];
    e[k] = s;
    m = fmaxf(m, s);
  }
  float sum = 0.f;
#pragma unroll
  for (int k = 0; k < kTemporalMaxW; ++k) {
    if (k >= p.w) break;
    e[k] = expf(e[k] - m);
    sum += e[k];
  }
#pragma unroll
  for (int k = 0; k < kTemporalMaxW; ++k) {
    if (k >= p.w) break;
    e[k] /= sum;
    if (cg == 0 && r < p.n) p.a[r * p.w + k] = e[k];
  }
  if (r < p.n && ok) {
#pragma unroll
    for (int c = 0; c < CW; c += 8) {
      const int col = cg * CW + c;
      float h[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int k = 0; k < kTemporalMaxW; ++k) {
        if (k >= p.w) break;
        float x[8];
        tile_row8(Cimg + k * C::kA, row, col, x);
#pragma unroll
        for (int t = 0; t < 8; ++t) h[t] = fmaf(e[k], x[t], h[t]);
      }
      st16(p.Ht + r * D + col, pack(h, __nv_bfloat16()));
    }
  }
  fence_before_sync();
  __syncthreads();
  if (!ok && tid == 0) lg.drain(bars);  // give-up path: nothing issued is still in flight
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, tcols);
}

struct TGruArgs {
  int64_t n;
  const __nv_bfloat16* b_i;
  const __nv_bfloat16* b_h;
  __nv_bfloat16* out;         // forward: H^t
  const __nv_bfloat16* dOut;  // backward: dL/dH^t
  __nv_bfloat16* dG;          // backward: [dpre_r; dpre_z; dpre_n; dhn], 4 blocks of n x D
  __nv_bfloat16* dh;          // backward: z dH^t
  float* part;                // backward: [grid][4 D] column partials of the four dG blocks
  int* status;
};

// Phase 1: acc_g = x W_i[:, gD..] (g < 3); phase 2: acc_r, acc_z += H~ W_h[:, ..2D], acc_3 = H~ W_h[:, 2D..].
template <int D, bool kBwd>
__global__ void __launch_bounds__(kThreads, 1)
    temporal_gru_tc(const __grid_constant__ CUtensorMap tm_X, const __grid_constant__ CUtensorMap tm_Ht,
                    const __grid_constant__ CUtensorMap tm_Wi, const __grid_constant__ CUtensorMap tm_Wh, TGruArgs p) {
  using C = TCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Ximg = smem;
  uint8_t* Himg = Ximg + C::kA;
  uint8_t* Wimg = Himg + C::kA;  // 3 NB blocks of D rows
  uint64_t* bars = reinterpret_cast<uint64_t*>(Wimg + 3 * C::kW);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 4);
  float* bias = reinterpret_cast<float*>(bars + 6);  // b_i (3D) then b_h (3D)
  float* colred = bias + 6 * D;                     // [4 warps][4D] (backward)
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int64_t r0 = (int64_t)blockIdx.x * kRows;
  constexpr uint32_t kCols = 4 * D;
  if (tid == 0) {
    for (int i = 0; i < 3; ++i) mbar_init(&bars[i], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, kCols);
  for (int c = tid; c < 3 * D; c += kThreads) {
    bias[c] = __bfloat162float(p.b_i[c]);
    bias[3 * D + c] = __bfloat162float(p.b_h[c]);
  }
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  bool ok = true;
  IssueLog<3> lg;  // thread 0's copies and MMAs, for the give-up path
  if (tid == 0) {
    const uint32_t idesc = idesc_bf16(128, D, false, true);
    mbar_expect_tx(&bars[0], (uint32_t)(2 * C::kA + 3 * C::kW));
    lg.begin(0);
    for (int b = 0; b < C::NB; ++b) {
      tma_load_2d(Ximg + b * kABlk, &tm_X, b * 64, (int)r0, &bars[0]);
      tma_load_2d(Himg + b * kABlk, &tm_Ht, b * 64, (int)r0, &bars[0]);
    }
    for (int b = 0; b < 3 * C::NB; ++b) tma_load_2d(Wimg + b * C::kWBlk, &tm_Wi, b * 64, 0, &bars[0]);
    ok = mbar_wait(&bars[0], 0);
    if (ok) {
      fence_after_sync();
      for (int g = 0; g < 3; ++g)
        mma_kmaj_mn<D>(tmem + g * D, smem_u32(Ximg), smem_u32(Wimg + g * C::NB * C::kWBlk), idesc, false);
      mma_commit(&bars[1]);
      lg.begin(1);
      ok = mbar_wait(&bars[1], 0);  // W_i no longer read: load W_h into its buffer
    }
    if (ok) {
      mbar_expect_tx(&bars[0], (uint32_t)(3 * C::kW));
      lg.begin(0);
      for (int b = 0; b < 3 * C::NB; ++b) tma_load_2d(Wimg + b * C::kWBlk, &tm_Wh, b * 64, 0, &bars[0]);
      ok = mbar_wait(&bars[0], 1);
    }
    if (ok) {
      fence_after_sync();
      mma_kmaj_mn<D>(tmem + 0 * D, smem_u32(Himg), smem_u32(Wimg), idesc, true);
      mma_kmaj_mn<D>(tmem + 1 * D, smem_u32(Himg), smem_u32(Wimg + C::NB * C::kWBlk), idesc, true);
      mma_kmaj_mn<D>(tmem + 3 * D, smem_u32(Himg), smem_u32(Wimg + 2 * C::NB * C::kWBlk), idesc, false);
      mma_commit(&bars[2]);
      lg.begin(2);
    }
    if (!ok) record_device_error(p.status, kErrTimeout);
  }
  ok = __syncthreads_and(ok);
  if (ok && !mbar_wait(&bars[2], 0)) {
    record_device_error(p.status, kErrTimeout);
    ok = false;
  }
  fence_after_sync();
  constexpr int CW = D / kGroups;
  const int q = warp & 3, cg = warp >> 2;
  const int row = q * 32 + lane;
  const int64_t r = r0 + row;
  const bool live = ok && r < p.n;
  const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
#pragma unroll
  for (int c0 = 0; c0 < CW; c0 += 8) {
    const int c = cg * CW + c0;
    float ar[8], az[8], anx[8], anh[8], h[8], g[8];
    tmem_ld8(trow + 0 * D + c, ar);
    tmem_ld8(trow + 1 * D + c, az);
    tmem_ld8(trow + 2 * D + c, anx);
    tmem_ld8(trow + 3 * D + c, anh);
    tile_row8(Himg, row, c, h);
    if (kBwd) {
      if (live) {
        unpack(ld16(p.dOut + r * D + c), g, __nv_bfloat16());
      } else {
#pragma unroll
        for (int t = 0; t < 8; ++t) g[t] = 0.f;
      }
    }
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const int col = c + t;
      const float rg = sigm(ar[t] + bias[col] + bias[3 * D + col]);
      const float z = sigm(az[t] + bias[D + col] + bias[4 * D + col]);
      const float hn = anh[t] + bias[5 * D + col];
      const float nn = tanhf(anx[t] + bias[2 * D + col] + rg * hn);
      if (!kBwd) {
        ar[t] = (1.f - z) * nn + z * h[t];
      } else {
        const float dn = g[t] * (1.f - z);
        const float dz = g[t] * (h[t] - nn);
        const float dpn = dn * (1.f - nn * nn);
        ar[t] = dpn * hn * rg * (1.f - rg);  // dpre_r
        az[t] = dz * z * (1.f - z);          // dpre_z
        anx[t] = dpn;                        // dpre_n
        anh[t] = dpn * rg;                   // dhn
        h[t] = g[t] * z;                     // direct gradient of H~
      }
    }
    if (!kBwd) {
      if (live) st16(p.out + r * D + c, pack(ar, __nv_bfloat16()));
    } else {
      if (live) {
        __nv_bfloat16* dst = p.dG + r * D + c;
        const int64_t blk = p.n * D;
        st16(dst, pack(ar, __nv_bfloat16()));
        st16(dst + blk, pack(az, __nv_bfloat16()));
        st16(dst + 2 * blk, pack(anx, __nv_bfloat16()));
        st16(dst + 3 * blk, pack(anh, __nv_bfloat16()));
        st16(p.dh + r * D + c, pack(h, __nv_bfloat16()));
      }
      const float s0 = tsum8(ar), s1 = tsum8(az), s2 = tsum8(anx), s3 = tsum8(anh);
      if (lane < 8) {
        float* cr = colred + q * 4 * D + c + lane;
        cr[0 * D] = s0;
        cr[1 * D] = s1;
        cr[2 * D] = s2;
        cr[3 * D] = s3;
      }
    }
  }
  if (kBwd) {
    __syncthreads();
    for (int t = tid; t < 4 * D; t += kThreads)
      p.part[(int64_t)blockIdx.x * 4 * D + t] =
          ((colred[t] + colred[4 * D + t]) + colred[8 * D + t]) + colred[12 * D + t];
  }
  fence_before_sync();
  __syncthreads();
  if (!ok && tid == 0) lg.drain(bars);  // give-up path: nothing issued is still in flight
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kCols);
}

struct TDxArgs {
  int64_t n;
  const __nv_bfloat16* dh;  // z dH^t
  __nv_bfloat16* dX;
  __nv_bfloat16* dHt;
  int* status;
};

// K-major A (three gate tiles, K = 3D) times K-major B (D rows x 3D, as stored): 3 D / 16 instructions.
template <int D>
__device__ __forceinline__ void mma_gates_kmaj(uint32_t acc, const uint32_t (&A)[3], uint32_t B, uint32_t idesc) {
#pragma unroll
  for (int g = 0; g < 3; ++g)
#pragma unroll
    for (int j = 0; j < D / 16; ++j)
      mma_bf16(acc, desc_sw128(A[g] + (j >> 2) * kABlk + (j & 3) * 32, 16, 1024),
               desc_sw128(B + (g * TCfg<D>::NB + (j >> 2)) * TCfg<D>::kWBlk + (j & 3) * 32, 16, 1024), idesc,
               (g > 0 || j > 0) ? 1u : 0u);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    temporal_dx_tc(const __grid_constant__ CUtensorMap tm_dG, const __grid_constant__ CUtensorMap tm_Wi,
                   const __grid_constant__ CUtensorMap tm_Wh, TDxArgs p) {
  using C = TCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Aimg = smem;                // 3 tiles: dpre_r, dpre_z, then dpre_n / dhn
  uint8_t* Wimg = Aimg + 3 * C::kA;    // 3 NB blocks of D rows
  uint64_t* bars = reinterpret_cast<uint64_t*>(Wimg + 3 * C::kW);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 4);
  const int tid = threadIdx.x, warp = tid >> 5;
  const int64_t r0 = (int64_t)blockIdx.x * kRows;
  constexpr uint32_t kCols = 2 * D;
  if (tid == 0) {
    for (int i = 0; i < 3; ++i) mbar_init(&bars[i], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, kCols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  bool ok = true;
  IssueLog<3> lg;  // thread 0's copies and MMAs, for the give-up path
  if (tid == 0) {
    const uint32_t idesc = idesc_bf16(128, D, false, false);
    const uint32_t A[3] = {smem_u32(Aimg), smem_u32(Aimg + C::kA), smem_u32(Aimg + 2 * C::kA)};
    mbar_expect_tx(&bars[0], (uint32_t)(3 * C::kA + 3 * C::kW));
    lg.begin(0);
    for (int g = 0; g < 3; ++g)
      for (int b = 0; b < C::NB; ++b)
        tma_load_2d(Aimg + g * C::kA + b * kABlk, &tm_dG, b * 64, (int)(g * p.n + r0), &bars[0]);
    for (int b = 0; b < 3 * C::NB; ++b) tma_load_2d(Wimg + b * C::kWBlk, &tm_Wi, b * 64, 0, &bars[0]);
    ok = mbar_wait(&bars[0], 0);
    if (ok) {
      fence_after_sync();
      mma_gates_kmaj<D>(tmem, A, smem_u32(Wimg), idesc);
      mma_commit(&bars[1]);
      lg.begin(1);
      ok = mbar_wait(&bars[1], 0);  // third tile and W_i no longer read
    }
    if (ok) {
      mbar_expect_tx(&bars[0], (uint32_t)(C::kA + 3 * C::kW));
      lg.begin(0);
      for (int b = 0; b < C::NB; ++b)
        tma_load_2d(Aimg + 2 * C::kA + b * kABlk, &tm_dG, b * 64, (int)(3 * p.n + r0), &bars[0]);
      for (int b = 0; b < 3 * C::NB; ++b) tma_load_2d(Wimg + b * C::kWBlk, &tm_Wh, b * 64, 0, &bars[0]);
      ok = mbar_wait(&bars[0], 1);
    }
    if (ok) {
      fence_after_sync();
      mma_gates_kmaj<D>(tmem + D, A, smem_u32(Wimg), idesc);
      mma_commit(&bars[2]);
      lg.begin(2);
    }
    if (!ok) record_device_error(p.status, kErrTimeout);
  }
  ok = __syncthreads_and(ok);
  if (ok && !mbar_wait(&bars[2], 0)) {
    record_device_error(p.status, kErrTimeout);
    ok = false;
  }
  fence_after_sync();
  constexpr int CW = D / kGroups;
  const int q = warp & 3, cg = warp >> 2, lane = tid & 31;
  const int64_t r = r0 + q * 32 + lane;
  const bool live = ok && r < p.n;
  const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16);
#pragma unroll
  for (int c0 = 0; c0 < CW; c0 += 8) {
    const int c = cg * CW + c0;
    float x[8], h[8];
    tmem_ld8(trow + c, x);
    tmem_ld8(trow + D + c, h);
    if (live) {
      float d0[8];
      unpack(ld16(p.dh + r * D + c), d0, __nv_bfloat16());
#pragma unroll
      for (int t = 0; t < 8; ++t) h[t] += d0[t];
      st16(p.dX + r * D + c, pack(x, __nv_bfloat16()));
      st16(p.dHt + r * D + c, pack(h, __nv_bfloat16()));
    }
  }
  fence_before_sync();
  __syncthreads();
  if (!ok && tid == 0) lg.drain(bars);  // give-up path: nothing issued is still in flight
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, kCols);
}

struct TAttnBwdArgs {
  int64_t n;
  int w;
  int tiles;
  const __nv_bfloat16* r;
  const float* a;
  const __nv_bfloat16* dHt;
  float* dWa_part;  // [grid][D x D]
  float* dr_part;   // [grid][D]
  int* status;
};

// Persistent: the CTA's tiles in turn; TMEM holds U_0..U_{w-1} (w D columns) and the dW_a
// accumulator (D columns after them).
template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    temporal_attn_bwd_tc(const __grid_constant__ CUtensorMap tm_C, const __grid_constant__ CUtensorMap tm_Wa,
                         TAttnBwdArgs p) {
  using C = TCfg<D>;
  constexpr int CW = D / kGroups;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Wimg = smem;
  uint8_t* Cimg = smem + C::kW;              // w tiles
  uint8_t* Pimg = Cimg + p.w * C::kA;        // one tile (followed by at least one block of shared memory)
  uint64_t* bars = reinterpret_cast<uint64_t*>(Pimg + C::kA + kABlk);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 4);
  float* rf = reinterpret_cast<float*>(bars + 6);
  float* drred = rf + D;                    // [4 quarters][D]
  float* dapart = drred + 4 * D;            // [kGroups][w][128]
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q = warp & 3, cg = warp >> 2;
  const int row = q * 32 + lane;
  uint32_t tcols = 32;
  while (tcols < (uint32_t)((p.w + 1) * D)) tcols <<= 1;
  if (tid == 0) {
    for (int i = 0; i < 3; ++i) mbar_init(&bars[i], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, tcols);
  for (int c = tid; c < D; c += kThreads) rf[c] = __bfloat162float(p.r[c]);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  const uint32_t acc_w = tmem + p.w * D;
  const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + cg * CW;
  float drl[CW / 8];
#pragma unroll
  for (int i = 0; i < CW / 8; ++i) drl[i] = 0.f;
  bool ok = true;
  IssueLog<3> lg;  // thread 0's copies and MMAs, for the give-up path
  uint32_t it = 0, mm = 0;  // tiles done, dW_a commits done
  for (int t = blockIdx.x; t < p.tiles && ok; t += gridDim.x, ++it) {
    const int64_t r0 = (int64_t)t * kRows;
    if (tid == 0) {
      const uint32_t bytes = (uint32_t)(p.w * C::kA + (it == 0 ? C::kW : 0));
      mbar_expect_tx(&bars[0], bytes);
      lg.begin(0);
      if (it == 0)
        for (int b = 0; b < C::NB; ++b) tma_load_2d(Wimg + b * C::kWBlk, &tm_Wa, b * 64, 0, &bars[0]);
      for (int k = 0; k < p.w; ++k)
        for (int b = 0; b < C::NB; ++b)
          tma_load_2d(Cimg + k * C::kA + b * kABlk, &tm_C, b * 64, (int)(k * p.n + r0), &bars[0]);
      ok = mbar_wait(&bars[0], it & 1);
      if (ok) {
        fence_after_sync();
        const uint32_t idesc = idesc_bf16(128, D, false, true);
        for (int k = 0; k < p.w; ++k)
          mma_kmaj_mn<D>(tmem + k * D, smem_u32(Cimg + k * C::kA), smem_u32(Wimg), idesc, false);
        mma_commit(&bars[1]);
        lg.begin(1);
      }
    }
    ok = __syncthreads_and(ok);
    if (!ok) break;
    if (!mbar_wait(&bars[1], it & 1)) ok = false;
    ok = __syncthreads_and(ok);
    if (!ok) break;
    fence_after_sync();
    const int64_t r = r0 + row;
    const bool live = r < p.n;
    // partial da_k = <dH~, c_k> over this warp's columns, combined over the groups in order
    {
      float da[kTemporalMaxW];
#pragma unroll
      for (int k = 0; k < kTemporalMaxW; ++k) da[k] = 0.f;
      if (live) {
#pragma unroll
        for (int c0 = 0; c0 < CW; c0 += 8) {
          const int col = cg * CW + c0;
          float g[8];
          unpack(ld16(p.dHt + r * D + col), g, __nv_bfloat16());
#pragma unroll
          for (int k = 0; k < kTemporalMaxW; ++k) {
            if (k >= p.w) break;
            float x[8];
            tile_row8(Cimg + k * C::kA, row, col, x);
#pragma unroll
            for (int e = 0; e < 8; ++e) da[k] = fmaf(g[e], x[e], da[k]);
          }
        }
      }
#pragma unroll
      for (int k = 0; k < kTemporalMaxW; ++k) {
        if (k >= p.w) break;
        dapart[(cg * p.w + k) * kRows + row] = da[k];
      }
    }
    __syncthreads();
    float de[kTemporalMaxW];
    {
      float da[kTemporalMaxW];
      float s = 0.f;
#pragma unroll
      for (int k = 0; k < kTemporalMaxW; ++k) {
        if (k >= p.w) break;
        float v = 0.f;
#pragma unroll
        for (int g = 0; g < kGroups; ++g) v += dapart[(g * p.w + k) * kRows + row];
        da[k] = v;
        de[k] = live ? p.a[r * p.w + k] : 0.f;
        s = fmaf(de[k], v, s);
      }
#pragma unroll
      for (int k = 0; k < kTemporalMaxW; ++k) {
        if (k >= p.w) break;
        de[k] = de[k] * (da[k] - s);
      }
    }
    for (int k = 0; k < p.w; ++k) {
      float dek = 0.f;
#pragma unroll
      for (int kk = 0; kk < kTemporalMaxW; ++kk)
        if (kk == k) dek = de[kk];
#pragma unroll
      for (int c0 = 0; c0 < CW; c0 += 8) {
        const int col = cg * CW + c0;
        float u[8], pk[8];
        tmem_ld8(trow + k * D + c0, u);
#pragma unroll
        for (int e = 0; e < 8; ++e) {
          const float th = tanhf(u[e]);
          pk[e] = dek * rf[col + e] * (1.f - th * th);
          u[e] = dek * th;
        }
        tile_put8(Pimg, row, col, pk);
        const float cs = tsum8(u);
#pragma unroll
        for (int i = 0; i < CW / 8; ++i)
          if (i == c0 / 8) drl[i] += cs;
      }
      fence_async_smem();
      __syncthreads();
      if (tid == 0) {
        fence_after_sync();
        // dW_a += C_k^T P_k: both operands MN-major over the tile's 128 rows (K), M = 128 (rows of
        // dW_a past D read whatever follows the tile and are never stored)
        const uint32_t idesc = idesc_bf16(128, D, true, true);
        const uint32_t A = smem_u32(Cimg + k * C::kA), B = smem_u32(Pimg);
#pragma unroll
        for (int j = 0; j < kRows / 16; ++j)
          mma_bf16(acc_w, desc_sw128(A + j * 2048, kABlk, 1024), desc_sw128(B + j * 2048, kABlk, 1024), idesc,
                   (it > 0 || k > 0 || j > 0) ? 1u : 0u);
        mma_commit(&bars[2]);
        lg.begin(2);
      }
      if (!mbar_wait(&bars[2], mm & 1)) ok = false;
      ++mm;
      ok = __syncthreads_and(ok);
      if (!ok) break;
      fence_after_sync();
    }
  }
  if (!ok) record_device_error(p.status, kErrTimeout);
  // dW_a partial: TMEM lane t holds row t of the accumulator (rows < D are the gradient's); the four
  // column groups write their columns
  float* outw = p.dWa_part + (int64_t)blockIdx.x * D * D;
#pragma unroll
  for (int c0 = 0; c0 < CW; c0 += 8) {
    float v[8];
    tmem_ld8(tmem + ((uint32_t)(q * 32) << 16) + p.w * D + cg * CW + c0, v);
    if (row < D) {
      const bool good = ok && it > 0;
      float* o = outw + (int64_t)row * D + cg * CW + c0;
      *reinterpret_cast<float4*>(o) = good ? make_float4(v[0], v[1], v[2], v[3]) : make_float4(0.f, 0.f, 0.f, 0.f);
      *reinterpret_cast<float4*>(o + 4) = good ? make_float4(v[4], v[5], v[6], v[7]) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
  }
  // dr partial: lane L of a warp holds column (L & 7) of each of its 8-column chunks
  if (lane < 8) {
#pragma unroll
    for (int i = 0; i < CW / 8; ++i) drred[q * D + cg * CW + i * 8 + lane] = drl[i];
  }
  fence_before_sync();
  __syncthreads();
  for (int c = tid; c < D; c += kThreads)
    p.dr_part[(int64_t)blockIdx.x * D + c] = ((drred[c] + drred[D + c]) + drred[2 * D + c]) + drred[3 * D + c];
  if (!ok && tid == 0) lg.drain(bars);  // give-up path: nothing issued is still in flight
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, tcols);
}

// dst[row][g D + c] = G[c][row]: the transposed block of a gate (d x d into d x 3d).
__global__ void temporal_place_t(const float* __restrict__ G, int d, int g, float* __restrict__ dst) {
  for (int q = blockIdx.x * blockDim.x + threadIdx.x; q < d * d; q += gridDim.x * blockDim.x) {
    const int row = q / d, c = q % d;
    dst[(int64_t)row * 3 * d + g * d + c] = G[(int64_t)c * d + row];
  }
}

// db_i = [s_r, s_z, s_n], db_h = [s_r, s_z, s_hn] from the four column sums s (4 d).
__global__ void temporal_bias_finish(const float* __restrict__ s, int d, float* __restrict__ db_i,
                                     float* __restrict__ db_h) {
  for (int q = blockIdx.x * blockDim.x + threadIdx.x; q < 3 * d; q += gridDim.x * blockDim.x) {
    db_i[q] = s[q];
    db_h[q] = q < 2 * d ? s[q] : s[q + d];
  }
}

int num_sms() {
  static int sms = 0;
  if (!sms) {
    int dev = 0;
    cudaGetDevice(&dev);
    if (cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || sms <= 0) sms = 148;
  }
  return sms;
}

// Tensor-memory columns a kernel allocates (a power of two >= 32).
inline uint32_t tmem_cols(int need) {
  uint32_t c = 32;
  while (c < (uint32_t)need) c <<= 1;
  return c;
}

// Dynamic shared memory of a launch: what the kernel uses, raised so that no more CTAs share an SM
// than its 512 tensor-memory columns hold (233,472 bytes of shared memory per SM, 1 KB reserved
// per CTA), so that every tcgen05.alloc is served at once.
inline size_t smem_for(size_t need, uint32_t tcols) {
  const size_t ctas = 512 / tcols;
  const size_t floor = 233472 / (ctas + 1) - 1024 + 16;
  return std::max(need, floor);
}

template <int D>
size_t attn_smem(int w) {
  return smem_for((size_t)TCfg<D>::kW + (size_t)w * TCfg<D>::kA + 32 + 4 * D + 4 * kGroups * w * kRows + 1024,
                  tmem_cols(w * D));
}
template <int D>
size_t gru_smem() { return smem_for(2 * TCfg<D>::kA + 3 * TCfg<D>::kW + 48 + 88 * D + 1024, 4 * D); }
template <int D>
size_t dx_smem() { return smem_for(3 * TCfg<D>::kA + 3 * TCfg<D>::kW + 48 + 1024, 2 * D); }
template <int D>
size_t attn_bwd_smem(int w) {
  // persistent: one CTA per SM
  return smem_for((size_t)TCfg<D>::kW + (size_t)(w + 1) * TCfg<D>::kA + kABlk + 48 + 20 * D +
                      4 * kGroups * w * kRows + 1024, 512);
}

template <int D>
hg_status smem_attrs() {
  static bool done = false;
  if (!done) {
    const int big = 232448;  // the largest dynamic shared memory a CTA may request
    HG_CUDA(cudaFuncSetAttribute(temporal_attn_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, big));
    HG_CUDA(cudaFuncSetAttribute(temporal_gru_tc<D, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, big));
    HG_CUDA(cudaFuncSetAttribute(temporal_gru_tc<D, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, big));
    HG_CUDA(cudaFuncSetAttribute(temporal_dx_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, big));
    HG_CUDA(cudaFuncSetAttribute(temporal_attn_bwd_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, big));
    done = true;
  }
  return HG_OK;
}

template <int D>
hg_status fwd_tc_t(const TemporalTcIn& in, void* H_out, cudaStream_t s) {
  HG_TRY(smem_attrs<D>());
  const int64_t n = in.n;
  const int w = in.p->w;
  const unsigned tiles = (unsigned)ceil_div(n, kRows);
  CUtensorMap tm_C, tm_Wa, tm_X, tm_Ht, tm_Wi, tm_Wh;
  HG_TRY(make_tmap_bf16(&tm_C, in.C, (uint64_t)(w * n), D, kRows));
  HG_TRY(make_tmap_bf16(&tm_Wa, in.p->Wa, D, D, D));
  HG_TRY(make_tmap_bf16(&tm_X, in.X, (uint64_t)n, D, kRows));
  HG_TRY(make_tmap_bf16(&tm_Ht, in.Ht, (uint64_t)n, D, kRows));
  HG_TRY(make_tmap_bf16(&tm_Wi, in.p->W_i, D, 3 * D, D));
  HG_TRY(make_tmap_bf16(&tm_Wh, in.p->W_h, D, 3 * D, D));
  TAttnArgs a{n, w, (const __nv_bfloat16*)in.p->r, (__nv_bfloat16*)in.Ht, in.a, device_status_ptr()};
  HG_TRY(launch("temporal_attn_tc", temporal_attn_tc<D>, dim3(tiles), dim3(kThreads), attn_smem<D>(w), s, tm_C, tm_Wa,
                a));
  TGruArgs g{n, (const __nv_bfloat16*)in.p->b_i, (const __nv_bfloat16*)in.p->b_h, (__nv_bfloat16*)H_out, nullptr,
             nullptr, nullptr, nullptr, device_status_ptr()};
  return launch("temporal_gru_tc", temporal_gru_tc<D, false>, dim3(tiles), dim3(kThreads), gru_smem<D>(), s, tm_X,
                tm_Ht, tm_Wi, tm_Wh, g);
}

template <int D>
hg_status bwd_tc_t(const TemporalTcIn& in, const void* dOut, void* dX, const hg_temporal_grads* gr,
                   const TemporalTcScratch& sc, cudaStream_t s) {
  HG_TRY(smem_attrs<D>());
  const int64_t n = in.n;
  const int w = in.p->w;
  const unsigned tiles = (unsigned)ceil_div(n, kRows);
  CUtensorMap tm_C, tm_Wa, tm_X, tm_Ht, tm_Wi, tm_Wh, tm_dG;
  HG_TRY(make_tmap_bf16(&tm_C, in.C, (uint64_t)(w * n), D, kRows));
  HG_TRY(make_tmap_bf16(&tm_Wa, in.p->Wa, D, D, D));
  HG_TRY(make_tmap_bf16(&tm_X, in.X, (uint64_t)n, D, kRows));
  HG_TRY(make_tmap_bf16(&tm_Ht, in.Ht, (uint64_t)n, D, kRows));
  HG_TRY(make_tmap_bf16(&tm_Wi, in.p->W_i, D, 3 * D, D));
  HG_TRY(make_tmap_bf16(&tm_Wh, in.p->W_h, D, 3 * D, D));
  HG_TRY(make_tmap_bf16(&tm_dG, sc.dG, (uint64_t)(4 * n), D, kRows));
  // gate gradients (Eq. 13 backward) and their column sums
  TGruArgs g{n, (const __nv_bfloat16*)in.p->b_i, (const __nv_bfloat16*)in.p->b_h, nullptr,
             (const __nv_bfloat16*)dOut, (__nv_bfloat16*)sc.dG, (__nv_bfloat16*)sc.dh, sc.part, device_status_ptr()};
  HG_TRY(launch("temporal_gru_bwd_tc", temporal_gru_tc<D, true>, dim3(tiles), dim3(kThreads), gru_smem<D>(), s, tm_X,
                tm_Ht, tm_Wi, tm_Wh, g));
  HG_TRY(reduce_partials(sc.part, 4 * D, (int)tiles, 4 * D, sc.sums, sc.tmp, s));
  HG_TRY(launch("temporal_bias_finish", temporal_bias_finish, dim3(1), dim3(256), 0, s, (const float*)sc.sums, D,
                gr->db_i, gr->db_h));
  // dX and dH~
  TDxArgs x{n, (const __nv_bfloat16*)sc.dh, (__nv_bfloat16*)dX, (__nv_bfloat16*)sc.dHt, device_status_ptr()};
  HG_TRY(launch("temporal_dx_tc", temporal_dx_tc<D>, dim3(tiles), dim3(kThreads), dx_smem<D>(), s, tm_dG, tm_Wi,
                tm_Wh, x));
  // Eq. 12 backward: dW_a and dr
  const int grid = std::max(1, std::min((int)tiles, num_sms()));
  TAttnBwdArgs b{n, w, (int)tiles, (const __nv_bfloat16*)in.p->r, in.a, (const __nv_bfloat16*)sc.dHt, sc.part,
                 sc.part + (int64_t)grid * D * D, device_status_ptr()};
  HG_TRY(launch("temporal_attn_bwd_tc", temporal_attn_bwd_tc<D>, dim3(grid), dim3(kThreads), attn_bwd_smem<D>(w), s,
                tm_C, tm_Wa, b));
  HG_TRY(reduce_partials(sc.part, (int64_t)D * D, grid, (int64_t)D * D, gr->dWa, sc.tmp, s));
  HG_TRY(reduce_partials(sc.part + (int64_t)grid * D * D, D, grid, D, gr->dr, sc.tmp, s));
  // dW_i = x^T dG_i and dW_h = H~^T dG_h, as (dG_g^T x)^T: the three gate blocks share x (or H~)
  const int64_t x0i[3] = {0, n, 2 * n}, x0h[3] = {0, n, 3 * n};
  float* outs[3] = {sc.G, sc.G + D * D, sc.G + 2 * D * D};
  HG_TRY(tc_weight_grad(D, sc.dG, x0i, 3, in.X, 0, n, sc.part, outs, sc.tmp, s));
  for (int q = 0; q < 3; ++q)
    HG_TRY(launch("temporal_place_t", temporal_place_t, dim3(64), dim3(256), 0, s, (const float*)outs[q], D, q,
                  gr->dW_i));
  HG_TRY(tc_weight_grad(D, sc.dG, x0h, 3, in.Ht, 0, n, sc.part, outs, sc.tmp, s));
  for (int q = 0; q < 3; ++q)
    HG_TRY(launch("temporal_place_t", temporal_place_t, dim3(64), dim3(256), 0, s, (const float*)outs[q], D, q,
                  gr->dW_h));
  return HG_OK;
}

}  // namespace

bool temporal_tc_supported(hg_dtype dt, int d, int w) {
  return dt == HG_BF16 && (d == 64 || d == 128) && (w + 1) * d <= 512;
}

size_t temporal_tc_part_floats(int64_t n, int d) {
  const int64_t tiles = std::max<int64_t>(1, ceil_div(n, kRows));
  const int64_t grid = std::min<int64_t>(tiles, 160);
  const int64_t wg = 3 * (int64_t)wgrad_tc_splits(std::max<int64_t>(n, 1), d) * d * d;
  return (size_t)std::max({tiles * 4 * d, grid * ((int64_t)d * d + d), wg});
}

hg_status temporal_fwd_tc(const TemporalTcIn& in, void* H_out, cudaStream_t s) {
  if (in.n <= 0) return HG_OK;
  if (in.p->d == 64) return fwd_tc_t<64>(in, H_out, s);
  if (in.p->d == 128) return fwd_tc_t<128>(in, H_out, s);
  set_error("temporal tensor-core path: unsupported d=%d", in.p->d);
  return HG_ERR_UNSUPPORTED;
}

hg_status temporal_bwd_tc(const TemporalTcIn& in, const void* dOut, void* dX, const hg_temporal_grads* g,
                          const TemporalTcScratch& sc, cudaStream_t s) {
  if (in.n <= 0) return HG_OK;
  if (in.p->d == 64) return bwd_tc_t<64>(in, dOut, dX, g, sc, s);
  if (in.p->d == 128) return bwd_tc_t<128>(in, dOut, dX, g, sc, s);
  set_error("temporal tensor-core path: unsupported d=%d", in.p->d);
  return HG_ERR_UNSUPPORTED;
}

}  // namespace hg
