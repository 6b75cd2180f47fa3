// Dense row products on the tensor cores (bf16 storage, fp32 accumulation):
//   out[r][ocol0 + c] (=, or +=) scale * sum_k A[r][k] B[k][c] (+ bias[c]),   rows r < n, c < D,
//   k < D, with scale = scale_mul * (*scale_ptr) (scale_ptr a device fp32 scalar, or null for 1):
//   a scalar factor of a weight is applied here in fp32 instead of being folded into B, where the
//   product would have to be rounded to bf16.
// One CTA per 128 rows: the A tile arrives by TMA as a K-major operand, B (D x D, row-major, as
// stored) by TMA as an MN-major operand, one tcgen05 chain puts the 128 x D product in tensor
// memory, and sixteen warps (four per 32-lane quarter, each a column group) add the bias or the
// existing output and store bf16 rows.  Used by the attention layer's key / value / query maps
// and the products of its backward.
#include <algorithm>

#include "layer_kernels.cuh"
#include "tc_util.cuh"

namespace hg {

using namespace tc;

namespace {

constexpr int kRows = 128;
constexpr int kABlk = kRows * 128;
constexpr int kGroups = 4;
constexpr int kThreads = 128 * kGroups;

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

template <int D>
struct GCfg {
  static constexpr int NB = D / 64;
  static constexpr int kWBlk = D * 128;
  static constexpr int kW = NB * kWBlk;
  static constexpr int kA = NB * kABlk;
  static constexpr int kTail = 32 + 4 * D;
  static constexpr int kNeed = kW + kA + kTail + 1024;
};

struct GArgs {
  int64_t n;
  const float* scale_ptr;
  float scale_mul;
  const __nv_bfloat16* bias;
  __nv_bfloat16* out;
  int64_t ldo;
  int ocol0;
  int accumulate;
  int* status;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 1)
    rows_gemm_tc_kernel(const __grid_constant__ CUtensorMap tm_A, const __grid_constant__ CUtensorMap tm_B, GArgs p) {
  using C = GCfg<D>;
  constexpr int CW = D / kGroups;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* Bimg = smem;
  uint8_t* Aimg = smem + C::kW;
  uint64_t* bars = reinterpret_cast<uint64_t*>(Aimg + C::kA);
  uint32_t* tslot = reinterpret_cast<uint32_t*>(bars + 2);
  float* bf = reinterpret_cast<float*>(bars + 4);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int q = warp & 3, cg = warp >> 2;
  const int64_t r0 = (int64_t)blockIdx.x * kRows;
  if (tid == 0) {
    mbar_init(&bars[0], 1);
    mbar_init(&bars[1], 1);
    fence_mbar_init();
  }
  if (warp == 0) tmem_alloc(tslot, D);
  for (int c = tid; c < D; c += kThreads) bf[c] = p.bias ? __bfloat162float(p.bias[c]) : 0.f;
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  bool ok = true;
  if (tid == 0) {
    mbar_expect_tx(&bars[0], (uint32_t)(C::kW + C::kA));
    for (int b = 0; b < C::NB; ++b) {
      tma_load_2d(Bimg + b * C::kWBlk, &tm_B, b * 64, 0, &bars[0]);
      tma_load_2d(Aimg + b * kABlk, &tm_A, b * 64, (int)r0, &bars[0]);
    }
    ok = mbar_wait(&bars[0], 0);
    if (ok) {
      fence_after_sync();
      const uint32_t A = smem_u32(Aimg), B = smem_u32(Bimg);
      const uint32_t idesc = idesc_bf16(128, D, false, true);
#pragma unroll
      for (int j = 0; j < D / 16; ++j)
        mma_bf16(tmem, desc_sw128(A + (j >> 2) * kABlk + (j & 3) * 32, 16, 1024),
                 desc_sw128(B + j * 2048, C::kWBlk, 1024), idesc, j > 0 ? 1u : 0u);
      mma_commit(&bars[1]);
    } else {
      record_device_error(p.status, kErrTimeout);
      mbar_wait(&bars[0], 0);  // give-up path: the loads land before the CTA moves on
    }
  }
  ok = __syncthreads_and(ok);
  if (ok && !mbar_wait(&bars[1], 0)) {
    record_device_error(p.status, kErrTimeout);
    ok = false;
    if (tid == 0) mbar_wait(&bars[1], 0);  // the MMAs issued complete before TMEM is released
  }
  fence_after_sync();
  const int64_t r = r0 + q * 32 + lane;
  const bool live = ok && r < p.n;
  const uint32_t trow = tmem + ((uint32_t)(q * 32) << 16) + cg * CW;
  const float sc = p.scale_mul * (p.scale_ptr ? *p.scale_ptr : 1.f);
#pragma unroll
  for (int c0 = 0; c0 < CW; c0 += 8) {
    const int c = cg * CW + c0;
    float v[8];
    tmem_ld8(trow + c0, v);
    if (live) {
      __nv_bfloat16* o = p.out + r * p.ldo + p.ocol0 + c;
      float x[8];
      if (p.accumulate) {
        unpack(ld16(o), x, __nv_bfloat16());
      } else {
#pragma unroll
        for (int e = 0; e < 8; ++e) x[e] = 0.f;
      }
#pragma unroll
      for (int e = 0; e < 8; ++e) x[e] += fmaf(sc, v[e], bf[c + e]);
      st16(o, pack(x, __nv_bfloat16()));
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, D);
}

// No more CTAs on an SM than its 512 tensor-memory columns hold.
inline size_t gemm_smem(size_t need, int tcols) {
  const size_t ctas = 512 / tcols;
  return std::max(need, (size_t)(233472 / (ctas + 1) - 1024 + 16));
}

template <int D>
hg_status rows_gemm_t(const void* A, int64_t n, const void* B, const void* bias, void* out, int64_t ldo, int ocol0,
                      int accumulate, const float* scale_ptr, float scale_mul, cudaStream_t s) {
  static bool done = false;
  if (!done) {
    HG_CUDA(cudaFuncSetAttribute(rows_gemm_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, 232448));
    done = true;
  }
  CUtensorMap tm_A, tm_B;
  HG_TRY(make_tmap_bf16(&tm_A, A, (uint64_t)n, D, kRows));
  HG_TRY(make_tmap_bf16(&tm_B, B, D, D, D));
  GArgs g{n, scale_ptr, scale_mul, (const __nv_bfloat16*)bias, (__nv_bfloat16*)out, ldo, ocol0, accumulate,
          device_status_ptr()};
  return launch("rows_gemm_tc", rows_gemm_tc_kernel<D>, dim3((unsigned)ceil_div(n, kRows)), dim3(kThreads),
                gemm_smem(GCfg<D>::kNeed, D), s, tm_A, tm_B, g);
}

}  // namespace

hg_status rows_gemm_tc(int d, const void* A, int64_t n, const void* B, const void* bias, void* out, int64_t ldo,
                       int ocol0, int accumulate, const float* scale_ptr, float scale_mul, cudaStream_t s) {
  if (n <= 0) return HG_OK;
  if (((uintptr_t)A & 15) || ((uintptr_t)B & 15) || ((uintptr_t)out & 15) || (ldo % 8) || (ocol0 % 8)) {
    set_error("rows_gemm_tc: operands must be 16-byte aligned");
    return HG_ERR_INVALID_ARG;
  }
  if (d == 64) return rows_gemm_t<64>(A, n, B, bias, out, ldo, ocol0, accumulate, scale_ptr, scale_mul, s);
  if (d == 128) return rows_gemm_t<128>(A, n, B, bias, out, ldo, ocol0, accumulate, scale_ptr, scale_mul, s);
  if (d == 256) return rows_gemm_t<256>(A, n, B, bias, out, ldo, ocol0, accumulate, scale_ptr, scale_mul, s);
  set_error("rows_gemm_tc: unsupported d=%d", d);
  return HG_ERR_UNSUPPORTED;
}

}  // namespace hg
