// Shared pieces of the overlap-alignment translation units (Section 3.3, Eq. 14-17): row
// clamping, the device overlap count, the layout of the statistics kept between the loss and its
// gradient, and the tensor-core kernels of the bf16 path.
#pragma once

#include "hg_internal.cuh"

namespace hg {

// Row r of an overlap list, clamped into [0, rows) so that a bad index can never address memory
// outside the embedding table; bad indices are reported through the flag in `saved` instead.
__device__ __forceinline__ int64_t safe_row(const int32_t* __restrict__ idx, int64_t r, int64_t rows) {
  const int64_t x = idx[r];
  return x < 0 ? 0 : (x >= rows ? rows - 1 : x);
}

// Number of overlap rows in use: the device count clamped into [0, n_max], else n_max.
__device__ __forceinline__ int64_t count_of(const int64_t* n_dev, int64_t n_max) {
  if (!n_dev) return n_max;
  const int64_t n = *n_dev;
  return n < 0 ? 0 : (n > n_max ? n_max : n);
}

// Column sums over the overlap rows kept in `saved` (each d floats, in this order), with
// z = (x - mu) / (s sqrt(n)) per view (Eq. 14):
//   sum z_a, sum z_b, sum z_a z_b, sum (z_a - z_b)^2, sum z_a^2, sum z_b^2.
enum CrossSum { kSumZa = 0, kSumZb, kSumZaZb, kSumDiff2, kSumZa2, kSumZb2, kNumCross };

// bf16 Gram partials on the tensor cores: part[split][view][d][d] = sum over the split's rows of
// z z^T with z rounded to bf16 (fp32 accumulation); stats = [mu_a, mu_b, s_a, s_b].
int align_gram_tc_splits(int64_t n_max, int d, int max_splits);
hg_status align_gram_tc(int d, const void* Ha, int64_t rows_a, const int32_t* ia, const void* Hb, int64_t rows_b,
                        const int32_t* ib, int64_t n_max, const int64_t* n_dev, const float* stats, int splits,
                        float* part, cudaStream_t s);

// bf16 gradient: dH_v[idx_v[r]] += dX_v[r] for the views whose dH is non-null, with the product
// Z_v (C_v - I) on the tensor cores.  Scratch: cmi (2 d^2 bf16), means (4 d floats).
hg_status align_bwd_tc(int d, const void* Ha, int64_t rows_a, const int32_t* ia, const void* Hb, int64_t rows_b,
                       const int32_t* ib, int64_t n_max, const int64_t* n_dev, const float* stats, const float* C,
                       const float* cross, const int32_t* bad, float lambda_n, float dloss, void* cmi, float* means,
                       void* dHa, void* dHb, cudaStream_t s);

}  // namespace hg
