// Internal declarations of the temporal module (Section 3.2, Eq. 12-13); not part of the public ABI.
#pragma once

#include "hg_internal.cuh"

namespace hg {

// Largest context window the kernels accept.
constexpr int kTemporalMaxW = 8;

}  // namespace hg

namespace hg {

// Inputs of the tensor-core path (bf16, d in {64, 128}, (w + 1) d <= 512).
struct TemporalTcIn {
  const hg_temporal_params* p;
  const void* X;
  const void* C;
  int64_t n;
  void* Ht;  // saved H~ (written by the forward)
  float* a;  // saved attention weights [n][w]
};

struct TemporalTcScratch {
  void* dG;    // 4 x n x d bf16: dpre_r, dpre_z, dpre_n, dhn
  void* dh;    // n x d bf16: z dH^t
  void* dHt;   // n x d bf16: dL/dH~
  float* part; // temporal_tc_part_floats
  float* sums; // 4 d
  float* G;    // 3 d x d
  float* tmp;
};

bool temporal_tc_supported(hg_dtype dt, int d, int w);
size_t temporal_tc_part_floats(int64_t n, int d);
hg_status temporal_fwd_tc(const TemporalTcIn& in, void* H_out, cudaStream_t s);
hg_status temporal_bwd_tc(const TemporalTcIn& in, const void* dOut, void* dX, const hg_temporal_grads* g,
                          const TemporalTcScratch& sc, cudaStream_t s);

}  // namespace hg
