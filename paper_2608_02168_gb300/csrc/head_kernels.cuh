// Argument blocks and internal entry points of the prediction-head kernels (shared by the CUDA-core
// and tensor-core translation units; not part of the public ABI).
#pragma once

#include "hg_internal.cuh"

namespace hg {

struct HeadFwdArgs {
  const void* H;
  int64_t rows;
  const void* H_rep;
  const int32_t* map;  // [rows] replica row in H_rep or -1
  const int32_t* lab;
  const float* y;
  int64_t n;
  float inv_n;
  const void* W1;
  const void* b1;
  const void* w2;
  const void* b2;
  void* Hm;             // saved [n][D]: MeanAgg rows
  void* dA;             // saved [n][D]: unit gradient of the hidden pre-activation
  int32_t* rep_row;     // saved [n]: replica row of each labelled row, -1 none, -2 invalid row
  float* logits;        // [n] or null
  float* part;          // [blocks][2 + 2D]: loss, dz, dA column sums, dz * relu(a) column sums
  int* status;          // library status word (timeouts of bounded waits)
};

struct HeadBwdArgs {
  const void* dA;
  const int32_t* lab;
  const int32_t* rep_row;
  int64_t n, rows;
  const void* W1;   // D x D (tensor-core kernel)
  const void* W1t;  // W1^T (CUDA-core kernel)
  float dloss;
  void* dH;
  void* dH_rep;
  int* status;
};

// Rows per block of the tensor-core head kernels.
constexpr int kHeadTcRows = 128;

// bf16 storage, d in {64, 128, 256}: the forward tile kernel (gather, h W1 on the tensor cores, the
// logit, loss and unit gradients, block partials over kHeadTcRows rows) and the input-gradient
// kernel (dA W1^T on the tensor cores, added to the rows of dH / dH_rep).
hg_status head_fwd_tc(int d, const HeadFwdArgs& a, cudaStream_t s);
hg_status head_dx_tc(int d, const HeadBwdArgs& a, cudaStream_t s);

}  // namespace hg
