// Argument blocks and internal entry points of the layer kernels (shared by the translation
// units; not part of the public ABI).
#pragma once

#include <cuda_bf16.h>

#include "hg_internal.cuh"

namespace hg {

struct FwdArgs {
  const void* M;                 // saved relation means, concatenated CSR rows (or compact rows)
  const int32_t* mrow;           // compact index of each CSR row (>= msent: empty); null: M by CSR row
  int64_t msent;
  int nrel;
  int64_t mrow0[kMaxRels];       // first CSR row of each relation into this type
  const void* W_rel[kMaxRels];   // its D x D message matrix (d_in x d_out)
  const void* W_agg;
  const void* b;
  const void* gamma;
  const void* beta;
  const void* H_in;
  void* H_out;
  void* Z;                       // saved, node rows
  void* U;                       // saved, node rows
  float2* stats;                 // saved (mean, rstd) per node row
  int64_t off, n;                // node rows [off, off + n) of this type
  int act, ln;
  float eps;
};

struct BwdArgs {
  const void* dH_out;
  const void* H_in;
  const void* U;
  const float2* stats;
  const void* gamma;
  const void* W_aggT;            // W_agg^T, D x D row-major
  int nrel;
  int64_t mrow0[kMaxRels];
  const void* W_relT[kMaxRels];  // W_r^T
  const int32_t* csr_ptr;        // degrees of the relation rows (null: no 1/deg scaling)
  void* dY;                      // node rows
  void* dU;                      // node rows
  void* dZ;                      // node rows
  void* dMs;                     // concatenated CSR rows (scaled by 1/deg), or compact rows
  const int32_t* mrow;           // compact index of each CSR row (>= msent: empty, not stored); null: CSR rows
  int64_t msent;
  float* part;                   // [blocks][3][D]: db, dgamma, dbeta partials
  int64_t off, n;
  int act, ln;
};

// tensor-core kernels (bf16 storage)
struct TcFwdArgs {
  int nrel;
  int rel[kMaxRels];          // relation ids into this type (row block of W_rel^T)
  int64_t mrow0[kMaxRels];    // first CSR row of each
  const int32_t* mrow;        // row of M holding each CSR row (>= msent: an empty row, read as zeros);
  int64_t msent;              // null: M is indexed by CSR row.  msent = the row extent of M
  const __nv_bfloat16* M;     // relation means, [msent][D]
  const int32_t* perm;        // tile position -> local node (the type's nodes by relation mask); null: identity
  const int32_t* tmask;       // per tile, the relations (bit k = rel[k]) with a stored row in it; null: all
  // the fused mean layer (M unused): the means are summed from H_in over the CSR runs in the
  // projection; rows above kFuseRuns runs read theirs from Mlong at slot long_ofs[row]
  const int32_t* agg_ptr;
  const int32_t* agg_col;
  const int32_t* agg_cnt;
  const int32_t* csr_ptr;     // deg = the CSR row length
  const int32_t* long_ofs;
  const __nv_bfloat16* Mlong;
  int type;
  const __nv_bfloat16* b;
  const __nv_bfloat16* gamma;
  const __nv_bfloat16* beta;
  const __nv_bfloat16* H_in;
  __nv_bfloat16* H_out;
  __nv_bfloat16* U;
  float2* stats;
  int64_t off, n;
  int act, ln;
  float eps;
  int* status;  // library status word (timeouts of bounded waits)
};

struct TcBwdArgs {
  int nrel;
  int rel[kMaxRels];
  int64_t mrow0[kMaxRels];
  const int32_t* mlist;       // CSR row of each compact row; mbase[r] .. mbase[r + 1] = relation r's
  const int32_t* mbase;       // compact rows (device).  null: every CSR row, dMs indexed by CSR row
  int type;
  const __nv_bfloat16* dH_out;
  const __nv_bfloat16* H_in;
  const __nv_bfloat16* U;     // the stored pre-activation without its bias (bf16(Z W_agg))
  const float2* stats;
  const __nv_bfloat16* gamma;
  const __nv_bfloat16* b;     // the type's bias b_agg, added back to U in fp32
  const int32_t* csr_ptr;
  __nv_bfloat16* dY;
  __nv_bfloat16* dU;
  __nv_bfloat16* dMs;
  float* part;  // [gridDim.x][3][D]
  int64_t off, n;
  int act, ln;
  int* status;
};

// destination type of each relation, passed by value to kernels
struct RelDst {
  int v[kMaxRels];
};
hg_status tc_fuse_weights(int d, const void* W_rel, const void* W_agg, RelDst rd, int num_rels, void* V, void* Vt,
                          cudaStream_t s);
hg_status tc_proj_forward(int d, const TcFwdArgs& a, const void* M, int64_t m_rows, const void* Vt, int num_rels,
                          cudaStream_t s);
// The fused mean layer's projection (d = 128): the relation means are summed into the operand tiles
// from a.H_in (a.agg_ptr .. a.Mlong set; a.M unused).
hg_status tc_proj_forward_gather(int d, const TcFwdArgs& a, const void* Vt, int num_rels, cudaStream_t s);
hg_status tc_ln_act_backward(int d, const TcBwdArgs& a, int* blocks, cudaStream_t s);
hg_status tc_proj_backward(int d, const TcBwdArgs& a, const void* V, int num_rels, cudaStream_t s);
// outs[r] = X[x0[r] .. x0[r]+n)^T Y[y0 .. y0+n) for r < R (R <= wgrad_tc_max_rels(d)); the R
// products share the loads of Y.  part: R x wgrad_tc_splits(n, d) x d x d floats.
// out = G_r = M^T dU over relation `rel`'s stored rows: compact rows mbase[rel] .. mbase[rel + 1]
// of M (m_rows rows in all) paired with dU rows mlist[k] - row0 (of the type's n rows at y0).
hg_status tc_weight_grad_rows(int d, const void* M, int64_t m_rows, const int32_t* mlist, const int32_t* mbase, int rel,
                              int64_t row0, const void* dU, int64_t y0, int64_t n, float* part, float* out, float* tmp,
                              cudaStream_t s);
// The same with M_r's rows summed from H over the CSR runs (rows above kFuseRuns runs read from Mlong
// at their long slot): the fused mean layer's backward (d = 128).
hg_status tc_weight_grad_gather(int d, const hg_graph* g, const void* H, const void* Mlong, int rel, int64_t row0,
                                const void* dU, int64_t y0, int64_t n, float* part, float* out, float* tmp,
                                cudaStream_t s);
hg_status tc_weight_grad(int d, const void* X, const int64_t* x0, int R, const void* Y, int64_t y0, int64_t n,
                         float* part, float* const* outs, float* tmp, cudaStream_t s);
int wgrad_tc_max_rels(int d);
hg_status tc_wgrad_finish(int d, const float* G, const void* W_rel, const void* W_agg, RelDst rd, int num_rels,
                          int num_types, float* dW_rel, float* dW_agg, cudaStream_t s);
int wgrad_tc_splits(int64_t n, int d);
int* device_status_ptr();  // device address of the library status word

hg_status aggregate_forward(const hg_graph* g, hg_dtype dt, int d, const void* H, void* M, float* partials,
                            int32_t* work,
                            cudaStream_t s);
// The fused mean layer's long rows (more than kFuseRuns runs, bf16): Mlong[k] = the mean of CSR row
// long_list[k], the same sum as aggregate_forward's.
hg_status aggregate_forward_long(const hg_graph* g, int d, const void* H, void* Mlong, float* partials, int32_t* work,
                                 cudaStream_t s);
hg_status aggregate_backward(const hg_graph* g, hg_dtype dt, int d, const void* dMs, const void* dY, void* dH,
                             float* partials, int32_t* work, cudaStream_t s);
hg_status proj_forward(hg_dtype dt, int d, const FwdArgs& a, cudaStream_t s);
hg_status proj_backward(hg_dtype dt, int d, const BwdArgs& a, cudaStream_t s);
// out = X^T Y over rows [x0, x0 + n) of X and [y0, y0 + n) of Y; with xmap, X row x0 + k is
// X[xmap[x0 + k]] and a mapped row >= xsent is zero (X stored for non-empty rows only).
hg_status weight_grad(hg_dtype dt, int d, const void* X, int64_t x0, const void* Y, int64_t y0, int64_t n, float* part,
                      float* out, float* tmp, cudaStream_t s, const int32_t* xmap = nullptr, int64_t xsent = 0);
hg_status transpose_weights(hg_dtype dt, int d, const void* W, void* Wt, int count, cudaStream_t s);
// fixed-order sum of `splits` partial arrays (tmp: reduce_tmp_floats(splits, count) floats)
hg_status reduce_partials(const float* part, int64_t stride, int splits, int64_t count, float* out, float* tmp,
                          cudaStream_t s);
size_t reduce_tmp_floats(int splits, int64_t count);
// The same over the first 1 to 3 segments of `seg` entries of each partial (entry k * seg + i of a
// partial adds into out_k[i]); out1 / out2 NULL = fewer segments.
hg_status reduce_partials3(const float* part, int64_t stride, int splits, int64_t seg, float* out0, float* out1,
                           float* out2, cudaStream_t s);
int wgrad_splits(int64_t n);
// Tensor-core row product (bf16): out[r][ocol0 + c] (=, or += when accumulate) scale A[r] B + bias,
// A: n x d rows (row stride d), B: d x d row-major, bias: d or null; out row stride ldo; scale =
// scale_mul * (*scale_ptr), scale_ptr a device fp32 scalar or null (1).
hg_status rows_gemm_tc(int d, const void* A, int64_t n, const void* B, const void* bias, void* out, int64_t ldo,
                       int ocol0, int accumulate, const float* scale_ptr, float scale_mul, cudaStream_t s);

// Buffers of one layer (saved for the backward, and scratch).
struct LayerLayout {
  void* M;        // saved: csr_rows x d relation rows (means, or attention-weighted sums)
  void* Mlong;    // saved (fused mean layer): long_cap x d means of the rows above kFuseRuns runs
  void* Z;        // saved (fp32 storage only): N x d
  void* U;        // saved: N x d pre-activation
  float2* stats;  // saved: N row statistics
  void* V;        // saved (bf16 only): R x 2 x d x d fused weights W_r W_agg (hi, lo halves)
  void* Vt;       // saved (bf16 only): their transposes (same order)
  float* agg_part;  // scratch: chunk partials
  int32_t* work;    // scratch: work counter of the forward row kernel (zeroed before each launch)
  void* dY;       // scratch: N x d
  void* dU;
  void* dZ;       // scratch (fp32 storage only)
  void* dMs;      // scratch: csr_rows x d
  float* cpart;   // scratch: column partials (blocks x 3 x d)
  float* wpart;   // scratch: splits x d x d
  float* rtmp;    // scratch: levels of the fixed-order reductions
  float* G;       // scratch (bf16 only): R x d x d products M_r^T dU
  void* WrelT;    // scratch (fp32 storage only): R x d x d
  void* WaggT;    // scratch (fp32 storage only): T x d x d
};
// fused: the mean layer without stored relation means (L->M null; L->Mlong holds the long rows')
void carve_layer(const hg_graph* g, int d, hg_dtype dt, void* saved, void* scratch, LayerLayout* L,
                 size_t* saved_bytes, size_t* scratch_bytes, bool fused = false);
RelDst rel_dst_of(const GraphMeta& m);
// Eq. 7 and Eq. 11 from the relation rows in L.M (bias, activation, residual, optional LayerNorm).
// compact: L.M holds the non-empty CSR rows only, in the graph's compact order (the mean layer);
// otherwise one row per CSR row (the attention layer's weighted sums).
hg_status project_forward(const hg_graph* graph, const hg_layer_params* p, const void* H_in, void* H_out,
                          const LayerLayout& L, bool compact, cudaStream_t s);
// Its backward: L.dY (residual path), L.dMs (dL/dM_r, divided by deg_r when deg_scale; compact rows
// when compact), the weight gradients into grads.
hg_status project_backward(const hg_graph* graph, const hg_layer_params* p, const void* H_in, const void* dH_out,
                           const hg_layer_grads* grads, const LayerLayout& L, bool deg_scale, bool compact,
                           cudaStream_t s);

}  // namespace hg
