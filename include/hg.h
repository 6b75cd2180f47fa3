/*
 * hg.h -- C ABI of the GB300 hot path of risk-aware overlapping-subgraph GNN training.
 *
 * The library computes, on one GPU and on the caller's stream:
 *   - the relation-typed adjacency of one overlapping subgraph as CSR (by destination) and CSC
 *     (by source) per relation (Section 2.2: node types, relations, meta-relation triplets;
 *     Section 3.1, Eq. 5 and Algorithm 1: the induced overlapping subgraph);
 *   - the forward and backward pass of one heterogeneous message-passing layer (Eq. 7 with one
 *     message matrix W_r per relation, Eq. 10 with the mean over each relation's neighbours,
 *     per-relation means summed into the target, Eq. 11: per-type Linear_agg, activation,
 *     residual; optional LayerNorm per node type after the residual);
 *   - the overlap batch B between two subgraphs as pairs of local rows (Section 3.3);
 *   - the cross-subgraph CCA alignment loss on B (Eq. 14-17) and its gradient.
 *
 * Conventions for every entry point:
 *   - Pointers named *_dev, H_*, dH_*, idx_*, gid_*, workspace, saved, scratch, and the edge
 *     arrays are DEVICE pointers; everything else (type_offsets, rels, sizes) is HOST memory.
 *   - The library allocates no device memory.  All device buffers are owned by the caller; the
 *     *_size queries give the bytes each call needs.  Buffers must be 256-byte aligned.
 *   - Work is enqueued on `stream` (a cudaStream_t; NULL = legacy default stream).  No entry point
 *     synchronises except hg_graph_check and hg_timing_report, which say so.
 *   - Arguments are validated on the host before any launch.  A failed check returns a status
 *     (never traps or aborts) and leaves a message in hg_last_error().  Device-side input
 *     problems (an edge id out of range, unsorted global ids) never cause out-of-bounds
 *     accesses: the offending items are dropped or flagged as documented per call.
 *   - Node ids are local to the subgraph and contiguous per node type: type t owns ids
 *     [type_offsets[t], type_offsets[t+1]).  Features are row-major N x d.
 *   - Supported feature widths: d in {64, 128, 256}; dtypes HG_F32 and HG_BF16 (storage type of
 *     features, weights and activations; arithmetic accumulates in fp32).  Edge counts < 2^31.
 *   - One process drives one GPU through this library (one process per GPU, as in data-parallel
 *     training): kernel attributes (large shared-memory carve-outs) and the address of the device
 *     status word are set up once, and the library binds itself to the device current at its
 *     first kernel-launching call (or to the one named by hg_bind_device).  A later call made
 *     with another device current returns HG_ERR_UNSUPPORTED before launching anything.
 */
#ifndef HG_H_
#define HG_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef struct CUstream_st* hg_stream; /* identical to cudaStream_t */

typedef enum {
  HG_OK = 0,
  HG_ERR_INVALID_ARG = 1,  /* null pointer, bad size, mismatched shapes */
  HG_ERR_UNSUPPORTED = 2,  /* valid request outside what the kernels handle (d, dtype, > 2^31 edges) */
  HG_ERR_WORKSPACE = 3,    /* caller buffer smaller than the matching *_size query */
  HG_ERR_CUDA = 4,         /* a CUDA runtime call or launch failed */
  HG_ERR_DEVICE_CHECK = 5, /* a device-side input check failed (reported by hg_graph_check) */
  HG_ERR_TIMEOUT = 6       /* a bounded wait inside a kernel gave up (see hg_device_status) */
} hg_status;

typedef enum { HG_F32 = 0, HG_BF16 = 1 } hg_dtype;
typedef enum { HG_ACT_RELU = 0, HG_ACT_GELU_TANH = 1, HG_ACT_NONE = 2 } hg_act;

/* Relation r connects a source node of type src_type to a destination node of type dst_type
 * (the meta-relation triplet <tau(i), phi(e), tau(j)> of Section 2.2). */
typedef struct {
  int32_t src_type;
  int32_t dst_type;
} hg_rel_desc;

typedef struct hg_graph hg_graph; /* opaque host handle; its arrays live in the caller's workspace */

/* Static description of a status code. */
const char* hg_status_string(hg_status status);
/* Detail of the last failure on the calling thread ("" if none).  Valid until the next call. */
const char* hg_last_error(void);
/* Version of this ABI (bumped on any incompatible change). */
int32_t hg_abi_version(void);
/* Binds the library to device ordinal `device` (the CUDA runtime's numbering) before its first
 * kernel-launching call; without it the first such call binds the device current then.  HG_OK if
 * the library is unbound or already bound to `device`; HG_ERR_UNSUPPORTED if it is bound to
 * another device; HG_ERR_INVALID_ARG for a negative ordinal.  Makes no CUDA call. */
hg_status hg_bind_device(int32_t device);
/* Diagnostic of the bounded waits: launches one CTA whose thread waits `polls` times (1 <= polls
 * <= 2^20) on an mbarrier that nothing arrives at -- with no copy, store or MMA in flight -- and
 * records the give-up in the device status word exactly as a tensor-core kernel whose wait runs
 * out does, so a caller can check that hg_device_status reports it and that the context stays
 * usable.  The paper has no counterpart. */
hg_status hg_selftest_bounded_wait(uint32_t polls, hg_stream stream);
/* SYNCHRONISES the device, then reports and clears the library's device status word.  Every wait
 * inside a kernel of this library is bounded; a wait that gave up sets a flag here (its kernel's
 * results are then invalid) and this call returns HG_ERR_TIMEOUT.  flags may be NULL. */
hg_status hg_device_status(int32_t* flags);

/* ------------------------------------------------------------------------------------------- */
/* Graph layout (Section 2.2, Section 3.1 / Eq. 5: the adjacency of one overlapping subgraph)   */
/* ------------------------------------------------------------------------------------------- */

/* Bytes of device workspace hg_build_csr needs for this many edges and these types/relations. */
hg_status hg_graph_workspace_size(int64_t num_edges, const int64_t* type_offsets, int32_t num_types,
                                  const hg_rel_desc* rels, int32_t num_rels, size_t* bytes);

/* Builds, on the device, per relation r: CSR by destination (rows = destination nodes of type
 * rels[r].dst_type in local order; each row lists its in-edges by ascending (source id, input edge
 * id)) and CSC by source (rows = source nodes of type rels[r].src_type; out-edges by ascending
 * (destination id, edge id)), plus the per-CSC-edge coefficient 1/deg_r(destination) as an IEEE
 * fp32 quotient, the split tables the aggregation kernels use for high-degree rows, and the
 * aggregation lists of the mean layer, in which the parallel edges of a node pair (adjacent in
 * that order) are one entry with their multiplicity.
 *   src, dst, rel : device int32 arrays of num_edges entries (COO, any order).
 *   type_offsets  : host int64 [num_types + 1], type_offsets[0] = 0, non-decreasing.
 *   rels          : host [num_rels].
 *   workspace     : device buffer of at least hg_graph_workspace_size bytes, owned by the caller
 *                   and kept alive (and unmodified) for the lifetime of the graph.
 *   out           : receives a host handle; release it with hg_graph_destroy.
 * Edges with an id out of range, a relation out of range, or endpoint types that differ from their
 * relation are dropped (never dereferenced out of bounds); hg_graph_check reports how many.
 * The src/dst/rel arrays may be freed once the work on `stream` has completed. */
hg_status hg_build_csr(const int32_t* src, const int32_t* dst, const int32_t* rel, int64_t num_edges,
                       const int64_t* type_offsets, int32_t num_types, const hg_rel_desc* rels,
                       int32_t num_rels, void* workspace, size_t workspace_bytes, hg_stream stream,
                       hg_graph** out);

/* Releases the host handle (the workspace stays with the caller).  NULL is accepted. */
hg_status hg_graph_destroy(hg_graph* graph);

/* SYNCHRONISES the graph's build stream.  Writes the number of dropped (invalid) edges; returns
 * HG_ERR_DEVICE_CHECK if it is non-zero, HG_OK otherwise. */
hg_status hg_graph_check(const hg_graph* graph, int64_t* num_invalid_edges);

/* Read-only device views of one relation's layout (for tests and for callers that want the CSR).
 * row_ptr has n_dst + 1 entries and csc_ptr n_src + 1 entries; their values index the col/eid and
 * csc_col/csc_eid/csc_coef arrays directly (relations are stored one after another).
 * col holds source node ids, csc_col destination node ids, eid/csc_eid input edge ids. */
typedef struct {
  int64_t n_dst, n_src, num_edges;
  const int32_t* row_ptr;
  const int32_t* col;
  const int32_t* eid;
  const int32_t* csc_ptr;
  const int32_t* csc_col;
  const int32_t* csc_eid;
  const float* csc_coef;
} hg_graph_arrays;
hg_status hg_graph_view(const hg_graph* graph, int32_t rel, hg_graph_arrays* out);

/* The order in which the bf16 forward projection (hg_layer_fwd) visits the destination nodes of one
 * type, built by hg_build_csr.  The relation mask of a node has bit k set when the k-th relation
 * into the type (relations by ascending id) has an in-edge at the node (M_r of Eq. 10 non-zero).
 * perm[i] (n entries) is the local id of the node at position i: the type's nodes sorted stably by
 * their mask.  tile_mask[q] (tiles = ceil(n / tile_rows) entries) is the OR of the masks at positions
 * tile_rows q .. tile_rows q + tile_rows - 1: the relations whose products a tile computes.  Device
 * arrays inside the graph's workspace (read only; for tests).  HG_ERR_INVALID for a type out of
 * range. */
typedef struct {
  int64_t n, tiles;
  int32_t tile_rows;
  const int32_t* perm;
  const int32_t* tile_mask;
} hg_node_order;
hg_status hg_graph_node_order(const hg_graph* graph, int32_t type, hg_node_order* out);

/* ------------------------------------------------------------------------------------------- */
/* Layer (Eq. 7, Eq. 10 with mean aggregation, Eq. 11, optional LayerNorm)                      */
/* ------------------------------------------------------------------------------------------- */

/* Layer parameters, packed device arrays in `dtype`:
 *   W_rel    [num_rels  x d x d]  message matrix of relation r, row-major (d_in x d_out)
 *   W_agg    [num_types x d x d]  Linear_agg of the target type, row-major (d_in x d_out)
 *   b_agg    [num_types x d]
 *   ln_gamma [num_types x d], ln_beta [num_types x d]  (read only when layernorm != 0)
 * For destination node j of type t:
 *   Z[j]     = sum over relations r into t of M_r[j] W_rel[r],
 *   M_r[j]   = mean of H_in over j's in-neighbours under r (0 when j has none),
 *   U[j]     = Z[j] W_agg[t] + b_agg[t],
 *   Y[j]     = act(U[j]) + H_in[j],
 *   H_out[j] = layernorm ? (Y[j] - mean) / sqrt(var + ln_eps) * ln_gamma[t] + ln_beta[t] : Y[j]
 * (population variance over the d features of the row). */
typedef struct {
  int32_t d;
  hg_dtype dtype;
  hg_act act;
  int32_t layernorm;
  float ln_eps;
  const void* W_rel;
  const void* W_agg;
  const void* b_agg;
  const void* ln_gamma;
  const void* ln_beta;
  /* 1: the fused mean layer (bf16, d = 128; else HG_ERR_UNSUPPORTED).  The relation means of rows
   * with at most 32 runs of parallel edges are summed straight into the projection's operand tiles
   * and never stored; the backward sums them again for the weight gradient.  Only the means of
   * longer rows are kept in `saved`, which is then much smaller.  Results are bitwise those of
   * fused = 0. */
  int32_t fused;
} hg_layer_params;

/* Gradients, fp32 device arrays with the shapes of the parameters; OVERWRITTEN by hg_layer_bwd.
 * dln_gamma / dln_beta may be NULL when layernorm == 0. */
typedef struct {
  float* dW_rel;
  float* dW_agg;
  float* db_agg;
  float* dln_gamma;
  float* dln_beta;
} hg_layer_grads;

/* Bytes of the `saved` buffer (written by hg_layer_fwd, read by hg_layer_bwd) and of the `scratch`
 * buffer (contents undefined between calls) one layer of this graph needs. */
hg_status hg_layer_workspace_size(const hg_graph* graph, const hg_layer_params* params,
                                  size_t* saved_bytes, size_t* scratch_bytes);

/* Forward pass.  H_in, H_out: N x d in params->dtype (N = type_offsets[num_types]); they must not
 * overlap.  saved: keeps what the backward pass needs (the per-relation means of the destination
 * rows that have in-edges, Z, U, row statistics). */
hg_status hg_layer_fwd(const hg_graph* graph, const hg_layer_params* params, const void* H_in,
                       void* H_out, void* saved, void* scratch, hg_stream stream);

/* Backward pass of the layer whose forward wrote `saved` from the same H_in and params.
 *   dH_out : N x d upstream gradient (dtype).
 *   dH_in  : N x d, OVERWRITTEN with dL/dH_in (residual path plus the transposed aggregation);
 *            NULL skips that part (then only the weight gradients are produced).
 *   grads  : weight gradients, OVERWRITTEN. */
hg_status hg_layer_bwd(const hg_graph* graph, const hg_layer_params* params, const void* H_in,
                       const void* saved, const void* dH_out, void* dH_in, const hg_layer_grads* grads,
                       void* scratch, hg_stream stream);

/* ------------------------------------------------------------------------------------------- */
/* Overlap batch (Section 3.3) and CCA alignment (Eq. 14-17)                                     */
/* ------------------------------------------------------------------------------------------- */

hg_status hg_overlap_intersect_workspace_size(int64_t n_a, int64_t n_b, size_t* bytes);

/* B = the nodes present in both subgraphs.  gid_a [n_a], gid_b [n_b]: device int64 global ids of
 * each subgraph's local rows, STRICTLY ASCENDING (local ids follow global-id order).  Writes, for
 * k < *n_out, idx_a[k] / idx_b[k] = local rows of the k-th common node in ascending global id;
 * idx_a and idx_b need min(n_a, n_b) entries.  n_out: device int64 scalar; it is set to -1 if
 * either list is not strictly ascending (then idx_* are unspecified). */
hg_status hg_overlap_intersect(const int64_t* gid_a, int64_t n_a, const int64_t* gid_b, int64_t n_b,
                               int32_t* idx_a, int32_t* idx_b, int64_t* n_out, void* scratch,
                               size_t scratch_bytes, hg_stream stream);

/* Buffer sizes for the alignment calls with at most n_max overlap rows of width d. */
hg_status hg_overlap_align_workspace_size(int64_t n_max, int32_t d, size_t* saved_bytes,
                                          size_t* scratch_bytes);

/* Alignment loss between rows H_a[idx_a[k]] and H_b[idx_b[k]], k < n (H_a has rows_a rows,
 * H_b rows_b rows):
 *   Z = (X - mean) / (sqrt(var + var_eps) * sqrt(n)) per column (population variance, Eq. 14),
 *   loss_out[1] = L_inv = ||Z_a - Z_b||_F^2                                         (Eq. 15)
 *   loss_out[2] = L_dec = ||Z_a^T Z_a - I||_F^2 + ||Z_b^T Z_b - I||_F^2              (Eq. 16)
 *   loss_out[0] = L_inv + lambda_n * L_dec                                           (Eq. 17)
 * H_a, H_b: row-major, d columns, dtype.  idx_a, idx_b: device int32 [n_max]; each list must
 * hold distinct rows.  An index outside [0, rows) is never dereferenced: it is clamped, the loss
 * becomes NaN and hg_overlap_align_bwd then writes no gradient.  n_dev: optional device int64 with the actual n (<= n_max), e.g. the n_out
 * of hg_overlap_intersect, so no host round trip is needed; NULL means n = n_max.  n < 2 gives a
 * zero loss.  loss_out: device fp32 [3].  saved: kept for hg_overlap_align_bwd. */
hg_status hg_overlap_align_loss(const void* H_a, int64_t rows_a, const int32_t* idx_a, const void* H_b,
                                int64_t rows_b, const int32_t* idx_b, int64_t n_max, const int64_t* n_dev,
                                int32_t d, hg_dtype dtype, float lambda_n, float var_eps, float* loss_out,
                                void* saved, void* scratch, hg_stream stream);

/* Gradient of dloss * L (dloss = lambda_CCA of Eq. 20 in training) with respect to the overlap
 * rows, ACCUMULATED into dH_a[idx_a[k]] and dH_b[idx_b[k]] (dtype, same layout as H_a / H_b).
 * dH_b may be NULL (a detached view, e.g. embeddings received from another subgraph); dH_a may be
 * NULL too.  `saved` must come from hg_overlap_align_loss on the same inputs. */
hg_status hg_overlap_align_bwd(const void* H_a, int64_t rows_a, const int32_t* idx_a, const void* H_b,
                               int64_t rows_b, const int32_t* idx_b, int64_t n_max, const int64_t* n_dev,
                               int32_t d, hg_dtype dtype, float lambda_n, float var_eps, float dloss,
                               const void* saved, void* dH_a, void* dH_b, void* scratch, hg_stream stream);

/* The same loss as hg_overlap_align_loss for callers that cannot allocate device memory -- a host
 * program that links only this C ABI and owns no CUDA allocator, a process whose device memory is
 * fully reserved by another framework's caching allocator, or code for which cudaMalloc is off
 * limits because it can synchronise the device.  The paper has no counterpart; this is an
 * interface convenience.  Inputs, `loss_out` and `saved` are as for hg_overlap_align_loss (the
 * `saved` buffer still comes from the caller and feeds hg_overlap_align_bwd); the scratch is a
 * 12 MiB device array inside the library, which every GPU that loads the library holds until the
 * process exits.  It calls no allocating routine.  The array's device address is looked up on
 * the first call made on each device (with that device current), so that first call should come
 * before any stream capture.  All calls share the array: calls that overlap on the GPU race.
 * Returns HG_ERR_UNSUPPORTED for a width whose scratch would exceed the array (none of the
 * supported d do). */
hg_status hg_overlap_align_loss_static(const void* H_a, int64_t rows_a, const int32_t* idx_a, const void* H_b,
                                       int64_t rows_b, const int32_t* idx_b, int64_t n_max, const int64_t* n_dev,
                                       int32_t d, hg_dtype dtype, float lambda_n, float var_eps, float* loss_out,
                                       void* saved, hg_stream stream);

/* ------------------------------------------------------------------------------------------- */
/* Overlapping subgraph construction (Section 3.1, Eq. 4-5; Algorithm 1, construction loop)      */
/* ------------------------------------------------------------------------------------------- */

/* Subgraph k of K built from a global graph with global node ids [0, num_nodes), contiguous per
 * node type:
 *   base V_k     = { v : splitmix64(part_seed ^ v) mod K == k }   (random hash partition), where
 *                  splitmix64(x) is the SplitMix64 output for state x (x + 0x9E3779B97F4A7C15,
 *                  then the generator's two xor-shift-multiply steps and final xor-shift);
 *   degree(v)    = incident edges over all relations, both directions (a self-loop twice);
 *   h-index(v)   = the largest h with at least h incident edges leading to nodes of degree >= h;
 *   C_k          = nodes outside V_k with an edge v -> u, u in V_k                        (Eq. 4);
 *   C'_k         = the v in C_k with h-index(v) <= theta;
 *   C_{k,M}      = the M members of C'_k with the smallest key (high 32 bits of
 *                  splitmix64(sample_seed ^ (k << 40) ^ v)), ties by id; all of C'_k when fewer;
 *   V~_k         = V_k united with C_{k,M}                                                (Eq. 5);
 *   the induced subgraph: the edges with both endpoints in V~_k, in input order.
 * Local ids follow ascending global id (so node types stay contiguous).  Edges with an endpoint
 * outside [0, num_nodes) are ignored (neither incident nor induced).
 * Inputs (device): src, dst, rel [num_edges].  type_offsets (HOST, num_types + 1) are the global
 * type boundaries.  Outputs (device, capacities num_nodes / num_edges, entries past the counts
 * untouched): gid_out (int64, ascending global ids of V~_k), src_out / dst_out (local ids),
 * rel_out, eid_out (input edge ids), type_offsets_out (int64 [num_types + 1], local type
 * boundaries), h_out (int32 [num_nodes] h-index of every global node; may be NULL), counts_out
 * (int64 [6]: nodes, base nodes, expansion nodes, edges, |C_k|, |C'_k|).  K >= 1, 0 <= k < K,
 * theta >= 0, M >= 0, num_nodes < 2^31, num_edges < 2^31; otherwise HG_ERR_INVALID_ARG or
 * HG_ERR_UNSUPPORTED.  Integer work: the results are exact and reproducible. */
hg_status hg_overlap_build_workspace_size(int64_t num_nodes, int64_t num_edges, size_t* bytes);
hg_status hg_overlap_build(const int32_t* src, const int32_t* dst, const int32_t* rel, int64_t num_edges,
                           int64_t num_nodes, const int64_t* type_offsets, int32_t num_types, int32_t K,
                           int32_t k, int32_t theta, int64_t M, uint64_t part_seed, uint64_t sample_seed,
                           int64_t* gid_out, int32_t* src_out, int32_t* dst_out, int32_t* rel_out,
                           int32_t* eid_out, int64_t* type_offsets_out, int32_t* h_out, int64_t* counts_out,
                           void* workspace, size_t workspace_bytes, hg_stream stream);

/* ------------------------------------------------------------------------------------------- */
/* Attention layer (Heterogeneous Graph Transformer, Section 3.2, Eq. 6-11)                       */
/* ------------------------------------------------------------------------------------------- */

/* Parameters of one attention layer, device pointers of the storage type unless noted; T node
 * types, R relations, S heads of width d_h = d / S (S a power of two, 1 <= S <= 32):
 *   W_K, W_Q, W_V  [T][d][d] (input x output), b_K, b_Q, b_V [T][d]   key / query / value maps
 *   W_att, W_msg   [R][S][d_h][d_h]                                   per relation and head
 *   mu             [R] fp32 (device)                                  prior of each relation
 *   W_agg [T][d][d], b_agg [T][d], ln_gamma / ln_beta [T][d]           as in hg_layer_params */
typedef struct {
  int32_t d;
  int32_t heads;
  hg_dtype dtype;
  hg_act act;
  int32_t layernorm;
  float ln_eps;
  const void* W_K;
  const void* W_Q;
  const void* W_V;
  const void* b_K;
  const void* b_Q;
  const void* b_V;
  const void* W_att;
  const void* W_msg;
  const float* mu;
  const void* W_agg;
  const void* b_agg;
  const void* ln_gamma;
  const void* ln_beta;
} hg_hgt_params;

/* Gradients, device fp32, shapes as the parameters, OVERWRITTEN (dln_* may be NULL without
 * LayerNorm). */
typedef struct {
  float* dW_K;
  float* dW_Q;
  float* dW_V;
  float* db_K;
  float* db_Q;
  float* db_V;
  float* dW_att;
  float* dW_msg;
  float* dmu;
  float* dW_agg;
  float* db_agg;
  float* dln_gamma;
  float* dln_beta;
} hg_hgt_grads;

hg_status hg_hgt_workspace_size(const hg_graph* graph, const hg_hgt_params* params, size_t* saved_bytes,
                                size_t* scratch_bytes);

/* One attention layer on the graph (node features H_in, N x d, storage type):
 *   K, Q, V = H W_K + b_K, ... per node type;
 *   Eq. 6    score^s(e) = (K^s(i) W_att[r, s] . Q^s(j)) mu[r] / sqrt(d_h) for an edge e = i -> j of r;
 *   Eq. 8    alpha^s(e) = softmax over every in-edge of j (all relations);
 *   Eq. 7, 9, 10  h~_j = concat_s sum_e alpha^s(e) V^s(i) W_msg[r, s];
 *   Eq. 11   H_out = act(h~ W_agg + b_agg) + H_in, then LayerNorm per type when enabled.
 * H_out must not alias H_in.  `saved` feeds hg_hgt_bwd. */
hg_status hg_hgt_fwd(const hg_graph* graph, const hg_hgt_params* params, const void* H_in, void* H_out, void* saved,
                     void* scratch, hg_stream stream);

/* Backward: dH_in (N x d, OVERWRITTEN; NULL = skip) = dL/dH_in for the upstream gradient dH_out,
 * and every parameter gradient. */
hg_status hg_hgt_bwd(const hg_graph* graph, const hg_hgt_params* params, const void* H_in, const void* saved,
                     const void* dH_out, void* dH_in, const hg_hgt_grads* grads, void* scratch, hg_stream stream);

/* ------------------------------------------------------------------------------------------- */
/* Prediction head and joint objective (Section 3.4, Eq. 18-20; MeanAgg / MLP / loss steps of     */
/* Algorithm 1)                                                                                   */
/* ------------------------------------------------------------------------------------------- */

/* Two-layer head on final embeddings of width d (hidden width d, one output logit), device
 * pointers of the storage type: W1 d x d row-major (input x hidden, applied as h W1), b1 [d],
 * w2 [d], b2 [1].  W1, b1 and w2 must be 16-byte aligned. */
typedef struct {
  int32_t d;
  hg_dtype dtype;
  const void* W1;
  const void* b1;
  const void* w2;
  const void* b2;
} hg_head_params;

/* Head gradients, device fp32, OVERWRITTEN: dW1 [d x d], db1 [d], dw2 [d], db2 [1]. */
typedef struct {
  float* dW1;
  float* db1;
  float* dw2;
  float* db2;
} hg_head_grads;

/* Buffer sizes for n_lab labelled rows of an H with `rows` rows. */
hg_status hg_head_workspace_size(int64_t rows, int64_t n_lab, int32_t d, hg_dtype dtype, size_t* saved_bytes,
                                 size_t* scratch_bytes);

/* Masked BCE of the head over the labelled rows and the joint objective:
 *   MeanAgg  h_r = H[lab_idx[r]], or, when that row is idx_a[k] of an overlap pair k < n_rep,
 *            (H[idx_a[k]] + H_rep[idx_b[k]]) / 2 (the mean of the node's two replicas; the
 *            pre-activation below is formed from the two stored rows in fp32, the rows kept for
 *            the weight gradient are the mean rounded to the storage type);
 *   Eq. 18   z_r = relu(h_r W1 + b1) . w2 + b2 (a logit; the probability is sigmoid(z_r));
 *   Eq. 19   loss_out[1] = L_BCE = (1/n_lab) sum_r -[y_r log p_r + (1 - y_r) log(1 - p_r)];
 *   Eq. 20   loss_out[0] = L_BCE + lambda_cca * cca_loss[0]  (cca_loss: device fp32, e.g. the
 *            loss_out of hg_overlap_align_loss; NULL means L_BCE alone).
 * H: rows x d, H_rep: rows_rep x d (row-major, storage type, 16-byte aligned).  idx_a / idx_b:
 * device int32 [n_rep_max] overlap pairs (hg_overlap_intersect), each list of distinct rows;
 * n_rep_dev: optional device int64 with the actual count (NULL = n_rep_max; a negative count
 * means none); pairs with an index out of range are ignored.  lab_idx: device int32 [n_lab]
 * DISTINCT rows of H; lab_y: device fp32 [n_lab] labels in [0, 1].  A lab_idx entry outside
 * [0, rows) is never dereferenced: it makes the loss NaN and gets no gradient.  logits: device
 * fp32 [n_lab] (z_r) or NULL.  loss_out: device fp32 [2].  saved: kept for hg_head_bwd.
 * n_lab = 0 gives L_BCE = 0. */
hg_status hg_head_loss(const hg_head_params* params, const void* H, int64_t rows, const void* H_rep,
                       int64_t rows_rep, const int32_t* idx_a, const int32_t* idx_b, int64_t n_rep_max,
                       const int64_t* n_rep_dev, const int32_t* lab_idx, const float* lab_y, int64_t n_lab,
                       const float* cca_loss, float lambda_cca, float* loss_out, float* logits, void* saved,
                       void* scratch, hg_stream stream);

/* Gradient of dloss * L_BCE (dloss = 1 in training; the alignment term's gradient comes from
 * hg_overlap_align_bwd with dloss = lambda_CCA).  grads are OVERWRITTEN.  The gradient at each
 * labelled row's final embedding is added to dH[lab_idx[r]] (storage type), or, for a row with a
 * replica, half to dH[idx_a[k]] and half to dH_rep[idx_b[k]].  dH (rows x d) and dH_rep
 * (rows_rep x d) are ACCUMULATED into, or, when overwrite is nonzero, first set to zero (so they
 * end up holding the head's gradient alone, e.g. the last layer's upstream gradient before the
 * alignment term is added).  dH_rep may be NULL (a detached second view); dH may be NULL.  `saved`
 * must come from hg_head_loss with the same params, lab_idx and n_lab. */
hg_status hg_head_bwd(const hg_head_params* params, const int32_t* lab_idx, int64_t n_lab, float dloss,
                      const void* saved, void* dH, int64_t rows, void* dH_rep, int64_t rows_rep, int32_t overwrite,
                      const hg_head_grads* grads, void* scratch, hg_stream stream);

/* ------------------------------------------------------------------------------------------- */
/* Temporal module (Section 3.2, Eq. 12-13): attention over each node's last w states and a GRU  */
/* ------------------------------------------------------------------------------------------- */

/* Parameters, device pointers of the storage type: Wa = Q^T (d x d, input x output), r [d],
 * W_i = [W_ir | W_iz | W_in] and W_h = [W_hr | W_hz | W_hn] (d x 3d each, input x output), b_i and
 * b_h [3d].  1 <= w <= 8. */
typedef struct {
  int32_t d;
  int32_t w;
  hg_dtype dtype;
  const void* Wa;
  const void* r;
  const void* W_i;
  const void* W_h;
  const void* b_i;
  const void* b_h;
} hg_temporal_params;

/* Gradients, device fp32, OVERWRITTEN: dWa [d x d], dr [d], dW_i and dW_h [d x 3d], db_i, db_h [3d]. */
typedef struct {
  float* dWa;
  float* dr;
  float* dW_i;
  float* dW_h;
  float* db_i;
  float* db_h;
} hg_temporal_grads;

hg_status hg_temporal_workspace_size(int64_t n, int32_t d, int32_t w, hg_dtype dtype, size_t* saved_bytes,
                                     size_t* scratch_bytes);

/* H_out = H^t for n nodes:
 *   Eq. 12  u_k = tanh(c_k Wa), e_k = r . u_k, a = softmax over k < w of e, H~ = sum_k a_k c_k
 *           (rounded to the storage type);
 *   Eq. 13  r_g = sigmoid(x W_ir + b_ir + H~ W_hr + b_hr), z = sigmoid(x W_iz + b_iz + H~ W_hz + b_hz),
 *           n_g = tanh(x W_in + b_in + r_g * (H~ W_hn + b_hn)), H^t = (1 - z) n_g + z H~.
 * X: n x d, the spatial embeddings h^t (the last layer's output).  C: w x n x d, block k holding
 * every node's state k + 1 snapshots back (c_{k+1}); zero rows where a state does not exist.
 * H_out: n x d.  All row-major, storage type.  saved: H~ and a, kept for hg_temporal_bwd. */
hg_status hg_temporal_fwd(const hg_temporal_params* params, const void* X, const void* C, int64_t n, void* H_out,
                          void* saved, void* scratch, hg_stream stream);

/* Backward of hg_temporal_fwd for the upstream gradient dH_out (n x d): dX (n x d, OVERWRITTEN) =
 * dL/dX and every parameter gradient.  The context C receives no gradient (it holds earlier
 * snapshots' outputs).  X, C, params and `saved` must be those of the forward. */
hg_status hg_temporal_bwd(const hg_temporal_params* params, const void* X, const void* C, int64_t n,
                          const void* saved, const void* dH_out, void* dX, const hg_temporal_grads* grads,
                          void* scratch, hg_stream stream);

/* ------------------------------------------------------------------------------------------- */
/* Kernel timing (measurement support; off by default)                                          */
/* ------------------------------------------------------------------------------------------- */

/* When on, every kernel launch of this library is bracketed by CUDA events on its stream. */
hg_status hg_timing_enable(int32_t on);
/* SYNCHRONISES on the recorded events, then writes one line per kernel name,
 * "name launches total_ms\n", into buf (truncated to len) and clears the record. */
hg_status hg_timing_report(char* buf, size_t len);

#ifdef __cplusplus
}
#endif
#endif /* HG_H_ */
