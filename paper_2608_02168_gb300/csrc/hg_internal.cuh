// Internal helpers shared by the translation units of libhg (never part of the public ABI).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <utility>

#include "hg.h"

namespace hg {

// ---------------------------------------------------------------------------------------------
// limits of this implementation
// ---------------------------------------------------------------------------------------------
constexpr int kMaxTypes = 4;
constexpr int kMaxRels = 8;
constexpr int kProjTileRows = 128;  // output rows per tile of the tensor-core forward projection
// A CSR/CSC row with more than kHubDegree edges is split into chunks of kChunkEdges edges; each
// chunk's fp32 partial sum goes to scratch and the row is finished by adding the chunk partials
// in chunk order, so the reduction order is fixed (deterministic, atomic-free).
constexpr int kHubDegree = 512;
constexpr int kChunkEdges = 512;
// The fused mean layer (gathers into the projection's operand tiles) sums a CSR row in the
// projection only up to kFuseRuns runs; the means of longer rows are computed beforehand by the
// streaming row kernel into a compact buffer, so no row holds the tile's loads for long.
constexpr int kFuseRuns = 32;

// ---------------------------------------------------------------------------------------------
// errors
// ---------------------------------------------------------------------------------------------
void set_error(const char* fmt, ...);
void clear_error();
// HG_OK when the current device is the one this process's library state is bound to (binding it
// at the first call); HG_ERR_UNSUPPORTED, before any launch, when another device is current.
hg_status device_guard();

#define HG_REQUIRE(cond, ...)              \
  do {                                     \
    if (!(cond)) {                         \
      ::hg::set_error(__VA_ARGS__);        \
      return HG_ERR_INVALID_ARG;           \
    }                                      \
  } while (0)

#define HG_TRY(expr)                       \
  do {                                     \
    hg_status st_ = (expr);                \
    if (st_ != HG_OK) return st_;          \
  } while (0)

#define HG_CUDA(call)                                                                 \
  do {                                                                                \
    cudaError_t e_ = (call);                                                          \
    if (e_ != cudaSuccess) {                                                          \
      ::hg::set_error("%s failed: %s", #call, cudaGetErrorString(e_));               \
      return HG_ERR_CUDA;                                                             \
    }                                                                                 \
  } while (0)

// ---------------------------------------------------------------------------------------------
// launches (optionally bracketed by CUDA events for per-kernel timing)
// ---------------------------------------------------------------------------------------------
int timing_begin(const char* name, cudaStream_t s);  // -1 when timing is off
void timing_end(int slot, cudaStream_t s);

template <typename... KArgs, typename... Args>
hg_status launch(const char* name, void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                 cudaStream_t s, Args&&... args) {
  if (grid.x == 0 || grid.y == 0 || grid.z == 0) return HG_OK;
  int slot = timing_begin(name, s);
  kernel<<<grid, block, smem, s>>>(std::forward<Args>(args)...);
  cudaError_t e = cudaGetLastError();
  timing_end(slot, s);
  if (e != cudaSuccess) {
    set_error("launch of %s failed: %s", name, cudaGetErrorString(e));
    return HG_ERR_CUDA;
  }
  return HG_OK;
}

inline int64_t ceil_div(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline size_t align_up(size_t x, size_t a = 256) { return (x + a - 1) / a * a; }

// Bump allocator over a caller buffer (computes offsets when base == nullptr).
struct Carve {
  char* base;
  size_t used = 0;
  explicit Carve(void* b) : base(static_cast<char*>(b)) {}
  template <typename T>
  T* take(size_t count) {
    size_t off = used;
    used = align_up(used + count * sizeof(T));
    return base ? reinterpret_cast<T*>(base + off) : nullptr;
  }
};

// ---------------------------------------------------------------------------------------------
// graph handle
// ---------------------------------------------------------------------------------------------
struct GraphMeta {
  int32_t num_types;
  int32_t num_rels;
  int64_t type_off[kMaxTypes + 1];
  int32_t rel_src[kMaxRels];
  int32_t rel_dst[kMaxRels];
  int64_t row_base[kMaxRels + 1];  // CSR rows of relation r: [row_base[r], row_base[r+1])
  int64_t csc_base[kMaxRels + 1];  // CSC rows of relation r: [csc_base[r], csc_base[r+1])
};

}  // namespace hg

struct hg_graph {
  hg::GraphMeta meta;
  int64_t num_edges;      // input COO entries (valid and invalid)
  int64_t csr_rows;       // meta.row_base[num_rels]
  int64_t csc_rows;       // meta.csc_base[num_rels]
  int64_t chunk_cap_csr;  // capacity of the chunk tables
  int64_t chunk_cap_node;
  cudaStream_t stream;    // build stream (hg_graph_check synchronises it)
  int32_t* csr_ptr;       // [csr_rows + 1]
  int32_t* csr_col;       // [num_edges] (valid prefix)
  int32_t* csr_eid;
  int32_t* csc_ptr;       // [csc_rows + 1]
  int32_t* csc_col;
  int32_t* csc_eid;
  float* csc_coef;
  int32_t* node_ptr;        // [N + 1] node-major out-edges over all relations (backward aggregation)
  int32_t* node_col;        // [num_edges] dMs row of each out-edge's destination
  // Parallel edges coalesced (the aggregation lists of the mean and attention layers): the CSR rows
  // as runs of equal source ids (agg_col = source, agg_cnt = multiplicity; deg = sum of the counts =
  // CSR row length) and the node-major rows as runs of equal dMs rows (bagg_col = the compact index
  // of the target's CSR row); per-row chunk tables over runs for rows above kHubDegree runs
  // (chunk_ofs: exclusive scan of chunks per row, chunk_row: the row of each chunk).
  int32_t* agg_ptr;         // [csr_rows + 1]
  int32_t* agg_col;         // [runs]
  int32_t* agg_cnt;
  int32_t* agg_chunk_ofs;   // [csr_rows + 1]
  int32_t* agg_chunk_row;   // [chunk_cap_csr]
  int32_t* bagg_ptr;        // [N + 1]
  int32_t* bagg_col;
  int32_t* bagg_cnt;
  int32_t* bagg_chunk_ofs;  // [N + 1]
  int32_t* bagg_chunk_row;  // [chunk_cap_node]
  // Non-empty CSR rows (the mean layer stores M_r and dMs_r only for them, in compact order):
  // mrow[row] = compact index, or csr_rows for an empty row (an out-of-range row, read as zeros by
  // the tensor-core loads); mlist[k] = CSR row of compact row k; mbase[r] = first compact row of
  // relation r (mbase[num_rels] = their number).  The backward runs (bagg_col) hold compact rows.
  int32_t* mrow;            // [csr_rows + 1]
  int32_t* mlist;           // [csr_rows + 1]
  int32_t* mbase;           // [kMaxRels + 1], device
  // Node order of the bf16 forward projection, per type t: the type's nodes sorted stably by their
  // relation mask (bit k = the k-th relation into t, by ascending id, has an in-edge at the node),
  // so that a 128-row tile rarely mixes masks.  nperm[type_off[t] + i] = local id of position i;
  // tmask[tile_base[t] + q] = OR of the masks of positions 128 q .. 128 q + 127.
  int32_t* nperm;           // [N]
  int32_t* tmask;           // [tile_base[num_types]]
  int64_t tile_base[hg::kMaxTypes + 1];
  // CSR rows with more than kFuseRuns runs (the fused layer's long rows): long_ofs = exclusive scan
  // of the flags (row is long iff long_ofs[row + 1] > long_ofs[row]; long_ofs[row] is its compact
  // slot, long_ofs[csr_rows] their number), long_list[k] = the CSR row of slot k.
  int32_t* long_ofs;        // [csr_rows + 1]
  int32_t* long_list;       // [long_cap]
  int64_t long_cap;         // E / (kFuseRuns + 1) + 1: at most that many rows are long
  int32_t* invalid_count;  // device scalar
};

namespace hg {

// ---------------------------------------------------------------------------------------------
// device helpers: 16-byte vectors of fp32 or bf16, converted to / from fp32 registers
// ---------------------------------------------------------------------------------------------
template <typename T>
struct VecTraits;
template <>
struct VecTraits<float> {
  static constexpr int kElems = 4;
};
template <>
struct VecTraits<__nv_bfloat16> {
  static constexpr int kElems = 8;
};

__device__ __forceinline__ uint4 ldg16(const void* p) {
  return __ldg(reinterpret_cast<const uint4*>(p));
}
__device__ __forceinline__ uint4 ld16(const void* p) { return *reinterpret_cast<const uint4*>(p); }
__device__ __forceinline__ void st16(void* p, uint4 v) { *reinterpret_cast<uint4*>(p) = v; }

__device__ __forceinline__ void unpack(const uint4& v, float* f, float) {
  f[0] = __uint_as_float(v.x);
  f[1] = __uint_as_float(v.y);
  f[2] = __uint_as_float(v.z);
  f[3] = __uint_as_float(v.w);
}
__device__ __forceinline__ void unpack(const uint4& v, float* f, __nv_bfloat16) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}
__device__ __forceinline__ uint4 pack(const float* f, float) {
  return make_uint4(__float_as_uint(f[0]), __float_as_uint(f[1]), __float_as_uint(f[2]),
                    __float_as_uint(f[3]));
}
__device__ __forceinline__ uint32_t pack2_bf16(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}
__device__ __forceinline__ uint4 pack(const float* f, __nv_bfloat16) {
  return make_uint4(pack2_bf16(f[0], f[1]), pack2_bf16(f[2], f[3]), pack2_bf16(f[4], f[5]),
                    pack2_bf16(f[6], f[7]));
}

__device__ __forceinline__ float to_f32(float x) { return x; }
__device__ __forceinline__ float to_f32(__nv_bfloat16 x) { return __bfloat162float(x); }
template <typename T>
__device__ __forceinline__ T from_f32(float x);
template <>
__device__ __forceinline__ float from_f32<float>(float x) {
  return x;
}
template <>
__device__ __forceinline__ __nv_bfloat16 from_f32<__nv_bfloat16>(float x) {
  return __float2bfloat16_rn(x);
}

__device__ __forceinline__ int node_type_of(const GraphMeta& m, int64_t node) {
  int t = 0;
#pragma unroll
  for (int k = 1; k < kMaxTypes; ++k)
    if (k < m.num_types && node >= m.type_off[k]) t = k;
  return t;
}

// ---------------------------------------------------------------------------------------------
// internal entry points implemented in the other translation units
// ---------------------------------------------------------------------------------------------
// exclusive scan of n int32 counts into out[0..n] (out[n] = total); in may equal out.
size_t scan_scratch_bytes(int64_t n);
hg_status exclusive_scan(const int32_t* in, int32_t* out, int64_t n, void* scratch, cudaStream_t s);

}  // namespace hg
