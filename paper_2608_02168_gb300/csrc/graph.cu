// Relation-typed CSR / CSC construction on the device.
//
// The adjacency of one overlapping subgraph (Section 2.2 typed relations; Section 3.1, Eq. 5 and
// Algorithm 1: the induced subgraph of V_k extended by the sampled candidates) is laid out per
// relation twice: by destination (CSR, forward aggregation of Eq. 10) and by source (CSC, its
// transpose in the backward pass).  Rows of all relations are concatenated: relation r owns CSR
// rows [row_base[r], row_base[r+1]) = its destination type's nodes in local order, and CSC rows
// [csc_base[r], csc_base[r+1]) = its source type's nodes.
//
// Construction: each edge gets a row key (or a sentinel key past the last row when invalid), a
// STABLE least-significant-digit radix sort of (key, edge id) places every edge in its row with
// ascending edge ids, and the row pointers are read off the sorted keys (no atomics, so hub rows
// cost nothing extra).  The layout is therefore unique and bit-reproducible.
//
// Three stable sorts build both layouts: by source id, then by CSR row (so a CSR row lists its
// in-edges by (source, edge id)), then that order by CSC row (a CSC row lists its out-edges by
// (destination, edge id)).  Parallel edges are thus adjacent in both, and runs of equal neighbours
// become the mean layer's aggregation lists (column, multiplicity); the non-empty CSR rows get a
// compact numbering, the rows in which the mean layer stores M_r and dMs_r.
#include <algorithm>

#include "hg_internal.cuh"

namespace hg {

// ---------------------------------------------------------------------------------------------
// exclusive scan (int32), three phases: tile sums -> scan of tile sums (recursive) -> tile scan
// ---------------------------------------------------------------------------------------------
constexpr int kScanThreads = 256;
constexpr int kScanSub = 4;                                            // 128-item sub-blocks per warp
constexpr int kScanWarpItems = 128 * kScanSub;                         // a warp's contiguous segment
constexpr int kScanTile = kScanThreads / 32 * kScanWarpItems;          // 4096 items per block

__device__ __forceinline__ int warp_inclusive_scan(int v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    int y = __shfl_up_sync(0xffffffffu, v, o);
    if (lane >= o) v += y;
  }
  return v;
}

__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Items i .. i + 3 (zero past n): one 16-byte load where the array is aligned and the four are in
// range.  A warp's lanes cover 128 consecutive items per call, so every access is coalesced.
__device__ __forceinline__ int4 scan_load4(const int32_t* in, int64_t i, int64_t n, bool vec) {
  if (vec && i + 3 < n) return *reinterpret_cast<const int4*>(in + i);
  int4 r;
  r.x = i < n ? in[i] : 0;
  r.y = i + 1 < n ? in[i + 1] : 0;
  r.z = i + 2 < n ? in[i + 2] : 0;
  r.w = i + 3 < n ? in[i + 3] : 0;
  return r;
}

__device__ __forceinline__ void scan_store4(int32_t* out, int64_t i, int64_t n, int4 v, bool vec) {
  if (vec && i + 3 < n) {
    *reinterpret_cast<int4*>(out + i) = v;
    return;
  }
  if (i < n) out[i] = v.x;
  if (i + 1 < n) out[i + 1] = v.y;
  if (i + 2 < n) out[i + 2] = v.z;
  if (i + 3 < n) out[i + 3] = v.w;
}

// sums[tile] = sum of the tile's kScanTile items (warp w: items tile * kScanTile + w * 512 ..)
__global__ void __launch_bounds__(kScanThreads) scan_tile_sums(const int32_t* __restrict__ in, int64_t n,
                                                                int32_t* __restrict__ sums) {
  __shared__ int wt[kScanThreads / 32];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool vec = (reinterpret_cast<uintptr_t>(in) & 15) == 0;
  const int64_t seg = (int64_t)blockIdx.x * kScanTile + (int64_t)warp * kScanWarpItems;
  int s = 0;
#pragma unroll
  for (int j = 0; j < kScanSub; ++j) {
    const int4 v = scan_load4(in, seg + 128 * j + 4 * lane, n, vec);
    s += v.x + v.y + v.z + v.w;
  }
  s = warp_sum_i(s);
  if (lane == 0) wt[warp] = s;
  __syncthreads();
  if (threadIdx.x == 0) {
    int t = 0;
#pragma unroll
    for (int w = 0; w < kScanThreads / 32; ++w) t += wt[w];
    sums[blockIdx.x] = t;
  }
}

// Exclusive scan of one tile plus tile_off[tile] (nullptr: a single tile starting at 0); the last
// tile also writes out[n] = the grand total.  out may equal in.
__global__ void __launch_bounds__(kScanThreads) scan_tiles(const int32_t* in, int32_t* out, int64_t n,
                                                            const int32_t* __restrict__ tile_off) {
  __shared__ int wt[kScanThreads / 32 + 1];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const bool vec = ((reinterpret_cast<uintptr_t>(in) | reinterpret_cast<uintptr_t>(out)) & 15) == 0;
  const int64_t seg = (int64_t)blockIdx.x * kScanTile + (int64_t)warp * kScanWarpItems;
  int4 v[kScanSub];
  int ls[kScanSub];
  int s = 0;
#pragma unroll
  for (int j = 0; j < kScanSub; ++j) {
    v[j] = scan_load4(in, seg + 128 * j + 4 * lane, n, vec);
    ls[j] = v[j].x + v[j].y + v[j].z + v[j].w;
    s += ls[j];
  }
  s = warp_sum_i(s);
  if (lane == 0) wt[warp] = s;
  __syncthreads();
  if (threadIdx.x == 0) {  // exclusive prefix over the warps, block total last
    int run = tile_off ? tile_off[blockIdx.x] : 0;
#pragma unroll
    for (int w = 0; w < kScanThreads / 32; ++w) {
      const int t = wt[w];
      wt[w] = run;
      run += t;
    }
    wt[kScanThreads / 32] = run;
  }
  __syncthreads();
  int carry = wt[warp];
#pragma unroll
  for (int j = 0; j < kScanSub; ++j) {
    const int incl = warp_inclusive_scan(ls[j]);
    int run = carry + incl - ls[j];
    int4 o;
    o.x = run;
    run += v[j].x;
    o.y = run;
    run += v[j].y;
    o.z = run;
    run += v[j].z;
    o.w = run;
    scan_store4(out, seg + 128 * j + 4 * lane, n, o, vec);
    carry += __shfl_sync(0xffffffffu, incl, 31);
  }
  if (blockIdx.x == gridDim.x - 1 && threadIdx.x == 0) out[n] = wt[kScanThreads / 32];
}

size_t scan_scratch_bytes(int64_t n) {
  size_t b = 0;
  while (n > kScanTile) {
    n = ceil_div(n, kScanTile);
    b += align_up((size_t)(n + 1) * sizeof(int32_t));
  }
  return b + 256;
}

hg_status exclusive_scan(const int32_t* in, int32_t* out, int64_t n, void* scratch, cudaStream_t s) {
  if (n <= 0) {
    if (n == 0) HG_CUDA(cudaMemsetAsync(out, 0, sizeof(int32_t), s));
    return HG_OK;
  }
  if (n <= kScanTile)
    return launch("scan_tiles", scan_tiles, dim3(1), dim3(kScanThreads), 0, s, in, out, n,
                  (const int32_t*)nullptr);
  const int64_t tiles = ceil_div(n, kScanTile);
  int32_t* sums = static_cast<int32_t*>(scratch);
  char* rest = static_cast<char*>(scratch) + align_up((size_t)(tiles + 1) * sizeof(int32_t));
  HG_TRY(launch("scan_tile_sums", scan_tile_sums, dim3((unsigned)tiles), dim3(kScanThreads), 0, s,
                in, n, sums));
  HG_TRY(exclusive_scan(sums, sums, tiles, rest, s));
  return launch("scan_tiles", scan_tiles, dim3((unsigned)tiles), dim3(kScanThreads), 0, s, in, out,
                n, (const int32_t*)sums);
}

// ---------------------------------------------------------------------------------------------
// stable LSD radix sort of (uint32 key, uint32 value) pairs, 8-bit digits
// ---------------------------------------------------------------------------------------------
constexpr int kSortThreads = 512;
constexpr int kSortWarps = kSortThreads / 32;
constexpr int kSortItems = 8;                           // per thread
constexpr int kSortTile = kSortThreads * kSortItems;    // 4096 per block
constexpr int kWarpSlice = kSortTile / kSortWarps;      // 256 consecutive items per warp
constexpr int kRadix = 256;

// Per-tile digit counts hist[digit * tiles + tile]; each warp counts into its own shared
// histogram (atomics only contend within a warp), and the warp histograms are added at the end.
__global__ void __launch_bounds__(kSortThreads) radix_hist(const uint32_t* __restrict__ keys, int64_t n,
                                                           int shift, int32_t* __restrict__ hist,
                                                           int64_t tiles) {
  __shared__ int h[kSortWarps][kRadix];
  for (int i = threadIdx.x; i < kSortWarps * kRadix; i += kSortThreads) (&h[0][0])[i] = 0;
  __syncthreads();
  const int warp = threadIdx.x >> 5;
  // this thread's 8 consecutive keys, loaded before any of them is counted
  const int64_t first = (int64_t)blockIdx.x * kSortTile + (int64_t)threadIdx.x * kSortItems;
  uint32_t k[kSortItems];
  if (first + kSortItems <= n) {
    const uint4 a = *reinterpret_cast<const uint4*>(keys + first);
    const uint4 b = *reinterpret_cast<const uint4*>(keys + first + 4);
    k[0] = a.x; k[1] = a.y; k[2] = a.z; k[3] = a.w;
    k[4] = b.x; k[5] = b.y; k[6] = b.z; k[7] = b.w;
  } else {
#pragma unroll
    for (int i = 0; i < kSortItems; ++i) k[i] = first + i < n ? keys[first + i] : 0u;
  }
#pragma unroll
  for (int i = 0; i < kSortItems; ++i)
    if (first + i < n) atomicAdd(&h[warp][(k[i] >> shift) & (kRadix - 1)], 1);
  __syncthreads();
  if (threadIdx.x < kRadix) {
    int t = 0;
#pragma unroll
    for (int w = 0; w < kSortWarps; ++w) t += h[w][threadIdx.x];
    hist[(int64_t)threadIdx.x * tiles + blockIdx.x] = t;
  }
}

// Stable scatter of one 4096-item tile.  (1) Warp w reads its 256 consecutive items, 32 at a time
// (coalesced), into registers.  (2) It ranks them round by round with __match_any_sync, keeping
// per-digit running counts, so the item order inside the tile is (warp, round, lane).  (3) Per-digit
// prefixes over warps and over digits give every item its position in the tile sorted by digit
// (equal digits keep their order), where it is written in shared memory.  (4) Consecutive threads
// write consecutive sorted items to base[digit] + (position - tile start of the digit): runs of
// equal digits go out coalesced.
template <bool kTwo>
__global__ void __launch_bounds__(kSortThreads) radix_scatter(
    const uint32_t* __restrict__ keys_in, const uint32_t* __restrict__ vals_in,
    const uint32_t* __restrict__ vals2_in, uint32_t* __restrict__ keys_out, uint32_t* __restrict__ vals_out,
    uint32_t* __restrict__ vals2_out, int64_t n, int shift, const int32_t* __restrict__ offs, int64_t tiles) {
  constexpr int R = kWarpSlice / 32;  // rounds (items per thread)
  extern __shared__ uint32_t sort_smem[];
  uint32_t* skey = sort_smem;           // sorted tile
  uint32_t* sval = skey + kSortTile;
  uint32_t* sval2 = sval + kSortTile;   // (kTwo)
  int (*whist)[kRadix] = reinterpret_cast<int (*)[kRadix]>(sval2 + (kTwo ? kSortTile : 0));
  __shared__ int dstart[kRadix];  // tile position where each digit's run starts
  __shared__ int gbase[kRadix];   // global position of the digit's run of this tile
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t t0 = (int64_t)blockIdx.x * kSortTile;
  const int cnt = (int)min((int64_t)kSortTile, n - t0);
  for (int i = threadIdx.x; i < kSortWarps * kRadix; i += kSortThreads) (&whist[0][0])[i] = 0;
  if (threadIdx.x < kRadix) gbase[threadIdx.x] = offs[(int64_t)threadIdx.x * tiles + blockIdx.x];
  uint32_t k[R], v[R], v2[R];
  int rank[R];
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int j = warp * kWarpSlice + r * 32 + lane;
    if (j < cnt) {
      k[r] = keys_in[t0 + j];
      v[r] = vals_in ? vals_in[t0 + j] : (uint32_t)(t0 + j);  // first pass: the input position
      if (kTwo) v2[r] = vals2_in[t0 + j];
    }
  }
  __syncthreads();
  const unsigned lt_mask = (1u << lane) - 1u;
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int j = warp * kWarpSlice + r * 32 + lane;
    const int d = j < cnt ? (int)((k[r] >> shift) & (kRadix - 1)) : kRadix;
    const unsigned peers = __match_any_sync(0xffffffffu, d);
    const int c = d < kRadix ? whist[warp][d] : 0;
    __syncwarp();
    if (d < kRadix && lane == __ffs(peers) - 1) whist[warp][d] = c + __popc(peers);
    __syncwarp();
    rank[r] = c + __popc(peers & lt_mask);
  }
  __syncthreads();
  if (threadIdx.x < kRadix) {  // per digit: exclusive prefix over warps; tile total
    int run = 0;
#pragma unroll
    for (int w = 0; w < kSortWarps; ++w) {
      const int c = whist[w][threadIdx.x];
      whist[w][threadIdx.x] = run;
      run += c;
    }
    dstart[threadIdx.x] = run;
  }
  __syncthreads();
  if (warp == 0) {  // exclusive scan of the 256 digit totals
    int vv[kRadix / 32], sum = 0;
#pragma unroll
    for (int i = 0; i < kRadix / 32; ++i) {
      vv[i] = dstart[lane * (kRadix / 32) + i];
      sum += vv[i];
    }
    int incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    int run = incl - sum;
#pragma unroll
    for (int i = 0; i < kRadix / 32; ++i) {
      dstart[lane * (kRadix / 32) + i] = run;
      run += vv[i];
    }
  }
  __syncthreads();
#pragma unroll
  for (int r = 0; r < R; ++r) {
    const int j = warp * kWarpSlice + r * 32 + lane;
    if (j < cnt) {
      const int d = (int)((k[r] >> shift) & (kRadix - 1));
      const int p = dstart[d] + whist[warp][d] + rank[r];
      skey[p] = k[r];
      sval[p] = v[r];
      if (kTwo) sval2[p] = v2[r];
    }
  }
  __syncthreads();
  for (int p = threadIdx.x; p < cnt; p += kSortThreads) {
    const uint32_t kk = skey[p];
    const int d = (int)((kk >> shift) & (kRadix - 1));
    const int64_t pos = (int64_t)gbase[d] + (p - dstart[d]);
    keys_out[pos] = kk;
    vals_out[pos] = sval[p];
    if (kTwo) vals2_out[pos] = sval2[p];
  }
}

struct SortBuffers {
  uint32_t* ckeys;  // CSR row keys (payload of the first sort), then the CSC keys
  uint32_t* keys[2];
  uint32_t* vals[2];
  uint32_t* vals2[2];  // second payload (carried so the finish passes read sequentially)
  int32_t* hist;
  void* scan_scratch;
};

static int64_t sort_tiles(int64_t n) { return std::max<int64_t>(1, ceil_div(n, kSortTile)); }
// dynamic shared memory of radix_scatter<true>: the sorted tile (key, value, payload), warp histograms
constexpr size_t kScatterSmem = 3 * kSortTile * sizeof(uint32_t) + kSortWarps * kRadix * sizeof(int);

// Sorts (key, value, second payload) triples by the low `bits` key bits (at least one pass), stable.
// The first pass reads keys_src, vals_src (null: the input positions) and vals2_src, which may lie
// in buffer `start` (it writes buffer start ^ 1 first); returns the buffer index holding the sorted
// keys.  The last pass writes the payloads to vals_final / vals2_final when those are given (the
// caller's final arrays), else to the sort buffers beside the keys.
static hg_status radix_sort(SortBuffers& b, int64_t n, int bits, const uint32_t* keys_src, const uint32_t* vals_src,
                            const uint32_t* vals2_src, int start, cudaStream_t s, int* result,
                            uint32_t* vals_final = nullptr, uint32_t* vals2_final = nullptr) {
  static bool attr = false;
  if (!attr) {
    HG_CUDA(cudaFuncSetAttribute(radix_scatter<true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kScatterSmem));
    attr = true;
  }
  int cur = start;
  const int64_t tiles = sort_tiles(n);
  const uint32_t* k = keys_src;
  const uint32_t* v = vals_src;
  const uint32_t* v2 = vals2_src;
  const int nb = std::max(bits, 1);
  for (int shift = 0; shift < nb; shift += 8) {
    const bool last = shift + 8 >= nb;
    uint32_t* vo = last && vals_final ? vals_final : b.vals[cur ^ 1];
    uint32_t* v2o = last && vals2_final ? vals2_final : b.vals2[cur ^ 1];
    HG_TRY(launch("radix_hist", radix_hist, dim3((unsigned)tiles), dim3(kSortThreads), 0, s, k, n, shift, b.hist,
                  tiles));
    HG_TRY(exclusive_scan(b.hist, b.hist, tiles * kRadix, b.scan_scratch, s));
    HG_TRY(launch("radix_scatter", radix_scatter<true>, dim3((unsigned)tiles), dim3(kSortThreads), kScatterSmem, s, k, v, v2,
                  b.keys[cur ^ 1], vo, v2o, n, shift, (const int32_t*)b.hist, tiles));
    k = b.keys[cur ^ 1];
    v = vo;
    v2 = v2o;
    cur ^= 1;
  }
  *result = cur;
  return HG_OK;
}

// ---------------------------------------------------------------------------------------------
// CSR / CSC kernels
// ---------------------------------------------------------------------------------------------
// Keys of the first sort: the source node id of every valid edge (0 for invalid ones), and, as its
// payload, the CSR row key (destination row; the sentinel past the last row for an invalid edge:
// relation or endpoint out of range, endpoint of the wrong type).  The relation tables are read
// from shared memory.
__global__ void __launch_bounds__(256) edge_keys(const int32_t* __restrict__ src, const int32_t* __restrict__ dst,
                                                 const int32_t* __restrict__ rel, int64_t E, GraphMeta m,
                                                 int64_t rows, uint32_t* __restrict__ skeys,
                                                 uint32_t* __restrict__ rkeys) {
  __shared__ int64_t row0[kMaxRels];  // first row of relation r minus its destination type's offset
  __shared__ int32_t rsrc[kMaxRels], rdst[kMaxRels];
  if (threadIdx.x < kMaxRels) {
    const int r = threadIdx.x;
    if (r < m.num_rels) {
      rsrc[r] = m.rel_src[r];
      rdst[r] = m.rel_dst[r];
      row0[r] = m.row_base[r] - m.type_off[m.rel_dst[r]];
    }
  }
  __syncthreads();
  const int64_t N = m.type_off[m.num_types];
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < E; e += (int64_t)gridDim.x * blockDim.x) {
    const int r = rel[e];
    const int64_t sn = src[e], tn = dst[e];
    bool ok = r >= 0 && r < m.num_rels && sn >= 0 && sn < N && tn >= 0 && tn < N;
    int64_t key = rows;  // invalid edges sort after every row
    if (ok && node_type_of(m, sn) == rsrc[r] && node_type_of(m, tn) == rdst[r]) key = row0[r] + tn;
    else ok = false;
    skeys[e] = ok ? (uint32_t)sn : 0u;
    rkeys[e] = (uint32_t)key;
  }
}

// Keys of the CSC sort, read off the CSR order (row key, source id) position by position: the CSC
// row (relation, source) of each valid edge and its destination node id; invalid edges (positions
// from ptr[rows] on) get the sentinel past the last CSC row.  A stable sort of the CSR order by
// these keys lists each CSC row by (destination, edge id).  dst_out may alias rkey (each position
// is read before it is written, by the same thread).
__global__ void csc_keys_from_csr(const uint32_t* rkey, const uint32_t* __restrict__ srcs, int64_t E,
                                  const int32_t* __restrict__ ptr, int64_t rows, int64_t crows, GraphMeta m,
                                  uint32_t* __restrict__ ckey, uint32_t* dst_out) {
  const int64_t nv = ptr[rows];
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < E; p += (int64_t)gridDim.x * blockDim.x) {
    if (p >= nv) {
      ckey[p] = (uint32_t)crows;
      dst_out[p] = 0u;
      continue;
    }
    const int64_t key = rkey[p];
    int r = 0;
#pragma unroll
    for (int k = 1; k < kMaxRels; ++k)
      if (k < m.num_rels && key >= m.row_base[k]) r = k;
    const int64_t d = m.type_off[m.rel_dst[r]] + (key - m.row_base[r]);
    ckey[p] = (uint32_t)(m.csc_base[r] + ((int64_t)srcs[p] - m.type_off[m.rel_src[r]]));
    dst_out[p] = (uint32_t)d;
  }
}

// ---------------------------------------------------------------------------------------------
// non-empty CSR rows: the relation rows the mean layer stores (a row without in-edges has M = 0
// and is never stored, read or gathered)
// ---------------------------------------------------------------------------------------------
__global__ void nonempty_flags(const int32_t* __restrict__ ptr, int64_t rows, int32_t* __restrict__ flag) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += (int64_t)gridDim.x * blockDim.x)
    flag[r] = ptr[r + 1] > ptr[r] ? 1 : 0;
}

// long rows of the fused layer: flag[r] = 1 when CSR row r has more than kFuseRuns runs
__global__ void long_flags(const int32_t* __restrict__ aptr, int64_t rows, int32_t* __restrict__ flag) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += (int64_t)gridDim.x * blockDim.x)
    flag[r] = aptr[r + 1] - aptr[r] > kFuseRuns ? 1 : 0;
}

// list[ofs[r]] = r for every flagged row r (ofs = the exclusive scan of the flags)
__global__ void compact_list(const int32_t* __restrict__ flag, const int32_t* __restrict__ ofs, int64_t rows,
                             int32_t* __restrict__ list) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += (int64_t)gridDim.x * blockDim.x)
    if (flag[r]) list[ofs[r]] = (int32_t)r;
}

// mbase[r] = compact index of relation r's first non-empty row (pos = the scan of the flags, whose
// entry `rows` is the number of non-empty rows).
__global__ void compact_bases(const int32_t* __restrict__ pos, GraphMeta m, int32_t* __restrict__ mbase) {
  const int r = threadIdx.x;
  if (r <= m.num_rels) mbase[r] = pos[m.row_base[r]];
}

// In place: mrow[row] = its compact index when non-empty, `rows` (out of range) otherwise; mlist[k]
// = the CSR row of compact row k.
__global__ void compact_rows(const int32_t* __restrict__ flag, int64_t rows, int32_t* __restrict__ mrow,
                             int32_t* __restrict__ mlist) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += (int64_t)gridDim.x * blockDim.x) {
    const int32_t k = mrow[r];
    if (flag[r]) {
      mlist[k] = (int32_t)r;
    } else {
      mrow[r] = (int32_t)rows;
    }
  }
}

// ---------------------------------------------------------------------------------------------
// run-length coalescing of parallel edges: a row (ptr, col) whose equal entries are adjacent
// becomes (uptr, ucol, ucnt): one entry per distinct column with its multiplicity, in the same order
// ---------------------------------------------------------------------------------------------
// flag[p] = 1 where a run starts: p = 0 or col[p] != col[p - 1] (row starts are added next), for
// p < ptr[rows]; 0 up to cap (the capacity the scan runs over).
__global__ void run_flags(const int32_t* __restrict__ col, const int32_t* __restrict__ ptr, int64_t rows, int64_t cap,
                          int32_t* __restrict__ flag) {
  const int64_t n = ptr[rows];
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < cap; p += (int64_t)gridDim.x * blockDim.x)
    flag[p] = (p < n && (p == 0 || col[p] != col[p - 1])) ? 1 : 0;
}

// every non-empty row starts a run
__global__ void run_row_starts(const int32_t* __restrict__ ptr, int64_t rows, int32_t* __restrict__ flag) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows; r += (int64_t)gridDim.x * blockDim.x)
    if (ptr[r + 1] > ptr[r]) flag[ptr[r]] = 1;
}

// With u = the exclusive scan of the run-start flags (u[n] = number of runs): position p starts a
// run exactly when u[p + 1] != u[p]; run k = u[p] gets ucol[k] = col[p] (or map[col[p]] when a map
// is given) and its start upos[k] = p; upos[U] = n.  Four positions per thread, u read as 16-byte
// vectors (the flags themselves are not read again).
__global__ void run_write(const int32_t* __restrict__ u, const int32_t* __restrict__ col,
                          const int32_t* __restrict__ ptr, int64_t rows, const int32_t* __restrict__ map,
                          int32_t* __restrict__ ucol, int32_t* __restrict__ upos) {
  const int64_t n = ptr[rows];
  const bool vec = (reinterpret_cast<uintptr_t>(u) & 15) == 0;
  for (int64_t p = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) * 4; p <= n;
       p += (int64_t)gridDim.x * blockDim.x * 4) {
    int32_t v[5];
    if (vec && p + 4 <= n) {
      const int4 w = *reinterpret_cast<const int4*>(u + p);
      v[0] = w.x;
      v[1] = w.y;
      v[2] = w.z;
      v[3] = w.w;
      v[4] = u[p + 4];
    } else {
#pragma unroll
      for (int i = 0; i < 5; ++i) v[i] = p + i <= n ? u[p + i] : 0;
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int64_t q = p + i;
      if (q < n && v[i + 1] != v[i]) {
        ucol[v[i]] = map ? map[col[q]] : col[q];
        upos[v[i]] = (int32_t)q;
      } else if (q == n) {
        upos[v[i]] = (int32_t)n;
      }
    }
  }
}

// ucnt[k] = upos[k + 1] - upos[k] (the run's length) for k < U; uptr[r] = u[ptr[r]] for r <= rows.
__global__ void run_finish(const int32_t* __restrict__ u, const int32_t* __restrict__ upos,
                           const int32_t* __restrict__ ptr, int64_t rows, int32_t* __restrict__ ucnt,
                           int32_t* __restrict__ uptr) {
  const int64_t U = u[ptr[rows]];
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < U; k += stride) ucnt[k] = upos[k + 1] - upos[k];
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r <= rows; r += stride) uptr[r] = u[ptr[r]];
}

// Row pointers from the sorted keys: ptr[k] = first position whose key is >= k, k in [0, rows].
// Position p owns the rows k with key[p-1] < k <= key[p] (key[-1] = -1, key[n] = rows), so every
// entry is written exactly once and empty rows get the position of the next non-empty one.  The
// owner of k = rows also writes n - ptr[rows] (the positions with keys past the last row) to
// *invalid when that is given.
__global__ void row_ptr_from_keys(const uint32_t* __restrict__ keys, int64_t n, int64_t rows,
                                  int32_t* __restrict__ ptr, int32_t* __restrict__ invalid) {
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p <= n;
       p += (int64_t)gridDim.x * blockDim.x) {
    const int64_t lo = p == 0 ? 0 : (int64_t)keys[p - 1] + 1;
    const int64_t hi = p == n ? rows : min((int64_t)keys[p], rows);
    for (int64_t k = lo; k <= hi; ++k) ptr[k] = (int32_t)p;
    if (invalid && lo <= rows && rows <= hi) *invalid = (int32_t)(n - p);
  }
}

// Out-degree of every node over all relations leaving its type (the length of its node-major row).
__global__ void node_out_counts(const int32_t* __restrict__ cptr, GraphMeta m, int32_t* __restrict__ cnt) {
  __shared__ int64_t cbase[kMaxRels];  // CSC row of the type's node 0 in relation r, minus the type offset
  __shared__ int32_t rsrc[kMaxRels];
  if (threadIdx.x < kMaxRels) {
    const int r = threadIdx.x;
    rsrc[r] = r < m.num_rels ? m.rel_src[r] : -1;
    if (r < m.num_rels) cbase[r] = m.csc_base[r] - m.type_off[m.rel_src[r]];
  }
  __syncthreads();
  const int64_t N = m.type_off[m.num_types];
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < N; i += (int64_t)gridDim.x * blockDim.x) {
    const int t = node_type_of(m, i);
    int c = 0;
#pragma unroll
    for (int r = 0; r < kMaxRels; ++r)
      if (rsrc[r] == t) c += cptr[cbase[r] + i + 1] - cptr[cbase[r] + i];
    cnt[i] = c;
  }
}

// CSC coefficients and the node-major list of out-edges used by the backward aggregation, from
// the sorted CSC keys and destination ids (the sort's last pass wrote csc_col and csc_eid): the
// relation is read off the key, 1/deg_r(destination) from the CSR row pointers.  Node i's row holds,
// relation by relation (ascending) and in CSC order within a relation, the dMs row of each edge's
// destination (row_base[r] + local destination id).
__global__ void csc_finish(const uint32_t* __restrict__ key_sorted, const int32_t* __restrict__ ccol,
                           const int32_t* __restrict__ cptr, int64_t crows, GraphMeta m,
                           const int32_t* __restrict__ csr_ptr, const int32_t* __restrict__ nptr,
                           float* __restrict__ coef, int32_t* __restrict__ ncol) {
  const int64_t nv = cptr[crows];
  for (int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; p < nv;
       p += (int64_t)gridDim.x * blockDim.x) {
    const int64_t key = key_sorted[p];
    int r = 0;
#pragma unroll
    for (int k = 1; k < kMaxRels; ++k)
      if (k < m.num_rels && key >= m.csc_base[k]) r = k;
    const int32_t j = ccol[p];
    const int64_t row = m.row_base[r] + (j - m.type_off[m.rel_dst[r]]);
    const int deg = csr_ptr[row + 1] - csr_ptr[row];
    coef[p] = __fdiv_rn(1.0f, (float)deg);
    // node-major position: the node's row start, the edges of its earlier relations, the rank in this one
    const int t = m.rel_src[r];
    const int64_t il = key - m.csc_base[r];  // type-local source id
    int64_t pos = nptr[m.type_off[t] + il] + (p - cptr[key]);
#pragma unroll
    for (int k = 0; k < kMaxRels; ++k)
      if (k < r && m.rel_src[k] == t) pos += cptr[m.csc_base[k] + il + 1] - cptr[m.csc_base[k] + il];
    ncol[pos] = (int32_t)row;
  }
}

__global__ void chunk_counts(const int32_t* __restrict__ ptr, int64_t rows, int32_t* __restrict__ cnt) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows;
       r += (int64_t)gridDim.x * blockDim.x) {
    const int deg = ptr[r + 1] - ptr[r];
    cnt[r] = deg > kHubDegree ? (deg + kChunkEdges - 1) / kChunkEdges : 0;
  }
}

__global__ void chunk_fill(const int32_t* __restrict__ ofs, int64_t rows, int32_t* __restrict__ chunk_row) {
  for (int64_t r = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; r < rows;
       r += (int64_t)gridDim.x * blockDim.x) {
    for (int c = ofs[r]; c < ofs[r + 1]; ++c) chunk_row[c] = (int32_t)r;
  }
}

// ---- node order of the forward projection: a stable counting sort of each type's nodes by relation
// mask (at most kMaxRels relations into a type: 2^8 mask values).  Blocks own kOrderTile nodes.
constexpr int kOrderTile = 2048;
constexpr int kMaskValues = 1 << kMaxRels;

struct TypeRels {
  int n;                     // relations into the type
  int64_t row0[kMaxRels];    // CSR row of the type's local node 0 in each, by ascending relation id
};

__device__ __forceinline__ uint32_t node_mask(const int32_t* __restrict__ csr_ptr, const TypeRels& tr, int64_t j) {
  uint32_t m = 0;
  for (int k = 0; k < tr.n; ++k) {
    const int64_t row = tr.row0[k] + j;
    if (__ldg(csr_ptr + row + 1) > __ldg(csr_ptr + row)) m |= 1u << k;
  }
  return m;
}

// hist[v * nblk + block] = nodes of the block with mask v
__global__ void __launch_bounds__(256) order_hist(const int32_t* __restrict__ csr_ptr, TypeRels tr, int64_t n,
                                                  int nblk, int32_t* __restrict__ hist) {
  __shared__ int32_t h[kMaskValues];
  const int V = 1 << tr.n;
  for (int v = threadIdx.x; v < V; v += blockDim.x) h[v] = 0;
  __syncthreads();
  const int64_t j0 = (int64_t)blockIdx.x * kOrderTile;
  for (int k = threadIdx.x; k < kOrderTile; k += blockDim.x) {
    const int64_t j = j0 + k;
    if (j < n) atomicAdd(&h[node_mask(csr_ptr, tr, j)], 1);
  }
  __syncthreads();
  for (int v = threadIdx.x; v < V; v += blockDim.x) hist[(int64_t)v * nblk + blockIdx.x] = h[v];
}

// perm[ofs[v * nblk + block] + rank] = j, rank = the node's place among the block's nodes with mask v
// in ascending id (rounds of 256 nodes; within a round, warp-level ranks plus earlier warps' counts)
__global__ void __launch_bounds__(256) order_scatter(const int32_t* __restrict__ csr_ptr, TypeRels tr, int64_t n,
                                                     int nblk, const int32_t* __restrict__ ofs,
                                                     int32_t* __restrict__ perm) {
  __shared__ int32_t next[kMaskValues];
  __shared__ int32_t wcnt[8][kMaskValues];
  const int V = 1 << tr.n;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int v = threadIdx.x; v < V; v += 256) next[v] = ofs[(int64_t)v * nblk + blockIdx.x];
  const int64_t j0 = (int64_t)blockIdx.x * kOrderTile;
  for (int k = 0; k < kOrderTile; k += 256) {
    for (int i = threadIdx.x; i < 8 * V; i += 256) wcnt[i / V][i % V] = 0;
    __syncthreads();
    const int64_t j = j0 + k + threadIdx.x;
    const bool live = j < n;
    const uint32_t mk = live ? node_mask(csr_ptr, tr, j) : 0xFFFFFFFFu;
    const uint32_t peers = __match_any_sync(0xffffffffu, mk);
    const int lrank = __popc(peers & ((1u << lane) - 1u));
    if (live && lrank == 0) wcnt[warp][mk] = __popc(peers);
    __syncthreads();
    if (live) {
      int pos = next[mk] + lrank;
      for (int w = 0; w < warp; ++w) pos += wcnt[w][mk];
      perm[pos] = (int32_t)j;
    }
    __syncthreads();
    for (int v = threadIdx.x; v < V; v += 256) {
      int c = 0;
      for (int w = 0; w < 8; ++w) c += wcnt[w][v];
      next[v] += c;
    }
    __syncthreads();
  }
}

// tmask[q] = OR of the masks at positions kProjTileRows q .. + kProjTileRows - 1 (one warp per tile)
__global__ void __launch_bounds__(256) order_tiles(const int32_t* __restrict__ csr_ptr, TypeRels tr, int64_t n,
                                                   const int32_t* __restrict__ perm, int64_t tiles,
                                                   int32_t* __restrict__ tmask) {
  const int64_t q = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (q >= tiles) return;
  uint32_t m = 0;
  for (int i = lane; i < kProjTileRows; i += 32) {
    const int64_t p = q * kProjTileRows + i;
    if (p < n) m |= node_mask(csr_ptr, tr, perm[p]);
  }
  m = __reduce_or_sync(0xffffffffu, m);
  if (lane == 0) tmask[q] = (int32_t)m;
}

static int64_t order_blocks(int64_t n) { return ceil_div(n, kOrderTile); }
// histogram entries over all types: sum_t 2^n_t ceil(n_t / kOrderTile) <= 2^8 (N / kOrderTile + kMaxTypes)
static int64_t order_hist_cap(int64_t N) { return (int64_t)kMaskValues * (N / kOrderTile + kMaxTypes); }
static int64_t order_tiles_cap(int64_t N) { return N / kProjTileRows + kMaxTypes; }

// Rows above kHubDegree hold sum ceil(deg / kChunkEdges) <= E / kChunkEdges + E / (kHubDegree + 1)
// chunks (each such row adds at most one partial chunk); +2 covers the integer floors.
static int64_t chunk_cap(int64_t E) { return E / kChunkEdges + E / (kHubDegree + 1) + 2; }
// a long row has more than kFuseRuns runs, each of at least one edge
static int64_t long_cap(int64_t E) { return E / (kFuseRuns + 1) + 1; }

struct GraphLayout {
  int32_t *csr_ptr, *csr_col, *csr_eid, *csc_ptr, *csc_col, *csc_eid;
  float* csc_coef;
  int32_t *node_ptr, *node_col;  // node-major out-edges (dMs rows) for the backward aggregation
  int32_t *invalid, *cnt;
  // parallel edges coalesced: CSR rows and node-major rows as (column, multiplicity) runs
  int32_t *agg_ptr, *agg_col, *agg_cnt, *agg_chunk_ofs, *agg_chunk_row;
  int32_t *bagg_ptr, *bagg_col, *bagg_cnt, *bagg_chunk_ofs, *bagg_chunk_row;
  int32_t *mrow, *mlist, *mbase;  // non-empty CSR rows: compact index per row, row per index, per relation
  int32_t *nperm, *tmask, *ohist, *oofs;  // node order by relation mask, tile masks, the sort's counts
  int32_t *long_ofs, *long_list;          // the fused layer's long rows
  SortBuffers sort;
};

static size_t carve_graph(void* ws, int64_t E, int64_t rows, int64_t crows, int64_t N, GraphLayout* L) {
  Carve c(ws);
  const int64_t Ea = std::max<int64_t>(E, 1);
  L->csr_ptr = c.take<int32_t>(rows + 1);
  L->csr_col = c.take<int32_t>(Ea);
  L->csr_eid = c.take<int32_t>(Ea);
  L->csc_ptr = c.take<int32_t>(crows + 1);
  L->csc_col = c.take<int32_t>(Ea);
  L->csc_eid = c.take<int32_t>(Ea);
  L->csc_coef = c.take<float>(Ea);
  L->node_ptr = c.take<int32_t>(N + 1);
  L->node_col = c.take<int32_t>(Ea);
  L->agg_ptr = c.take<int32_t>(rows + 1);
  L->agg_col = c.take<int32_t>(Ea);
  L->agg_cnt = c.take<int32_t>(Ea);
  L->agg_chunk_ofs = c.take<int32_t>(rows + 1);
  L->agg_chunk_row = c.take<int32_t>(chunk_cap(E));
  L->bagg_ptr = c.take<int32_t>(N + 1);
  L->bagg_col = c.take<int32_t>(Ea);
  L->bagg_cnt = c.take<int32_t>(Ea);
  L->bagg_chunk_ofs = c.take<int32_t>(N + 1);
  L->bagg_chunk_row = c.take<int32_t>(chunk_cap(E));
  L->mrow = c.take<int32_t>(rows + 1);
  L->mlist = c.take<int32_t>(rows + 1);
  L->mbase = c.take<int32_t>(kMaxRels + 1);
  L->nperm = c.take<int32_t>(std::max<int64_t>(N, 1));
  L->tmask = c.take<int32_t>(order_tiles_cap(N));
  L->long_ofs = c.take<int32_t>(rows + 1);
  L->long_list = c.take<int32_t>(long_cap(E));
  L->ohist = c.take<int32_t>(order_hist_cap(N) + 1);
  L->oofs = c.take<int32_t>(order_hist_cap(N) + 1);
  L->invalid = c.take<int32_t>(1);
  L->cnt = c.take<int32_t>(std::max(std::max(rows, crows), N) + 1);
  L->sort.ckeys = c.take<uint32_t>(Ea + 1);
  for (int i = 0; i < 2; ++i) {  // one entry more than the edges: the coalescing scans reuse them
    L->sort.keys[i] = c.take<uint32_t>(Ea + 1);
    L->sort.vals[i] = c.take<uint32_t>(Ea + 1);
    L->sort.vals2[i] = c.take<uint32_t>(Ea + 1);
  }
  const int64_t hist_n = sort_tiles(E) * kRadix;
  L->sort.hist = c.take<int32_t>(hist_n + 1);
  L->sort.scan_scratch =
      c.take<char>(scan_scratch_bytes(std::max(std::max(std::max(hist_n, rows), std::max(crows, N)),
                                               std::max(Ea, order_hist_cap(N)))));
  return c.used;
}

static hg_status make_meta(const int64_t* type_offsets, int32_t num_types, const hg_rel_desc* rels,
                           int32_t num_rels, GraphMeta* m) {
  HG_REQUIRE(type_offsets != nullptr && rels != nullptr, "type_offsets and rels must be non-null");
  if (num_types < 1 || num_types > kMaxTypes || num_rels < 1 || num_rels > kMaxRels) {
    set_error("need 1 <= num_types <= %d and 1 <= num_rels <= %d (got %d, %d)", kMaxTypes, kMaxRels,
              num_types, num_rels);
    return HG_ERR_UNSUPPORTED;
  }
  HG_REQUIRE(type_offsets[0] == 0, "type_offsets[0] must be 0");
  for (int t = 0; t < num_types; ++t)
    HG_REQUIRE(type_offsets[t + 1] >= type_offsets[t], "type_offsets must be non-decreasing");
  if (type_offsets[num_types] >= (int64_t(1) << 31)) {
    set_error("more than 2^31 - 1 nodes");
    return HG_ERR_UNSUPPORTED;
  }
  *m = GraphMeta{};
  m->num_types = num_types;
  m->num_rels = num_rels;
  for (int t = 0; t <= num_types; ++t) m->type_off[t] = type_offsets[t];
  for (int t = num_types + 1; t <= kMaxTypes; ++t) m->type_off[t] = type_offsets[num_types];
  m->row_base[0] = m->csc_base[0] = 0;
  for (int r = 0; r < num_rels; ++r) {
    const int s = rels[r].src_type, d = rels[r].dst_type;
    HG_REQUIRE(s >= 0 && s < num_types && d >= 0 && d < num_types,
               "relation %d has a node type out of range", r);
    m->rel_src[r] = s;
    m->rel_dst[r] = d;
    m->row_base[r + 1] = m->row_base[r] + (type_offsets[d + 1] - type_offsets[d]);
    m->csc_base[r + 1] = m->csc_base[r] + (type_offsets[s + 1] - type_offsets[s]);
  }
  if (m->row_base[num_rels] >= (int64_t(1) << 31) - 1 || m->csc_base[num_rels] >= (int64_t(1) << 31) - 1) {
    set_error("more than 2^31 - 2 relation rows");
    return HG_ERR_UNSUPPORTED;
  }
  return HG_OK;
}

static int bit_width(uint64_t x) {
  int b = 0;
  while (x) {
    ++b;
    x >>= 1;
  }
  return b;
}

static unsigned grid_for(int64_t n, int threads = 256) {
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(n, threads), 152 * 16));
}

// Runs of equal adjacent entries of (ptr, col): the flags, their scan (the run index of each
// position) and the runs' columns, multiplicities and row pointers.  Uses the sort buffers.
static hg_status coalesce_runs(const int32_t* col, const int32_t* ptr, int64_t rows, int64_t E, const int32_t* map,
                               GraphLayout& L, int32_t* ucol, int32_t* ucnt, int32_t* uptr, cudaStream_t s) {
  int32_t* flag = reinterpret_cast<int32_t*>(L.sort.keys[0]);
  int32_t* u = reinterpret_cast<int32_t*>(L.sort.keys[1]);
  int32_t* upos = reinterpret_cast<int32_t*>(L.sort.vals[0]);
  HG_TRY(launch("run_flags", run_flags, dim3(grid_for(E)), dim3(256), 0, s, col, ptr, rows, E, flag));
  HG_TRY(launch("run_row_starts", run_row_starts, dim3(grid_for(rows)), dim3(256), 0, s, ptr, rows, flag));
  HG_TRY(exclusive_scan(flag, u, E, L.sort.scan_scratch, s));
  HG_TRY(launch("run_write", run_write, dim3(grid_for(E / 4 + 1)), dim3(256), 0, s, (const int32_t*)u, col, ptr, rows,
                map, ucol, upos));
  return launch("run_finish", run_finish, dim3(grid_for(std::max(E, rows + 1))), dim3(256), 0, s, (const int32_t*)u,
                (const int32_t*)upos, ptr, rows, ucnt, uptr);
}

// ofs = exclusive scan of the chunk counts of the rows above the hub degree, row = the row of each chunk.
static hg_status chunk_table(const int32_t* ptr, int64_t rows, int32_t* ofs, int32_t* row, GraphLayout& L,
                             cudaStream_t s) {
  HG_TRY(launch("chunk_counts", chunk_counts, dim3(grid_for(rows)), dim3(256), 0, s, ptr, rows, L.cnt));
  HG_TRY(exclusive_scan(L.cnt, ofs, rows, L.sort.scan_scratch, s));
  return launch("chunk_fill", chunk_fill, dim3(grid_for(rows)), dim3(256), 0, s, (const int32_t*)ofs, rows, row);
}

}  // namespace hg

using namespace hg;

extern "C" hg_status hg_graph_workspace_size(int64_t num_edges, const int64_t* type_offsets,
                                             int32_t num_types, const hg_rel_desc* rels,
                                             int32_t num_rels, size_t* bytes) {
  clear_error();
  HG_REQUIRE(bytes != nullptr, "bytes must be non-null");
  HG_REQUIRE(num_edges >= 0, "num_edges must be >= 0");
  if (num_edges >= (int64_t(1) << 31)) {
    set_error("num_edges >= 2^31 is not supported");
    return HG_ERR_UNSUPPORTED;
  }
  GraphMeta m;
  HG_TRY(make_meta(type_offsets, num_types, rels, num_rels, &m));
  GraphLayout L;
  *bytes = carve_graph(nullptr, num_edges, m.row_base[num_rels], m.csc_base[num_rels], m.type_off[m.num_types], &L);
  return HG_OK;
}

extern "C" hg_status hg_build_csr(const int32_t* src, const int32_t* dst, const int32_t* rel,
                                  int64_t num_edges, const int64_t* type_offsets, int32_t num_types,
                                  const hg_rel_desc* rels, int32_t num_rels, void* workspace,
                                  size_t workspace_bytes, hg_stream stream, hg_graph** out) {
  clear_error();
  HG_TRY(device_guard());
  HG_REQUIRE(out != nullptr, "out must be non-null");
  *out = nullptr;
  HG_REQUIRE(num_edges >= 0, "num_edges must be >= 0");
  if (num_edges >= (int64_t(1) << 31)) {
    set_error("num_edges >= 2^31 is not supported");
    return HG_ERR_UNSUPPORTED;
  }
  HG_REQUIRE(num_edges == 0 || (src && dst && rel), "src, dst and rel must be non-null");
  HG_REQUIRE(workspace != nullptr, "workspace must be non-null");
  HG_REQUIRE(((uintptr_t)workspace & 255) == 0, "workspace must be 256-byte aligned");
  GraphMeta m;
  HG_TRY(make_meta(type_offsets, num_types, rels, num_rels, &m));
  const int64_t E = num_edges, rows = m.row_base[num_rels], crows = m.csc_base[num_rels];
  GraphLayout L;
  const int64_t N = m.type_off[num_types];
  const size_t need = carve_graph(nullptr, E, rows, crows, N, &L);
  if (workspace_bytes < need) {
    set_error("workspace has %zu bytes, %zu needed", workspace_bytes, need);
    return HG_ERR_WORKSPACE;
  }
  carve_graph(workspace, E, rows, crows, N, &L);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);

  const unsigned g = grid_for(E + 1);
  int res = 0;
  if (E == 0) {
    HG_CUDA(cudaMemsetAsync(L.csr_ptr, 0, (rows + 1) * sizeof(int32_t), s));
    HG_CUDA(cudaMemsetAsync(L.csc_ptr, 0, (crows + 1) * sizeof(int32_t), s));
    HG_CUDA(cudaMemsetAsync(L.node_ptr, 0, (N + 1) * sizeof(int32_t), s));
    HG_CUDA(cudaMemsetAsync(L.agg_ptr, 0, (rows + 1) * sizeof(int32_t), s));
    HG_CUDA(cudaMemsetAsync(L.bagg_ptr, 0, (N + 1) * sizeof(int32_t), s));
    HG_CUDA(cudaMemsetAsync(L.invalid, 0, sizeof(int32_t), s));
  } else {
    // CSR by (destination row, source, edge id): a stable sort by source, then by row
    HG_TRY(launch("edge_keys", edge_keys, dim3(g), dim3(256), 0, s, src, dst, rel, E, m, rows, L.sort.keys[0],
                  L.sort.ckeys));
    int r1 = 0;
    HG_TRY(radix_sort(L.sort, E, bit_width((uint64_t)N), (const uint32_t*)L.sort.keys[0], (const uint32_t*)nullptr,
                      (const uint32_t*)L.sort.ckeys, 0, s, &r1));
    // the last pass writes the edge ids and source ids straight into csr_eid and csr_col
    HG_TRY(radix_sort(L.sort, E, bit_width((uint64_t)rows), (const uint32_t*)L.sort.vals2[r1],
                      (const uint32_t*)L.sort.vals[r1], (const uint32_t*)L.sort.keys[r1], r1, s, &res,
                      (uint32_t*)L.csr_eid, (uint32_t*)L.csr_col));
    HG_TRY(launch("row_ptr_from_keys", row_ptr_from_keys, dim3(g), dim3(256), 0, s, (const uint32_t*)L.sort.keys[res],
                  E, rows, L.csr_ptr, L.invalid));
    // CSC by (source row, destination, edge id): the CSR order sorted stably by source row; the last
    // pass writes the edge ids and destination ids straight into csc_eid and csc_col
    const int r2 = res;
    HG_TRY(launch("csc_keys_from_csr", csc_keys_from_csr, dim3(g), dim3(256), 0, s, (const uint32_t*)L.sort.keys[r2],
                  (const uint32_t*)L.csr_col, E, (const int32_t*)L.csr_ptr, rows, crows, m, L.sort.ckeys,
                  L.sort.keys[r2]));
    HG_TRY(radix_sort(L.sort, E, bit_width((uint64_t)crows), (const uint32_t*)L.sort.ckeys,
                      (const uint32_t*)L.csr_eid, (const uint32_t*)L.sort.keys[r2], r2, s, &res,
                      (uint32_t*)L.csc_eid, (uint32_t*)L.csc_col));
    HG_TRY(launch("row_ptr_from_keys", row_ptr_from_keys, dim3(g), dim3(256), 0, s, (const uint32_t*)L.sort.keys[res],
                  E, crows, L.csc_ptr, (int32_t*)nullptr));
    // node-major rows: out-degree per node over its relations, their scan, then the edges
    HG_TRY(launch("node_out_counts", node_out_counts, dim3(grid_for(N)), dim3(256), 0, s, (const int32_t*)L.csc_ptr,
                  m, L.cnt));
    HG_TRY(exclusive_scan(L.cnt, L.node_ptr, N, L.sort.scan_scratch, s));
    HG_TRY(launch("csc_finish", csc_finish, dim3(g), dim3(256), 0, s, (const uint32_t*)L.sort.keys[res],
                  (const int32_t*)L.csc_col, (const int32_t*)L.csc_ptr, crows, m, (const int32_t*)L.csr_ptr,
                  (const int32_t*)L.node_ptr, L.csc_coef, L.node_col));
  }
  // non-empty CSR rows (the rows the mean layer stores) and their compact numbering
  HG_TRY(launch("nonempty_flags", nonempty_flags, dim3(grid_for(rows)), dim3(256), 0, s, (const int32_t*)L.csr_ptr,
                rows, L.cnt));
  HG_TRY(exclusive_scan(L.cnt, L.mrow, rows, L.sort.scan_scratch, s));
  HG_TRY(launch("compact_bases", compact_bases, dim3(1), dim3(32), 0, s, (const int32_t*)L.mrow, m, L.mbase));
  HG_TRY(launch("compact_rows", compact_rows, dim3(grid_for(rows)), dim3(256), 0, s, (const int32_t*)L.cnt, rows,
                L.mrow, L.mlist));
  if (E > 0) {
    // parallel edges coalesced into (column, multiplicity) runs, in both aggregation orders; the
    // backward runs name the compact row of the dMs row they read
    HG_TRY(coalesce_runs(L.csr_col, L.csr_ptr, rows, E, nullptr, L, L.agg_col, L.agg_cnt, L.agg_ptr, s));
    HG_TRY(coalesce_runs(L.node_col, L.node_ptr, N, E, L.mrow, L, L.bagg_col, L.bagg_cnt, L.bagg_ptr, s));
  }
  // the fused layer's long rows (more than kFuseRuns runs) and their compact slots
  HG_TRY(launch("long_flags", long_flags, dim3(grid_for(rows)), dim3(256), 0, s, (const int32_t*)L.agg_ptr, rows,
                L.cnt));
  HG_TRY(exclusive_scan(L.cnt, L.long_ofs, rows, L.sort.scan_scratch, s));
  HG_TRY(launch("compact_list", compact_list, dim3(grid_for(rows)), dim3(256), 0, s, (const int32_t*)L.cnt,
                (const int32_t*)L.long_ofs, rows, L.long_list));
  // node order of the forward projection, per type: sorted by relation mask, and each tile's mask
  int64_t tile_base[kMaxTypes + 1] = {0};
  for (int t = 0; t < m.num_types; ++t) {
    const int64_t n = m.type_off[t + 1] - m.type_off[t];
    tile_base[t + 1] = tile_base[t] + ceil_div(n, kProjTileRows);
    if (n == 0) continue;
    TypeRels tr{};
    for (int r = 0; r < num_rels; ++r)
      if (m.rel_dst[r] == t) tr.row0[tr.n++] = m.row_base[r];
    const int nblk = (int)order_blocks(n);
    const int64_t nh = ((int64_t)1 << tr.n) * nblk;
    HG_TRY(launch("order_hist", order_hist, dim3(nblk), dim3(256), 0, s, (const int32_t*)L.csr_ptr, tr, n, nblk,
                  L.ohist));
    HG_TRY(exclusive_scan(L.ohist, L.oofs, nh, L.sort.scan_scratch, s));
    int32_t* perm = L.nperm + m.type_off[t];
    HG_TRY(launch("order_scatter", order_scatter, dim3(nblk), dim3(256), 0, s, (const int32_t*)L.csr_ptr, tr, n,
                  nblk, (const int32_t*)L.oofs, perm));
    const int64_t tiles = tile_base[t + 1] - tile_base[t];
    HG_TRY(launch("order_tiles", order_tiles, dim3((unsigned)ceil_div(tiles * 32, 256)), dim3(256), 0, s,
                  (const int32_t*)L.csr_ptr, tr, n, (const int32_t*)perm, tiles, L.tmask + tile_base[t]));
  }
  // chunk tables over runs for rows above the hub degree (mean and attention layers)
  HG_TRY(chunk_table(L.agg_ptr, rows, L.agg_chunk_ofs, L.agg_chunk_row, L, s));
  HG_TRY(chunk_table(L.bagg_ptr, N, L.bagg_chunk_ofs, L.bagg_chunk_row, L, s));

  hg_graph* gh = new hg_graph{};
  gh->meta = m;
  gh->num_edges = E;
  gh->csr_rows = rows;
  gh->csc_rows = crows;
  gh->chunk_cap_csr = chunk_cap(E);
  gh->chunk_cap_node = chunk_cap(E);
  gh->stream = s;
  gh->csr_ptr = L.csr_ptr;
  gh->csr_col = L.csr_col;
  gh->csr_eid = L.csr_eid;
  gh->csc_ptr = L.csc_ptr;
  gh->csc_col = L.csc_col;
  gh->csc_eid = L.csc_eid;
  gh->csc_coef = L.csc_coef;
  gh->node_ptr = L.node_ptr;
  gh->node_col = L.node_col;
  gh->agg_ptr = L.agg_ptr;
  gh->agg_col = L.agg_col;
  gh->agg_cnt = L.agg_cnt;
  gh->agg_chunk_ofs = L.agg_chunk_ofs;
  gh->agg_chunk_row = L.agg_chunk_row;
  gh->bagg_ptr = L.bagg_ptr;
  gh->bagg_col = L.bagg_col;
  gh->bagg_cnt = L.bagg_cnt;
  gh->bagg_chunk_ofs = L.bagg_chunk_ofs;
  gh->bagg_chunk_row = L.bagg_chunk_row;
  gh->mrow = L.mrow;
  gh->mlist = L.mlist;
  gh->mbase = L.mbase;
  gh->nperm = L.nperm;
  gh->tmask = L.tmask;
  gh->long_ofs = L.long_ofs;
  gh->long_list = L.long_list;
  gh->long_cap = long_cap(E);
  for (int t = 0; t <= kMaxTypes; ++t) gh->tile_base[t] = tile_base[std::min(t, m.num_types)];
  gh->invalid_count = L.invalid;
  *out = gh;
  return HG_OK;
}

extern "C" hg_status hg_graph_node_order(const hg_graph* graph, int32_t type, hg_node_order* out) {
  clear_error();
  HG_REQUIRE(graph != nullptr && out != nullptr, "graph and out must be non-null");
  const GraphMeta& m = graph->meta;
  HG_REQUIRE(type >= 0 && type < m.num_types, "type %d out of range", type);
  out->n = m.type_off[type + 1] - m.type_off[type];
  out->tiles = graph->tile_base[type + 1] - graph->tile_base[type];
  out->tile_rows = kProjTileRows;
  out->perm = graph->nperm + m.type_off[type];
  out->tile_mask = graph->tmask + graph->tile_base[type];
  return HG_OK;
}

extern "C" hg_status hg_graph_destroy(hg_graph* graph) {
  delete graph;
  return HG_OK;
}

extern "C" hg_status hg_graph_check(const hg_graph* graph, int64_t* num_invalid_edges) {
  clear_error();
  HG_TRY(device_guard());
  HG_REQUIRE(graph != nullptr, "graph must be non-null");
  int32_t bad = 0;
  HG_CUDA(cudaMemcpyAsync(&bad, graph->invalid_count, sizeof(int32_t), cudaMemcpyDeviceToHost,
                          graph->stream));
  HG_CUDA(cudaStreamSynchronize(graph->stream));
  if (num_invalid_edges) *num_invalid_edges = bad;
  if (bad != 0) {
    set_error("%d edges were dropped (id out of range, relation out of range, or endpoint types "
              "that do not match the relation)", bad);
    return HG_ERR_DEVICE_CHECK;
  }
  return HG_OK;
}

extern "C" hg_status hg_graph_view(const hg_graph* graph, int32_t rel, hg_graph_arrays* out) {
  clear_error();
  HG_REQUIRE(graph != nullptr && out != nullptr, "graph and out must be non-null");
  const GraphMeta& m = graph->meta;
  HG_REQUIRE(rel >= 0 && rel < m.num_rels, "relation %d out of range", rel);
  out->n_dst = m.row_base[rel + 1] - m.row_base[rel];
  out->n_src = m.csc_base[rel + 1] - m.csc_base[rel];
  out->num_edges = graph->num_edges;
  out->row_ptr = graph->csr_ptr + m.row_base[rel];
  out->col = graph->csr_col;
  out->eid = graph->csr_eid;
  out->csc_ptr = graph->csc_ptr + m.csc_base[rel];
  out->csc_col = graph->csc_col;
  out->csc_eid = graph->csc_eid;
  out->csc_coef = graph->csc_coef;
  return HG_OK;
}
