// Overlapping subgraph construction (Section 3.1, Eq. 4-5; the construction loop of Algorithm 1).
//
// One subgraph k of K from a global graph, all on the device, integer arithmetic only:
//   degrees ........... incident edges per node (both directions), integer atomics;
//   incidence lists ... the degrees of every node's neighbours, one slot per incident edge (slots
//                       claimed by atomics: the order inside a list is arbitrary, and nothing
//                       below depends on it);
//   h-index ........... per node the largest h with at least h neighbour degrees >= h: short lists
//                       by warp ballots, longer ones by a bounded binary search on the count
//                       function (warp per node; a CTA per node above kBigList);
//   candidates (Eq. 4)  node flags from an edge-parallel pass (v -> u, u in V_k, v outside);
//   selection ......... the M smallest sampling keys among the candidates with h <= theta, by a
//                       four-pass radix select on the device (ties by id through a scan);
//   V~_k (Eq. 5) ...... membership scan -> local ids; stable compaction of the induced edges.
// The base partition and the sampling keys use the SplitMix64 output function, written here from
// its published definition.
#include <algorithm>

#include "hg_internal.cuh"

namespace hg {
namespace {

constexpr int kBigList = 4096;  // incidence lists longer than this get a CTA of their own

struct TypeOffsets {
  int64_t v[kMaxTypes + 1];
};

__device__ __forceinline__ uint64_t splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}
__device__ __forceinline__ int part_of(int64_t v, uint64_t seed, int K) {
  return (int)(splitmix64(seed ^ (uint64_t)v) % (uint64_t)K);
}
__device__ __forceinline__ uint32_t sample_key(int64_t v, int k, uint64_t seed) {
  return (uint32_t)(splitmix64(seed ^ ((uint64_t)k << 40) ^ (uint64_t)v) >> 32);
}
__device__ __forceinline__ bool edge_ok(int32_t s, int32_t t, int64_t N) {
  return s >= 0 && s < N && t >= 0 && t < N;
}

// Warp-aggregated increment of ctr[key] by the lanes holding the same key (key < 0: none);
// returns this lane's slot: the counter's old value plus its rank among those lanes.  Hub nodes
// recur within a warp's edges, so one atomic serves all of a hub's occurrences.
__device__ __forceinline__ int aggregated_claim(int32_t* ctr, int key) {
  const int lane = threadIdx.x & 31;
  const unsigned peers = __match_any_sync(0xffffffffu, key);
  const int leader = __ffs(peers) - 1;
  int base = 0;
  if (key >= 0 && lane == leader) base = atomicAdd(&ctr[key], __popc(peers));
  base = __shfl_sync(0xffffffffu, base, leader);
  return base + __popc(peers & ((1u << lane) - 1u));
}

// (the loops run whole warps together: lanes past the end take key -1)
__global__ void ob_degrees(const int32_t* __restrict__ src, const int32_t* __restrict__ dst, int64_t E, int64_t N,
                           int32_t* __restrict__ deg) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); e0 < E; e0 += stride) {
    const int64_t e = e0 + (threadIdx.x & 31);
    int32_t s = -1, t = -1;
    if (e < E) {
      s = src[e];
      t = dst[e];
      if (!edge_ok(s, t, N)) s = t = -1;
    }
    aggregated_claim(deg, s);
    aggregated_claim(deg, t);
  }
}

// nbr[ofs[v] + slot] = degree of the other endpoint, for every incident edge of v
__global__ void ob_fill_lists(const int32_t* __restrict__ src, const int32_t* __restrict__ dst, int64_t E, int64_t N,
                              const int32_t* __restrict__ deg, const int32_t* __restrict__ ofs,
                              int32_t* __restrict__ fill, int32_t* __restrict__ nbr) {
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t e0 = (int64_t)blockIdx.x * blockDim.x + (threadIdx.x & ~31); e0 < E; e0 += stride) {
    const int64_t e = e0 + (threadIdx.x & 31);
    int32_t s = -1, t = -1;
    if (e < E) {
      s = src[e];
      t = dst[e];
      if (!edge_ok(s, t, N)) s = t = -1;
    }
    const int ps = aggregated_claim(fill, s);
    const int pt = aggregated_claim(fill, t);
    if (s >= 0) {
      nbr[ofs[s] + ps] = deg[t];
      nbr[ofs[t] + pt] = deg[s];
    }
  }
}

// h-index from one incidence list nb[0 .. n): the largest h with #{i : nb[i] >= h} >= h.
// Warp version (all 32 lanes call it with the same list).
__device__ int warp_h_index(const int32_t* __restrict__ nb, int n) {
  const int lane = threadIdx.x & 31;
  if (n <= 32) {  // ballots: count(h) = lanes with nb >= h, h = 1 .. n
    const int x = lane < n ? nb[lane] : 0;
    int h = 0;
    for (int c = 1; c <= n; ++c)
      if (__popc(__ballot_sync(0xffffffffu, x >= c)) >= c) h = c;
    return h;
  }
  // count(h) is non-increasing in h: binary search for the last h in [0, n] with count(h) >= h
  int lo = 0, hi = n;  // count(lo) >= lo holds; the answer lies in [lo, hi]
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    int c = 0;
    for (int i = lane; i < n; i += 32) c += nb[i] >= mid;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) c += __shfl_xor_sync(0xffffffffu, c, o);
    if (c >= mid) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// one warp per node (grid-stride); lists longer than kBigList are left to ob_h_big
__global__ void ob_h_small(const int32_t* __restrict__ ofs, const int32_t* __restrict__ nbr, int64_t N,
                           int32_t* __restrict__ h) {
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t v = (int64_t)blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5); v < N; v += warps) {
    const int n = ofs[v + 1] - ofs[v];
    if (n > kBigList) continue;
    const int r = warp_h_index(nbr + ofs[v], n);
    if ((threadIdx.x & 31) == 0) h[v] = r;
  }
}

// One CTA per node with a list longer than kBigList: the CTAs stride over tiles of kBigThreads
// nodes, every thread testing one node, and take the tile's long lists one after another.
// The h-index is the largest h with S(h) = #{degrees >= h} >= h.  Each pass bins the degrees over
// [lo, hi] into at most kCap bins of width w (degrees above hi in the last bin, below lo dropped);
// the suffix sums give S at every bin start, the largest bin start still satisfying S >= h brackets
// the answer, and the next pass refines that bin.  Two passes cover lists of millions of entries
// (multi-edges between hubs give hubs h-indices in the thousands).  The lowest bins, where most of
// a hub's neighbours fall, are counted in registers before they reach shared memory.
constexpr int kCap = 8192;
constexpr int kRegBins = 8;
constexpr int kBigThreads = 1024;
__global__ void __launch_bounds__(kBigThreads) ob_h_big(const int32_t* __restrict__ ofs, const int32_t* __restrict__ nbr,
                                                        int64_t N, int32_t* __restrict__ h) {
  __shared__ int hist[kCap];
  __shared__ int part[kBigThreads / 32];
  __shared__ int best_s;
  __shared__ int64_t tile_big[kBigThreads];  // the tile's nodes with long lists
  __shared__ int tile_nbig;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  for (int64_t t0 = (int64_t)blockIdx.x * kBigThreads; t0 < N; t0 += (int64_t)gridDim.x * kBigThreads) {
    if (threadIdx.x == 0) tile_nbig = 0;
    __syncthreads();
    {
      const int64_t u = t0 + threadIdx.x;
      if (u < N && ofs[u + 1] - ofs[u] > kBigList) tile_big[atomicAdd(&tile_nbig, 1)] = u;
    }
    __syncthreads();
    const int nbig = tile_nbig;
    for (int ib = 0; ib < nbig; ++ib) {
      const int64_t v = tile_big[ib];
      const int n = ofs[v + 1] - ofs[v];
      const int32_t* nb = nbr + ofs[v];
      int lo = 0, hi = n;  // S(lo) >= lo holds; the answer lies in [lo, hi]
      while (true) {
        const int span = hi - lo + 1;
        int lw = 0;  // bin width 2^lw, the smallest giving at most kCap bins
        while (((span + (1 << lw) - 1) >> lw) > kCap) ++lw;
        const int w = 1 << lw;
        const int nbins = (span + w - 1) >> lw;
        for (int i = threadIdx.x; i < nbins; i += blockDim.x) hist[i] = 0;
        if (threadIdx.x == 0) best_s = 0;
        __syncthreads();
        int reg[kRegBins] = {0, 0, 0, 0, 0, 0, 0, 0};
        auto count = [&](int d) {
          if (d < lo) return;
          const int j = min((d - lo) >> lw, nbins - 1);
          if (j < kRegBins) {
  #pragma unroll
            for (int q = 0; q < kRegBins; ++q) reg[q] += j == q;
          } else {
            atomicAdd(&hist[j], 1);
          }
        };
        int i = threadIdx.x;
        for (; i + 3 * (int)blockDim.x < n; i += 4 * blockDim.x) {  // four loads in flight
          const int d0 = nb[i], d1 = nb[i + blockDim.x], d2 = nb[i + 2 * blockDim.x], d3 = nb[i + 3 * blockDim.x];
          count(d0);
          count(d1);
          count(d2);
          count(d3);
        }
        for (; i < n; i += blockDim.x) count(nb[i]);
  #pragma unroll
        for (int q = 0; q < kRegBins; ++q) {
          int t = reg[q];
  #pragma unroll
          for (int o = 16; o > 0; o >>= 1) t += __shfl_xor_sync(0xffffffffu, t, o);
          if (lane == 0 && t && q < nbins) atomicAdd(&hist[q], t);
        }
        __syncthreads();
        // suffix sums: thread j owns bins [blo, bhi) counted from the top
        const int per = (nbins + blockDim.x - 1) / blockDim.x;
        const int bhi = nbins - threadIdx.x * per, blo = max(0, bhi - per);
        int own = 0;
        for (int b = blo; b < bhi; ++b) own += hist[b];
        int incl = own;
  #pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
          const int y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        if (lane == 31) part[warp] = incl;
        __syncthreads();
        int run = incl - own;  // entries in higher bins of lower-numbered threads
  #pragma unroll
        for (int ww = 0; ww < kBigThreads / 32; ++ww) run += ww < warp ? part[ww] : 0;
        int found = -1;
        for (int b = bhi - 1; b >= blo; --b) {  // S(lo + b w) from the top of the range down
          run += hist[b];
          if (run >= lo + b * w) {
            found = b;
            break;
          }
        }
        if (found >= 0) atomicMax(&best_s, found);
        __syncthreads();
        const int j = best_s;  // bin 0 always qualifies (S(lo) >= lo)
        __syncthreads();
        if (w == 1) {
          if (threadIdx.x == 0) h[v] = lo + j;
          break;
        }
        const int nlo = lo + j * w;
        hi = min(hi, nlo + w - 1);
        lo = nlo;
      }
      __syncthreads();
    }
    __syncthreads();  // tile_big and tile_nbig are rewritten by the next tile
  }
}

// cand[v] = 1 for v outside V_k with an edge v -> u, u in V_k (Eq. 4)
__global__ void ob_candidates(const int32_t* __restrict__ src, const int32_t* __restrict__ dst, int64_t E, int64_t N,
                              uint64_t part_seed, int K, int k, int32_t* __restrict__ cand) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < E; e += (int64_t)gridDim.x * blockDim.x) {
    const int32_t s = src[e], t = dst[e];
    if (!edge_ok(s, t, N)) continue;
    if (part_of(t, part_seed, K) == k && part_of(s, part_seed, K) != k && cand[s] == 0) atomicOr(&cand[s], 1);
  }
}

// Selection state of the radix select, in device memory.
struct SelState {
  unsigned long long count_c, count_elig, count_base;  // |C_k|, |C'_k|, |V_k|
  unsigned long long take;                              // M' = min(M, |C'_k|)
  uint32_t prefix, mask;                                // key bits fixed so far
  long long rank;                                       // 0-based rank of the last taken key among the matching keys
};

// elig[v] = cand[v] && h[v] <= theta; counts of C_k, C'_k and V_k
__global__ void ob_eligible(const int32_t* __restrict__ cand, const int32_t* __restrict__ h, int64_t N, int theta,
                            uint64_t part_seed, int K, int k, int32_t* __restrict__ elig, SelState* st) {
  unsigned long long c = 0, ce = 0, cb = 0;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < N; v += (int64_t)gridDim.x * blockDim.x) {
    const int e = cand[v] && h[v] <= theta;
    elig[v] = e;
    c += cand[v] != 0;
    ce += e;
    cb += part_of(v, part_seed, K) == k;
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    c += __shfl_xor_sync(0xffffffffu, c, o);
    ce += __shfl_xor_sync(0xffffffffu, ce, o);
    cb += __shfl_xor_sync(0xffffffffu, cb, o);
  }
  if ((threadIdx.x & 31) == 0) {
    atomicAdd(&st->count_c, c);
    atomicAdd(&st->count_elig, ce);
    atomicAdd(&st->count_base, cb);
  }
}

// histogram of key digit (key >> shift) & 255 over the eligible nodes whose fixed key bits match
__global__ void ob_key_hist(const int32_t* __restrict__ elig, int64_t N, int k, uint64_t sample_seed, int shift,
                            const SelState* __restrict__ st, unsigned int* __restrict__ hist) {
  __shared__ unsigned int hs[256];
  hs[threadIdx.x] = 0;
  __syncthreads();
  const uint32_t prefix = st->prefix, mask = st->mask;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < N; v += (int64_t)gridDim.x * blockDim.x) {
    if (!elig[v]) continue;
    const uint32_t key = sample_key(v, k, sample_seed);
    if ((key & mask) == prefix) atomicAdd(&hs[(key >> shift) & 255u], 1u);
  }
  __syncthreads();
  if (hs[threadIdx.x]) atomicAdd(&hist[threadIdx.x], hs[threadIdx.x]);
}

// one thread: fixes the next 8 key bits from the histogram (first pass: also M' and the rank)
__global__ void ob_key_select(unsigned int* __restrict__ hist, int shift, long long M, SelState* st) {
  if (shift == 24) {
    st->take = (unsigned long long)min((long long)st->count_elig, M);
    st->rank = (long long)st->take - 1;  // the last key taken, 0-based
  }
  if (st->take > 0) {
    long long r = st->rank;
    int digit = 255;
    for (int b = 0; b < 256; ++b) {
      if (r < (long long)hist[b]) {
        digit = b;
        break;
      }
      r -= hist[b];
    }
    st->rank = r;
    st->prefix |= (uint32_t)digit << shift;
    st->mask |= 255u << shift;
  }
  for (int b = 0; b < 256; ++b) hist[b] = 0;
}

// eq[v] = eligible with key == the selected threshold key (for the tie ranks)
__global__ void ob_ties(const int32_t* __restrict__ elig, int64_t N, int k, uint64_t sample_seed,
                        const SelState* __restrict__ st, int32_t* __restrict__ eq) {
  const bool any = st->take > 0;
  const uint32_t T = st->prefix;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < N; v += (int64_t)gridDim.x * blockDim.x)
    eq[v] = any && elig[v] && sample_key(v, k, sample_seed) == T;
}

// member[v] = v in V_k or selected (key below the threshold, or equal with tie rank <= rank)
__global__ void ob_members(const int32_t* __restrict__ elig, const int32_t* __restrict__ eq_rank, int64_t N, int K,
                           int k, uint64_t part_seed, uint64_t sample_seed, const SelState* __restrict__ st,
                           int32_t* __restrict__ member) {
  const bool any = st->take > 0;
  const uint32_t T = st->prefix;
  const long long rank = st->rank;
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < N; v += (int64_t)gridDim.x * blockDim.x) {
    bool in = part_of(v, part_seed, K) == k;
    if (!in && any && elig[v]) {
      const uint32_t key = sample_key(v, k, sample_seed);
      in = key < T || (key == T && (long long)eq_rank[v] <= rank);  // eq_rank: exclusive scan of ties
    }
    member[v] = in;
  }
}

__global__ void ob_gids(const int32_t* __restrict__ mscan, int64_t N, int64_t* __restrict__ gid_out) {
  for (int64_t v = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; v < N; v += (int64_t)gridDim.x * blockDim.x)
    if (mscan[v + 1] > mscan[v]) gid_out[mscan[v]] = v;
}

// keep[e] = both endpoints in V~_k
__global__ void ob_keep(const int32_t* __restrict__ src, const int32_t* __restrict__ dst, int64_t E, int64_t N,
                        const int32_t* __restrict__ mscan, int32_t* __restrict__ keep) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < E; e += (int64_t)gridDim.x * blockDim.x) {
    const int32_t s = src[e], t = dst[e];
    keep[e] = edge_ok(s, t, N) && mscan[s + 1] > mscan[s] && mscan[t + 1] > mscan[t];
  }
}

__global__ void ob_compact(const int32_t* __restrict__ src, const int32_t* __restrict__ dst,
                           const int32_t* __restrict__ rel, int64_t E, const int32_t* __restrict__ mscan,
                           const int32_t* __restrict__ kscan, int32_t* __restrict__ src_out,
                           int32_t* __restrict__ dst_out, int32_t* __restrict__ rel_out, int32_t* __restrict__ eid_out) {
  for (int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; e < E; e += (int64_t)gridDim.x * blockDim.x) {
    if (kscan[e + 1] == kscan[e]) continue;
    const int32_t p = kscan[e];
    src_out[p] = mscan[src[e]];
    dst_out[p] = mscan[dst[e]];
    rel_out[p] = rel[e];
    eid_out[p] = (int32_t)e;
  }
}

// counts_out and the local type boundaries
__global__ void ob_finish(const int32_t* __restrict__ mscan, const int32_t* __restrict__ kscan, int64_t N, int64_t E,
                          TypeOffsets toff, int num_types, const SelState* __restrict__ st,
                          int64_t* __restrict__ type_offsets_out, int64_t* __restrict__ counts_out) {
  if (threadIdx.x == 0) {
    counts_out[0] = mscan[N];
    counts_out[1] = (int64_t)st->count_base;
    counts_out[2] = (int64_t)st->take;
    counts_out[3] = kscan[E];
    counts_out[4] = (int64_t)st->count_c;
    counts_out[5] = (int64_t)st->count_elig;
  }
  if (threadIdx.x <= num_types) type_offsets_out[threadIdx.x] = mscan[toff.v[threadIdx.x]];
}

static unsigned grid_of(int64_t n, int threads = 256) {
  return (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(n, threads), 152 * 16));
}

struct BuildLayout {
  int32_t *deg, *ofs, *fill, *nbr, *h, *cand, *elig, *eq, *member, *keep;
  unsigned int* hist;
  SelState* st;
  void* scan;
};

static size_t carve_build(void* ws, int64_t N, int64_t E, BuildLayout* L) {
  Carve c(ws);
  const int64_t Na = std::max<int64_t>(N, 1), Ea = std::max<int64_t>(E, 1);
  L->deg = c.take<int32_t>(Na);
  L->ofs = c.take<int32_t>(Na + 1);
  L->fill = c.take<int32_t>(Na);
  L->nbr = c.take<int32_t>(2 * Ea);
  L->h = c.take<int32_t>(Na);
  L->cand = c.take<int32_t>(Na);
  L->elig = c.take<int32_t>(Na);
  L->eq = c.take<int32_t>(Na + 1);
  L->member = c.take<int32_t>(Na + 1);
  L->keep = c.take<int32_t>(Ea + 1);
  L->hist = c.take<unsigned int>(256);
  L->st = c.take<SelState>(1);
  L->scan = c.take<char>(scan_scratch_bytes(std::max(Na, Ea) + 1));
  return c.used;
}

}  // namespace
}  // namespace hg

using namespace hg;

extern "C" hg_status hg_overlap_build_workspace_size(int64_t num_nodes, int64_t num_edges, size_t* bytes) {
  clear_error();
  HG_REQUIRE(bytes != nullptr && num_nodes >= 0 && num_edges >= 0, "bytes must be non-null and sizes >= 0");
  if (num_nodes >= (int64_t(1) << 31) || num_edges >= (int64_t(1) << 30)) {
    set_error("num_nodes must be < 2^31 and num_edges < 2^30");
    return HG_ERR_UNSUPPORTED;
  }
  BuildLayout L;
  *bytes = carve_build(nullptr, num_nodes, num_edges, &L);
  return HG_OK;
}

extern "C" hg_status hg_overlap_build(const int32_t* src, const int32_t* dst, const int32_t* rel, int64_t num_edges,
                                      int64_t num_nodes, const int64_t* type_offsets, int32_t num_types, int32_t K,
                                      int32_t k, int32_t theta, int64_t M, uint64_t part_seed, uint64_t sample_seed,
                                      int64_t* gid_out, int32_t* src_out, int32_t* dst_out, int32_t* rel_out,
                                      int32_t* eid_out, int64_t* type_offsets_out, int32_t* h_out,
                                      int64_t* counts_out, void* workspace, size_t workspace_bytes,
                                      hg_stream stream) {
  clear_error();
  HG_TRY(device_guard());
  size_t need = 0;
  HG_TRY(hg_overlap_build_workspace_size(num_nodes, num_edges, &need));
  HG_REQUIRE(K >= 1 && k >= 0 && k < K, "need K >= 1 and 0 <= k < K");
  HG_REQUIRE(theta >= 0 && M >= 0, "theta and M must be >= 0");
  HG_REQUIRE(type_offsets != nullptr && num_types >= 1 && num_types <= kMaxTypes, "bad type offsets");
  HG_REQUIRE(type_offsets[0] == 0 && type_offsets[num_types] == num_nodes, "type offsets must span [0, num_nodes)");
  for (int t = 0; t < num_types; ++t) HG_REQUIRE(type_offsets[t] <= type_offsets[t + 1], "type offsets must ascend");
  HG_REQUIRE(num_edges == 0 || (src && dst && rel && src_out && dst_out && rel_out && eid_out),
             "edge arrays must be non-null");
  HG_REQUIRE(num_nodes == 0 || gid_out, "gid_out must be non-null");
  HG_REQUIRE(type_offsets_out && counts_out && workspace, "type_offsets_out, counts_out, workspace must be non-null");
  HG_REQUIRE(((uintptr_t)workspace & 255) == 0, "workspace must be 256-byte aligned");
  if (workspace_bytes < need) {
    set_error("workspace has %zu bytes, %zu needed", workspace_bytes, need);
    return HG_ERR_WORKSPACE;
  }
  BuildLayout L;
  carve_build(workspace, num_nodes, num_edges, &L);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int64_t N = num_nodes, E = num_edges;
  int32_t* h = h_out ? h_out : L.h;
  TypeOffsets toff{};
  for (int t = 0; t <= num_types; ++t) toff.v[t] = type_offsets[t];

  HG_CUDA(cudaMemsetAsync(L.deg, 0, std::max<int64_t>(N, 1) * sizeof(int32_t), s));
  HG_CUDA(cudaMemsetAsync(L.fill, 0, std::max<int64_t>(N, 1) * sizeof(int32_t), s));
  HG_CUDA(cudaMemsetAsync(L.cand, 0, std::max<int64_t>(N, 1) * sizeof(int32_t), s));
  HG_CUDA(cudaMemsetAsync(L.hist, 0, 256 * sizeof(unsigned int), s));
  HG_CUDA(cudaMemsetAsync(L.st, 0, sizeof(SelState), s));
  // degrees, incidence lists of neighbour degrees, h-index
  if (E > 0)
    HG_TRY(launch("ob_degrees", ob_degrees, dim3(grid_of(E)), dim3(256), 0, s, src, dst, E, N, L.deg));
  HG_TRY(exclusive_scan(L.deg, L.ofs, N, L.scan, s));
  if (E > 0)
    HG_TRY(launch("ob_fill_lists", ob_fill_lists, dim3(grid_of(E)), dim3(256), 0, s, src, dst, E, N,
                  (const int32_t*)L.deg, (const int32_t*)L.ofs, L.fill, L.nbr));
  if (N > 0) {
    HG_TRY(launch("ob_h_small", ob_h_small, dim3(grid_of(32 * N)), dim3(256), 0, s, (const int32_t*)L.ofs,
                  (const int32_t*)L.nbr, N, h));
    HG_TRY(launch("ob_h_big", ob_h_big, dim3((unsigned)std::min<int64_t>(N, 152 * 2)), dim3(kBigThreads), 0, s,
                  (const int32_t*)L.ofs, (const int32_t*)L.nbr, N, h));
  }
  // candidates (Eq. 4), the h-index filter, the selection of the M smallest keys
  if (E > 0)
    HG_TRY(launch("ob_candidates", ob_candidates, dim3(grid_of(E)), dim3(256), 0, s, src, dst, E, N, part_seed, K, k,
                  L.cand));
  if (N > 0)
    HG_TRY(launch("ob_eligible", ob_eligible, dim3(grid_of(N)), dim3(256), 0, s, (const int32_t*)L.cand,
                  (const int32_t*)h, N, theta, part_seed, K, k, L.elig, L.st));
  for (int shift = 24; shift >= 0; shift -= 8) {
    if (N > 0)
      HG_TRY(launch("ob_key_hist", ob_key_hist, dim3(grid_of(N)), dim3(256), 0, s, (const int32_t*)L.elig, N, k,
                    sample_seed, shift, (const SelState*)L.st, L.hist));
    HG_TRY(launch("ob_key_select", ob_key_select, dim3(1), dim3(1), 0, s, L.hist, shift, (long long)M, L.st));
  }
  if (N > 0)
    HG_TRY(launch("ob_ties", ob_ties, dim3(grid_of(N)), dim3(256), 0, s, (const int32_t*)L.elig, N, k, sample_seed,
                  (const SelState*)L.st, L.eq));
  HG_TRY(exclusive_scan(L.eq, L.eq, N, L.scan, s));
  // V~_k (Eq. 5): membership, local ids, the induced edges
  if (N > 0)
    HG_TRY(launch("ob_members", ob_members, dim3(grid_of(N)), dim3(256), 0, s, (const int32_t*)L.elig,
                  (const int32_t*)L.eq, N, K, k, part_seed, sample_seed, (const SelState*)L.st, L.member));
  HG_TRY(exclusive_scan(L.member, L.member, N, L.scan, s));
  if (N > 0)
    HG_TRY(launch("ob_gids", ob_gids, dim3(grid_of(N)), dim3(256), 0, s, (const int32_t*)L.member, N, gid_out));
  if (E > 0)
    HG_TRY(launch("ob_keep", ob_keep, dim3(grid_of(E)), dim3(256), 0, s, src, dst, E, N, (const int32_t*)L.member,
                  L.keep));
  HG_TRY(exclusive_scan(L.keep, L.keep, E, L.scan, s));
  if (E > 0)
    HG_TRY(launch("ob_compact", ob_compact, dim3(grid_of(E)), dim3(256), 0, s, src, dst, rel, E,
                  (const int32_t*)L.member, (const int32_t*)L.keep, src_out, dst_out, rel_out, eid_out));
  return launch("ob_finish", ob_finish, dim3(1), dim3(32), 0, s, (const int32_t*)L.member, (const int32_t*)L.keep, N,
                E, toff, (int)num_types, (const SelState*)L.st, type_offsets_out, counts_out);
}
