// Per-relation mean aggregation (Eq. 10 with the mean as the aggregation operator) and its
// transpose for the backward pass.
//
// Forward:  M_r[j] = (1/deg_r(j)) * sum_{(i -> j) in r} H[i]          (CSR row j of relation r)
// Backward: dH[i]  = sum_r sum_{(i -> j) in r} dMs_r[j] + dY[i]
//           where dMs_r[j] = dM_r[j] / deg_r(j) is produced, already scaled, by the projection
//           backward kernel, and dY[i] is the residual-path gradient of Eq. 11.  The sum runs over
//           node i's row of the node-major out-edge list (its CSC rows of every relation leaving
//           its type, concatenated in relation order, each edge holding the dMs row it reads).
// M_r and dMs_r are stored for the non-empty CSR rows only, in the graph's compact order (a row
// without in-edges has M_r = 0 and is never stored, read or gathered; the projections read it as
// zeros), and the backward runs name those compact rows.
// Parallel edges (the same source, destination and relation) are summed once with their
// multiplicity: the rows read here are the build's runs (column, count), so each distinct
// neighbour row is gathered once per row and multiplied by its count (deg_r(j) is still the
// number of edges, the CSR row length).
//
// Mapping: the row kernels (agg_fwd_rows, agg_bwd_nodes) give a warp chunks of 16 consecutive
// rows, each lane owning d / 32 columns, and stream through the chunks' contiguous runs with eight
// gathered rows in flight (fp32 accumulation); chunks are claimed dynamically.  Rows above
// kHubDegree runs are split into kChunkEdges-run chunks: a whole CTA reduces one chunk (groups of
// d * sizeof(T) / 16 lanes interleave over the chunk's runs, gathering into shared memory by
// cp.async, then combine in group order) into an fp32 partial, runs of 64 partials are summed in
// order, and the row adds the run sums in order.  Every sum has a fixed order, so results are
// bitwise reproducible run to run.
#include <algorithm>

#include "layer_kernels.cuh"
#include "tc_util.cuh"

namespace hg {

template <typename T, int D>
struct AggShape {
  static constexpr int kVec = VecTraits<T>::kElems;  // elements per 16 bytes
  static constexpr int kRowVecs = D / kVec;          // 16-byte vectors per row
  static constexpr int G = kRowVecs < 32 ? kRowVecs : 32;
  static constexpr int V = kRowVecs / G;  // vectors per lane
  static constexpr int F = V * kVec;      // fp32 accumulators per lane
  static constexpr int kThreads = 256;
  static constexpr int kGroups = kThreads / G;
};

// Chunk partials are combined in two fixed-order levels: combine_chunk_partials sums every run of
// kPartRun consecutive chunks of a row into the run's first slot, and a row then adds its run
// sums in order (eight loads in flight).
constexpr int kPartRun = 64;

// Sums each run of kPartRun consecutive chunk partials of a row, in order, into the run's first
// slot (one block of d threads per run leader; grid-stride over the chunk list).
template <int D>
__global__ void __launch_bounds__(D) combine_chunk_partials(const int32_t* __restrict__ chunk_row,
                                                            const int32_t* __restrict__ chunk_ofs, int64_t rows,
                                                            float* __restrict__ partials) {
  const int nchunks = chunk_ofs[rows];
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x) {
    const int row = chunk_row[c];
    const int first = chunk_ofs[row];
    if ((c - first) % kPartRun != 0) continue;
    const int c1 = min(chunk_ofs[row + 1], c + kPartRun);
    if (c1 - c < 2) continue;
    const int k = threadIdx.x;
    float s = 0.f;
    int cc = c;
    for (; cc + 8 <= c1; cc += 8) {
      float v[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) v[u] = partials[(int64_t)(cc + u) * D + k];
#pragma unroll
      for (int u = 0; u < 8; ++u) s += v[u];
    }
    for (; cc < c1; ++cc) s += partials[(int64_t)cc * D + k];
    partials[(int64_t)c * D + k] = s;
  }
}

// Hub chunks: one CTA per chunk of kChunkEdges runs (grid-stride over the chunk list), fp32 partial
// sum of the chunk's rows, each times its multiplicity.  The chunk's run entries are copied to
// shared memory (cp.async) while the CTA sums the chunk before.  Group g sums runs g, g + kGroups,
// ... in order: each lane copies its 16-byte slices of eight gathered rows per stage into its own
// slots of a two-stage ring in shared memory (cp.async, so rows in flight hold no registers and no
// lane waits on another), and adds a stage while the next one lands.  The groups' sums are then
// added in group order (16-byte shared stores, the row stages reused).
template <typename T, int D>
struct ChunkCfg {
  using S = AggShape<T, D>;
  static constexpr int kRows = 8;  // gathered rows per stage and group
  static constexpr int kStageBytes = kRows * D * (int)sizeof(T);
  static constexpr int kRingBytes = S::kGroups * 2 * kStageBytes;  // also holds the groups' fp32 sums
  static_assert(S::kGroups * D * 4 <= kRingBytes, "reduction buffer");
  static constexpr int kIdxBytes = 2 * 2 * kChunkEdges * 4;  // column and count, two chunks
  static constexpr int kSmem = kRingBytes + kIdxBytes;
};

template <typename T, int D>
__global__ void __launch_bounds__(256) agg_chunks(const int32_t* __restrict__ ptr, const int32_t* __restrict__ col,
                                                  const int32_t* __restrict__ cnt,
                                                  const T* __restrict__ src, const int32_t* __restrict__ chunk_row,
                                                  const int32_t* __restrict__ chunk_ofs, int64_t rows,
                                                  float* __restrict__ partials) {
  using S = AggShape<T, D>;
  using C = ChunkCfg<T, D>;
  extern __shared__ uint4 chunk_smem[];
  uint8_t* ring = reinterpret_cast<uint8_t*>(chunk_smem);
  int32_t* sidx = reinterpret_cast<int32_t*>(ring + C::kRingBytes);  // [2][col | cnt][kChunkEdges]
  float* red = reinterpret_cast<float*>(ring);                        // [kGroups][D], after the sums
  const int grp = threadIdx.x / S::G, lane = threadIdx.x % S::G;
  const int nchunks = chunk_ofs[rows];
  // runs [beg, end) of chunk c
  auto span = [&](int c, int64_t& beg, int64_t& end) {
    const int row = chunk_row[c];
    beg = (int64_t)ptr[row] + (int64_t)(c - chunk_ofs[row]) * kChunkEdges;
    end = min((int64_t)ptr[row + 1], beg + kChunkEdges);
  };
  auto load_idx = [&](int c, int buf) {  // every thread: a few entries of chunk c's runs
    int64_t b, e;
    span(c, b, e);
    int32_t* d = sidx + buf * 2 * kChunkEdges;
    for (int k = threadIdx.x; k < e - b; k += blockDim.x) {
      tc::cp_async4(d + k, col + b + k);
      tc::cp_async4(d + kChunkEdges + k, cnt + b + k);
    }
  };
  uint8_t* myring = ring + grp * 2 * C::kStageBytes;
  if (blockIdx.x < nchunks) load_idx(blockIdx.x, 0);
  tc::cp_async_commit();
  int it = 0;
  for (int c = blockIdx.x; c < nchunks; c += gridDim.x, ++it) {
    const int buf = it & 1;
    int64_t beg, end;
    span(c, beg, end);
    const int n = (int)(end - beg);
    if (c + (int)gridDim.x < nchunks) load_idx(c + gridDim.x, buf ^ 1);  // the next chunk's runs
    tc::cp_async_commit();
    tc::cp_async_wait<1>();  // this chunk's run entries (this thread's copies) ...
    __syncthreads();         // ... and every thread's
    const int32_t* scol = sidx + buf * 2 * kChunkEdges;
    const int32_t* scnt = scol + kChunkEdges;
    const int mine = grp < n ? (n - grp + S::kGroups - 1) / S::kGroups : 0;  // runs of this group
    const int nb = (mine + C::kRows - 1) / C::kRows;
    auto issue = [&](int b) {  // batch b into stage b & 1 (an empty commit past the last batch)
      uint8_t* st = myring + (b & 1) * C::kStageBytes;
#pragma unroll
      for (int u = 0; u < C::kRows; ++u) {
        const int j = b * C::kRows + u;
        if (j < mine) {
          const int cidx = scol[grp + j * S::kGroups];
#pragma unroll
          for (int v = 0; v < S::V; ++v) {
            const int o = (lane + v * S::G) * S::kVec;
            tc::cp_async16(st + u * D * (int)sizeof(T) + o * (int)sizeof(T), src + (int64_t)cidx * D + o, true);
          }
        }
      }
      tc::cp_async_commit();
    };
    float acc[S::F];
#pragma unroll
    for (int q = 0; q < S::F; ++q) acc[q] = 0.f;
    issue(0);
    for (int b = 0; b < nb; ++b) {
      issue(b + 1);
      tc::cp_async_wait<1>();  // batch b (this lane's slices) has landed
      const uint8_t* st = myring + (b & 1) * C::kStageBytes;
#pragma unroll
      for (int u = 0; u < C::kRows; ++u) {
        const int j = b * C::kRows + u;
        if (j >= mine) break;
        const float w = (float)scnt[grp + j * S::kGroups];
#pragma unroll
        for (int v = 0; v < S::V; ++v) {
          const int o = (lane + v * S::G) * S::kVec;
          float f[S::kVec];
          unpack(*reinterpret_cast<const uint4*>(st + u * D * (int)sizeof(T) + o * (int)sizeof(T)), f, T());
#pragma unroll
          for (int q = 0; q < S::kVec; ++q) acc[v * S::kVec + q] = fmaf(w, f[q], acc[v * S::kVec + q]);
        }
      }
    }
    tc::cp_async_wait<0>();
    __syncthreads();  // every group is done with its ring: it becomes the reduction buffer
#pragma unroll
    for (int v = 0; v < S::V; ++v)
#pragma unroll
      for (int q = 0; q < S::kVec; q += 4)
        *reinterpret_cast<float4*>(red + grp * D + (lane + v * S::G) * S::kVec + q) =
            make_float4(acc[v * S::kVec + q], acc[v * S::kVec + q + 1], acc[v * S::kVec + q + 2],
                        acc[v * S::kVec + q + 3]);
    __syncthreads();
    for (int k = threadIdx.x; k < D; k += blockDim.x) {
      float s = 0.f;
#pragma unroll
      for (int g = 0; g < S::kGroups; ++g) s += red[g * D + k];
      partials[(int64_t)c * D + k] = s;
    }
    __syncthreads();
  }
  tc::cp_async_wait<0>();
}

// A lane's share of a feature row held by a whole warp: E = D / 32 consecutive elements (4 to 32
// bytes), loaded with one or two vector loads and widened to fp32.
template <typename T, int D>
struct Slice {
  static constexpr int E = D / 32;
  static constexpr int kWords = E * (int)sizeof(T) / 4;  // 32-bit words
  uint32_t w[kWords];
  __device__ __forceinline__ void load(const T* p) {
    if constexpr (kWords == 1) {
      w[0] = __ldg(reinterpret_cast<const uint32_t*>(p));
    } else if constexpr (kWords == 2) {
      const uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
      w[0] = v.x;
      w[1] = v.y;
    } else {
#pragma unroll
      for (int i = 0; i < kWords / 4; ++i) {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(p) + i);
        w[4 * i] = v.x;
        w[4 * i + 1] = v.y;
        w[4 * i + 2] = v.z;
        w[4 * i + 3] = v.w;
      }
    }
  }
  __device__ __forceinline__ void to_float(float* f) const {
    if constexpr (sizeof(T) == 4) {
#pragma unroll
      for (int i = 0; i < E; ++i) f[i] = __uint_as_float(w[i]);
    } else {
#pragma unroll
      for (int i = 0; i < kWords; ++i) {
        f[2 * i] = __uint_as_float(w[i] << 16);
        f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
      }
    }
  }
  // v * scale rounded to T, stored at p
  __device__ __forceinline__ static void store(T* p, const float* v, float scale) {
    uint32_t o[kWords];
    if constexpr (sizeof(T) == 4) {
#pragma unroll
      for (int i = 0; i < E; ++i) o[i] = __float_as_uint(v[i] * scale);
    } else {
#pragma unroll
      for (int i = 0; i < kWords; ++i) {
        __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * i] * scale, v[2 * i + 1] * scale);
        o[i] = *reinterpret_cast<uint32_t*>(&h);
      }
    }
    if constexpr (kWords == 1) {
      *reinterpret_cast<uint32_t*>(p) = o[0];
    } else if constexpr (kWords == 2) {
      *reinterpret_cast<uint2*>(p) = make_uint2(o[0], o[1]);
    } else {
#pragma unroll
      for (int i = 0; i < kWords / 4; ++i)
        reinterpret_cast<uint4*>(p)[i] = make_uint4(o[4 * i], o[4 * i + 1], o[4 * i + 2], o[4 * i + 3]);
    }
  }
};

// Row kernels, streamed (agg_fwd_rows, agg_bwd_nodes).  A warp takes a chunk of 16 consecutive rows
// (lane l < 16 holds row l's bounds and scale; every lane owns D / 32 columns) and streams through
// the chunk's runs, which are contiguous, in batches of eight gathered rows that cross row
// boundaries; a row is written when its last run is added, so the loads of a short row do not wait
// on those of the row before.  Each row's runs are added one by one, in run order, into an fp32
// accumulator that starts at 0.  The bounds of the next chunk (and the rows of the one after) are
// loaded while a chunk streams.  Rows above kHubDegree runs take their sum from the chunk partials.
// Persistent, with dynamic work: chunk costs are heavy-tailed, so a warp claims blocks of kClaim
// chunks from a counter (zeroed before the launch; the next block claimed a block ahead).
//   forward  (kBwd = false): rows = the non-empty CSR rows in compact order (row mlist[k]; their
//            count read on the device); M[k] = sum / deg (deg = the CSR row length, eptr).
//   backward (kBwd = true):  rows = nodes 0 .. n - 1 of the node-major lists; dH[i] = sum + dY[i],
//            the dY rows of the next chunk copied to shared memory (cp.async, each lane its own
//            slices, two buffers) while a chunk streams.
constexpr int kStreamRows = 16;  // rows per chunk
constexpr int kClaim = 4;        // chunks per claim

template <typename T, int D>
struct StreamCfg {
  static constexpr int kFwdThreads = 256;
  static constexpr int kBwdThreads = 128;
  static constexpr int kYBytes = kBwdThreads / 32 * 2 * kStreamRows * D * (int)sizeof(T);  // backward dY buffers
};

// kGapped: the listed rows' runs are not contiguous (a subset of the CSR rows, such as the fused
// layer's long rows): each row's batches start at its own first run and stop at its last.
template <typename T, int D, bool kBwd, bool kGapped = false>
__device__ __forceinline__ void stream_rows(const int32_t* __restrict__ ptr, const int32_t* __restrict__ col,
                                            const int32_t* __restrict__ cnt, const int32_t* __restrict__ eptr,
                                            const int32_t* __restrict__ mlist, int64_t nrows,
                                            const T* __restrict__ src, const T* __restrict__ dY, T* __restrict__ out,
                                            const int32_t* __restrict__ chunk_ofs, const float* __restrict__ partials,
                                            int32_t* __restrict__ work, T* __restrict__ ysm) {
  using SL = Slice<T, D>;
  constexpr int E = SL::E, CR = kStreamRows, U = 8;
  constexpr int kSliceBytes = E * (int)sizeof(T);
  constexpr unsigned kAll = 0xffffffffu;
  const int lane = threadIdx.x & 31;
  const int64_t nchunks = (nrows + CR - 1) / CR;
  const T* base = src + lane * E;
  T* ys = ysm + (size_t)(threadIdx.x >> 5) * 2 * CR * D;  // this warp's two dY buffers (backward)
  // the warp's chunk sequence: blocks of kClaim chunks claimed from the counter by lane 0; the
  // following block's claim is in flight while a block is processed
  int claim_next = 0, j = 0;
  int claim_cur = 0;
  if (lane == 0) {
    claim_cur = atomicAdd(work, 1);
    claim_next = atomicAdd(work, 1);
  }
  int blk = __shfl_sync(kAll, claim_cur, 0);
  auto take = [&]() -> int64_t {
    const int64_t r = (int64_t)blk * kClaim + j;
    if (++j == kClaim) {
      j = 0;
      blk = __shfl_sync(kAll, claim_next, 0);
      if (lane == 0) claim_next = atomicAdd(work, 1);
    }
    return r;
  };
  // list row of chunk ch's row `lane` (-1: none)
  auto row_of = [&](int64_t ch) -> int {
    const int64_t k = ch * CR + lane;
    if (ch >= nchunks || lane >= CR || k >= nrows) return -1;
    return kBwd ? (int)k : __ldg(mlist + k);
  };
  auto bounds = [&](int row, int& rb, int& re, float& sc) {
    rb = re = 0;
    sc = 1.f;
    if (row >= 0) {
      rb = __ldg(ptr + row);
      re = __ldg(ptr + row + 1);
      if (!kBwd) sc = __fdiv_rn(1.0f, (float)(__ldg(eptr + row + 1) - __ldg(eptr + row)));
    }
  };
  // backward: chunk ch's dY rows (this lane's slices) into buffer b; one commit group per call
  auto stage_y = [&](int64_t ch, int b) {
    if constexpr (kBwd) {
      if (ch < nchunks) {
        const int nr = (int)min((int64_t)CR, nrows - ch * CR);
        for (int r = 0; r < nr; ++r) {
          T* d = ys + (b * CR + r) * D + lane * E;
          const T* g = dY + (ch * CR + r) * D + lane * E;
          if constexpr (kSliceBytes == 4) {
            tc::cp_async4(d, g);
          } else if constexpr (kSliceBytes == 8) {
            tc::cp_async8(d, g);
          } else {
#pragma unroll
            for (int q = 0; q < kSliceBytes / 16; ++q) tc::cp_async16(d + q * (16 / (int)sizeof(T)), g + q * (16 / (int)sizeof(T)), true);
          }
        }
      }
      tc::cp_async_commit();
    }
  };
  int64_t ch = take(), nch = take(), nnch = take();
  int row = row_of(ch), rb, re;
  float sc;
  bounds(row, rb, re, sc);
  int nrow = row_of(nch);
  stage_y(ch, 0);
  for (int it = 0; ch < nchunks; ch = nch, nch = nnch, nnch = take(), ++it) {
    const int64_t k0 = ch * CR;
    const int nr = (int)min((int64_t)CR, nrows - k0);
    stage_y(nch, (it + 1) & 1);  // the next chunk's dY rows
    // the next chunk's bounds (its rows were loaded a chunk ago) and the rows of the one after
    int nrb, nre;
    float nsc;
    bounds(nrow, nrb, nre, nsc);
    const int nnrow = row_of(nnch);

    const unsigned hubs = __ballot_sync(kAll, lane < nr && re - rb > kHubDegree);
    const int chunk_end = __shfl_sync(kAll, re, nr - 1);
    int e = __shfl_sync(kAll, rb, 0);
    int cur = 0;                          // row of the chunk being summed
    int cend = __shfl_sync(kAll, re, 0);  // its last run + 1
    bool ywait = kBwd;                    // this chunk's dY rows not yet waited for
    const T* yb = ys + (it & 1) * CR * D + lane * E;
    float acc[E];
#pragma unroll
    for (int q = 0; q < E; ++q) acc[q] = 0.f;
    // writes row cur and moves to the next row
    auto flush = [&]() {
      if constexpr (kBwd) {
        if (ywait) {
          tc::cp_async_wait<1>();  // all but the next chunk's copies
          ywait = false;
        }
        SL y;
#pragma unroll
        for (int q = 0; q < SL::kWords; ++q) y.w[q] = reinterpret_cast<const uint32_t*>(yb + cur * D)[q];
        float f[E];
        y.to_float(f);
#pragma unroll
        for (int q = 0; q < E; ++q) acc[q] += f[q];
      }
      SL::store(out + (k0 + cur) * D + lane * E, acc, __shfl_sync(kAll, sc, cur));
#pragma unroll
      for (int q = 0; q < E; ++q) acc[q] = 0.f;
      ++cur;
      if (cur < nr) cend = __shfl_sync(kAll, re, cur);
      if constexpr (kGapped) {
        if (cur < nr) e = __shfl_sync(kAll, rb, cur);
      }
    };
    while (cur < nr) {
      if ((hubs >> cur) & 1u) {  // a hub row: the sum of its chunk partials, in chunk-run order
        const int hrow = __shfl_sync(kAll, row, cur);
        for (int c = chunk_ofs[hrow]; c < chunk_ofs[hrow + 1]; c += kPartRun) {
          const float* p = partials + (int64_t)c * D + lane * E;
#pragma unroll
          for (int q = 0; q < E; ++q) acc[q] += p[q];
        }
        e = cend;
        flush();
        continue;
      }
      if (e >= cend) {  // the row's runs are all added (or it has none)
        flush();
        continue;
      }
      // up to U runs from e on, stopping at the next hub row (whose runs are not gathered)
      const unsigned later = hubs & ~((2u << cur) - 1u);
      const int stop = kGapped ? cend : (later ? __shfl_sync(kAll, rb, __ffs(later) - 1) : chunk_end);
      const int nb = min(U, stop - e);
      int c[U];
      float w[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        c[u] = u < nb ? __ldg(col + e + u) : 0;
        w[u] = u < nb ? (float)__ldg(cnt + e + u) : 0.f;
      }
      SL x[U];
#pragma unroll
      for (int u = 0; u < U; ++u)
        if (u < nb) x[u].load(base + (int64_t)c[u] * D);
#pragma unroll
      for (int u = 0; u < U; ++u) {
        if (u >= nb) break;
        while (e + u >= cend) flush();  // run e + u belongs to a later row (not a hub: nb stops before)
        float f[E];
        x[u].to_float(f);
#pragma unroll
        for (int q = 0; q < E; ++q) acc[q] = fmaf(w[u], f[q], acc[q]);
      }
      e += nb;
    }
    row = nrow;
    rb = nrb;
    re = nre;
    sc = nsc;
    nrow = nnrow;
  }
  if constexpr (kBwd) tc::cp_async_wait<0>();  // no copy outlives the kernel
}

template <typename T, int D, bool kGapped = false>
__global__ void __launch_bounds__(StreamCfg<T, D>::kFwdThreads) agg_fwd_rows(
    const int32_t* __restrict__ ptr, const int32_t* __restrict__ col, const int32_t* __restrict__ cnt,
    const int32_t* __restrict__ eptr, const int32_t* __restrict__ mlist, const int32_t* __restrict__ nnz_p,
    const T* __restrict__ H, T* __restrict__ M, const int32_t* __restrict__ chunk_ofs,
    const float* __restrict__ partials, int32_t* __restrict__ work) {
  stream_rows<T, D, false, kGapped>(ptr, col, cnt, eptr, mlist, (int64_t)*nnz_p, H, nullptr, M, chunk_ofs, partials, work,
                           nullptr);
}

template <typename T, int D>
__global__ void __launch_bounds__(StreamCfg<T, D>::kBwdThreads) agg_bwd_nodes(
    int64_t N, const int32_t* __restrict__ nptr, const int32_t* __restrict__ ncol, const int32_t* __restrict__ ncnt,
    const T* __restrict__ dMs, const T* __restrict__ dY, T* __restrict__ dH, const int32_t* __restrict__ chunk_ofs,
    const float* __restrict__ partials, int32_t* __restrict__ work) {
  extern __shared__ uint4 ysm_raw[];
  stream_rows<T, D, true>(nptr, ncol, ncnt, nullptr, nullptr, N, dMs, dY, dH, chunk_ofs, partials, work,
                          reinterpret_cast<T*>(ysm_raw));
}

// ---------------------------------------------------------------------------------------------
// host dispatch
// ---------------------------------------------------------------------------------------------
// Persistent grids: as many 256-thread blocks as are resident at once (occupancy of the kernel).
template <typename K>
static hg_status persist_blocks(K kernel, int64_t* blocks, size_t smem = 0, int threads = 256) {
  int dev = 0, sms = 0, per_sm = 0;
  HG_CUDA(cudaGetDevice(&dev));
  HG_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  HG_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, smem));
  *blocks = (int64_t)sms * std::max(1, per_sm);
  return HG_OK;
}

static unsigned chunk_grid(int64_t cap) { return (unsigned)std::max<int64_t>(1, std::min<int64_t>(cap, 152 * 8)); }

// resident blocks of the hub-chunk kernel (its shared memory set up once)
template <typename T, int D>
static hg_status chunk_blocks(int64_t* blocks) {
  static int64_t cb = 0;
  if (cb == 0) {
    HG_CUDA(cudaFuncSetAttribute(agg_chunks<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, ChunkCfg<T, D>::kSmem));
    HG_TRY(persist_blocks(agg_chunks<T, D>, &cb, ChunkCfg<T, D>::kSmem));
  }
  *blocks = cb;
  return HG_OK;
}

// The means of the rows listed in mlist (their count at nnz_p, at most cap): the hub rows' chunk
// partials first, then the streaming row kernel.
template <typename T, int D, bool kGapped>
static hg_status agg_fwd_t(const hg_graph* g, const void* H, void* M, float* partials, int32_t* work,
                           const int32_t* mlist, const int32_t* nnz_p, int64_t cap, cudaStream_t s) {
  int64_t cb = 0;
  HG_TRY((chunk_blocks<T, D>(&cb)));
  HG_TRY(launch("agg_fwd_chunks", agg_chunks<T, D>, dim3((unsigned)std::max<int64_t>(1, std::min<int64_t>(g->chunk_cap_csr, cb))), dim3(256),
                ChunkCfg<T, D>::kSmem, s,
                (const int32_t*)g->agg_ptr, (const int32_t*)g->agg_col, (const int32_t*)g->agg_cnt, (const T*)H,
                (const int32_t*)g->agg_chunk_row, (const int32_t*)g->agg_chunk_ofs, g->csr_rows, partials));
  HG_TRY(launch("combine_chunk_partials", combine_chunk_partials<D>, dim3(chunk_grid(g->chunk_cap_csr)), dim3(D), 0, s,
                (const int32_t*)g->agg_chunk_row, (const int32_t*)g->agg_chunk_ofs, g->csr_rows, partials));
  constexpr int kT = StreamCfg<T, D>::kFwdThreads;
  static int64_t pb = 0;
  if (pb == 0) HG_TRY(persist_blocks(agg_fwd_rows<T, D, kGapped>, &pb, 0, kT));
  const int64_t chunks = ceil_div(std::max<int64_t>(cap, 1), kStreamRows);  // a warp per chunk
  HG_CUDA(cudaMemsetAsync(work, 0, sizeof(int32_t), s));
  return launch(kGapped ? "agg_fwd_long_rows" : "agg_fwd_rows", agg_fwd_rows<T, D, kGapped>,
                dim3((unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(chunks, kT / 32), pb))), dim3(kT), 0,
                s, (const int32_t*)g->agg_ptr, (const int32_t*)g->agg_col, (const int32_t*)g->agg_cnt,
                (const int32_t*)g->csr_ptr, mlist, nnz_p, (const T*)H, (T*)M, (const int32_t*)g->agg_chunk_ofs,
                (const float*)partials, work);
}

template <typename T, int D>
static hg_status agg_fwd_dense_t(const hg_graph* g, const void* H, void* M, float* partials, int32_t* work,
                                 const int32_t* mlist, const int32_t* nnz_p, int64_t cap, cudaStream_t s) {
  return agg_fwd_t<T, D, false>(g, H, M, partials, work, mlist, nnz_p, cap, s);
}
template <typename T, int D>
static hg_status agg_fwd_gapped_t(const hg_graph* g, const void* H, void* M, float* partials, int32_t* work,
                                  const int32_t* mlist, const int32_t* nnz_p, int64_t cap, cudaStream_t s) {
  return agg_fwd_t<T, D, true>(g, H, M, partials, work, mlist, nnz_p, cap, s);
}

template <typename T, int D>
static hg_status agg_bwd_t(const hg_graph* g, const void* dMs, const void* dY, void* dH, float* partials,
                           int32_t* work, cudaStream_t s) {
  int64_t cb = 0;
  const int64_t N = g->meta.type_off[g->meta.num_types];
  HG_TRY((chunk_blocks<T, D>(&cb)));
  HG_TRY(launch("agg_bwd_chunks", agg_chunks<T, D>, dim3((unsigned)std::max<int64_t>(1, std::min<int64_t>(g->chunk_cap_node, cb))), dim3(256),
                ChunkCfg<T, D>::kSmem, s,
                (const int32_t*)g->bagg_ptr, (const int32_t*)g->bagg_col, (const int32_t*)g->bagg_cnt, (const T*)dMs,
                (const int32_t*)g->bagg_chunk_row, (const int32_t*)g->bagg_chunk_ofs, N, partials));
  HG_TRY(launch("combine_chunk_partials", combine_chunk_partials<D>, dim3(chunk_grid(g->chunk_cap_node)), dim3(D), 0,
                s, (const int32_t*)g->bagg_chunk_row, (const int32_t*)g->bagg_chunk_ofs, N, partials));
  constexpr int kT = StreamCfg<T, D>::kBwdThreads, kY = StreamCfg<T, D>::kYBytes;
  static int64_t pb = 0;
  if (pb == 0) {
    HG_CUDA(cudaFuncSetAttribute(agg_bwd_nodes<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize, kY));
    HG_TRY(persist_blocks(agg_bwd_nodes<T, D>, &pb, kY, kT));
  }
  const int64_t chunks = ceil_div(N, kStreamRows);
  HG_CUDA(cudaMemsetAsync(work + 1, 0, sizeof(int32_t), s));
  return launch("agg_bwd_nodes", agg_bwd_nodes<T, D>,
                dim3((unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(chunks, kT / 32), pb))), dim3(kT), kY, s,
                N, (const int32_t*)g->bagg_ptr, (const int32_t*)g->bagg_col, (const int32_t*)g->bagg_cnt,
                (const T*)dMs, (const T*)dY, (T*)dH, (const int32_t*)g->bagg_chunk_ofs, (const float*)partials,
                work + 1);
}

#define HG_DISPATCH_TD(dtype, d, FN, ...)                                                   \
  do {                                                                                      \
    if (dtype == HG_F32) {                                                                  \
      if (d == 64) return FN<float, 64>(__VA_ARGS__);                                       \
      if (d == 128) return FN<float, 128>(__VA_ARGS__);                                     \
      if (d == 256) return FN<float, 256>(__VA_ARGS__);                                     \
    } else {                                                                                \
      if (d == 64) return FN<__nv_bfloat16, 64>(__VA_ARGS__);                               \
      if (d == 128) return FN<__nv_bfloat16, 128>(__VA_ARGS__);                             \
      if (d == 256) return FN<__nv_bfloat16, 256>(__VA_ARGS__);                             \
    }                                                                                       \
    set_error("unsupported feature width %d", d);                                           \
    return HG_ERR_UNSUPPORTED;                                                              \
  } while (0)

hg_status aggregate_forward(const hg_graph* g, hg_dtype dt, int d, const void* H, void* M, float* partials,
                            int32_t* work, cudaStream_t s) {
  // the non-empty rows, in compact order (at most csr_rows)
  HG_DISPATCH_TD(dt, d, agg_fwd_dense_t, g, H, M, partials, work, (const int32_t*)g->mlist,
                 (const int32_t*)(g->mbase + g->meta.num_rels), g->csr_rows, s);
}

hg_status aggregate_forward_long(const hg_graph* g, int d, const void* H, void* Mlong, float* partials, int32_t* work,
                                 cudaStream_t s) {
  HG_DISPATCH_TD(HG_BF16, d, agg_fwd_gapped_t, g, H, Mlong, partials, work, (const int32_t*)g->long_list,
                 (const int32_t*)(g->long_ofs + g->csr_rows), g->long_cap, s);
}

hg_status aggregate_backward(const hg_graph* g, hg_dtype dt, int d, const void* dMs, const void* dY, void* dH,
                             float* partials, int32_t* work, cudaStream_t s) {
  HG_DISPATCH_TD(dt, d, agg_bwd_t, g, dMs, dY, dH, partials, work, s);
}

}  // namespace hg
