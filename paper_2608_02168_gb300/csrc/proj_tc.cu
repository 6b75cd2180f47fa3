// Dense projections of the layer on the 5th-generation tensor cores (tcgen05, bf16 operands,
// fp32 accumulation in tensor memory).  Used for bf16 storage; fp32 storage stays on CUDA cores.
//
// The two products of Eq. 7 and Eq. 11 are associated as U = sum_r M_r V_r + b with the fused
// weights V_r = W_r W_agg[t_r] (computed once per layer in fp64): the same value as
// (sum_r M_r W_r) W_agg, with one GEMM instead of two and no intermediate Z.  A product of two
// weight matrices is not a bf16 number, and one rounding of V_r would shift every row's
// pre-activation the same way (an error that the weight gradients, sums over all rows, do not
// average out), so V_r is kept as an unevaluated pair V_r = V_hi + V_lo of bf16 matrices (V_hi =
// bf16(V_r), V_lo = bf16(V_r - V_hi); about 16 significant bits) and every product with it is two
// MMAs into the same fp32 accumulator.
//
// Forward, one CTA per 128 destination rows of type t, rows in the graph's node order (the type's
// nodes sorted by which relations have in-edges at them, so that a tile's rows share their stored
// relation rows):
//   U = sum_{r -> t} M_r V_r      over the relations with a stored row in the tile; A = the rows'
//                                 relation means (cp.async gathers, 128 x 64 tiles, empty rows zero),
//                                 B = V_r^T chunks (hi and lo halves of a chunk in one stage)
//   epilogue: U_s = bf16(U) stored, then U = U_s + b in fp32; Y = act(U) + H_in;
//             H_out = LayerNorm(Y); row statistics saved.  U is stored without its bias: the
//             rounding then scales with the data (Z W_agg), not with a large bias, and the
//             backward adds the same bias back, so both passes see the same U.
// Backward:
//   ln_act_bwd   (warp per row)  dY = LayerNorm backward, dU = dY act'(U); column partials of the
//                                bias / gain / shift gradients
//   proj_bwd_tc  (persistent, jobs of 128 stored rows)  dMs_r = (dU V_r^T) / deg_r   (A = the rows'
//                                dU gathered by TMA, B = V_r chunks, hi and lo halves)
//   weight gradients: G_r = M_r^T dU over a relation's stored rows (wgrad_rows_tc: split-K, MN-major
//                     operands copied by cp.async; wgrad_tc: the dense variant with TMA operands for
//                     callers whose rows are all stored), then dW_r = G_r W_agg^T and
//                     dW_agg[t] = sum_{r -> t} W_r^T G_r (wgrad_finish).
//
// Epilogue threads own one accumulator row each (warp w reads TMEM lanes 32 (w % 4) ..); one
// thread issues the MMAs.  All waits are bounded (tc::kSpinLimit) and report through the library
// status word.
#include <algorithm>
#include <cstring>

#include "layer_kernels.cuh"
#include "simt_tile.cuh"
#include "tc_util.cuh"

namespace hg {

using namespace tc;

namespace {

constexpr int kTileRows = 128;
constexpr int kATile = kTileRows * 128;  // 128 rows x 64 bf16

// Persistent forward: one CTA per SM.  Warps 0-1 load the operands (cp.async gathers of A rows,
// thread 0 also the weight chunks by TMA), warp 2 issues the MMAs, warps 3-10 run the epilogue, two
// threads per row (one per column half; eight warps, two per scheduler).  Two TMEM accumulators and
// two residual tiles let the epilogue of one 128-row tile overlap the loads and MMAs of the next,
// and every role loads the next tile's metadata (relations, node order, rows of M) ahead of time.
template <int D, bool kGather = false>
struct FwdCfg {
  static constexpr int kStages = D == 256 ? 2 : (D == 128 ? 3 : 4);
  static constexpr int kB = D * 128;  // D rows x 64 bf16 (one half of the weight pair)
  static constexpr int kStage = kATile + 2 * kB;  // A | B_hi | B_lo
  // The H_in rows (residual) are staged in shared memory, double-buffered, where it has room; at
  // D = 256 the epilogue reads H_in from global memory.
  static constexpr bool kHTile = D <= 128;
  static constexpr int kH = kHTile ? kTileRows * D * 2 : 0;
  static constexpr int kParams = 3 * D * 4;  // bias, gamma, beta in fp32
  static constexpr int kRed = 2 * 2 * kTileRows * 4;  // row partial sums of the two column halves
  static constexpr int kSmem = kStages * kStage + 2 * kH + kParams + kRed + 256 + 1024;
  static_assert(kSmem <= 227 * 1024, "shared memory of proj_fwd_tc");
  static constexpr int kAccCols = D < 32 ? 32 : D;
  static constexpr int kTmemCols = 2 * kAccCols;
  // Roles.  Plain: warps 0-1 copy the stored rows of M (64 A rows each), warp 2 issues the MMAs,
  // warps 3-10 run the epilogue.  Gather variant (the fused mean layer): sixteen warps whose
  // registers are split by warpgroup (setmaxnreg): warps 0-3 and 5-7 sum the relation means into
  // the A stages and warp 4 issues the MMAs, at kLowRegs; warps 8-15 run the epilogue at kHighRegs.
  static constexpr int kGatherWarps = 7;
  static constexpr int kProducers = kGather ? 32 * kGatherWarps : 64;  // producer threads (stage arrivals)
  static constexpr int kMmaWarp = kGather ? 4 : 2;
  static constexpr int kEpiWarp0 = kGather ? 8 : 3;
  static constexpr int kEpiThreads = 2 * kTileRows;
  static constexpr int kThreads = kGather ? 512 : 96 + kEpiThreads;
  static constexpr int kHalf = D / 2;  // columns per epilogue thread
  static constexpr int kLowRegs = 88, kHighRegs = 168;
  // the two register levels use exactly the launch's 128 registers per thread
  static_assert(!kGather || (256 * (kLowRegs + kHighRegs) == kThreads * 128 && kEpiWarp0 == 8), "register split");
};
static_assert(kTileRows == kProjTileRows, "tile of the node order");

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<uint32_t*>(&h);
}

__device__ __forceinline__ uint8_t* align1024(uint8_t* p) {
  return reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(p) + 1023) & ~uintptr_t(1023));
}

__device__ __forceinline__ void load16_bf16(const __nv_bfloat16* p, float* v) {
  unpack(ld16(p), v, __nv_bfloat16());
  unpack(ld16(p + 8), v + 8, __nv_bfloat16());
}
__device__ __forceinline__ void store16_bf16(__nv_bfloat16* p, const float* v) {
  st16(p, pack(v, __nv_bfloat16()));
  st16(p + 8, pack(v + 8, __nv_bfloat16()));
}

}  // namespace

// ---------------------------------------------------------------------------------------------
// forward projection
// ---------------------------------------------------------------------------------------------

template <int D>
__global__ void __launch_bounds__(FwdCfg<D>::kThreads, 1)
    proj_fwd_tc(const __grid_constant__ CUtensorMap tm_Vt, TcFwdArgs a);
template <int D>
__global__ void __launch_bounds__(FwdCfg<D, true>::kThreads, 1)
    proj_fwd_gather_tc(const __grid_constant__ CUtensorMap tm_Vt, TcFwdArgs a);

template <int D, bool kGather>
__device__ __forceinline__ void proj_fwd_body(const CUtensorMap& tm_Vt, const TcFwdArgs& a) {
  using C = FwdCfg<D, kGather>;
  constexpr int S = C::kStages;
  constexpr int KC = D / 64;        // 64-wide K chunks per D
  constexpr uint32_t kLag = S - 1;  // stages a producer thread keeps in flight before releasing one
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* stage = smem;                  // S x (A | B)
  uint8_t* htile = smem + S * C::kStage;  // 2 x KC x 16 KB, 128B-swizzled rows
  float* params = reinterpret_cast<float*>(htile + 2 * C::kH);  // [3][D]: b, gamma, beta
  float* red = params + 3 * D;                                  // [2 sums][2 halves][128 rows]
  uint64_t* full = reinterpret_cast<uint64_t*>(red + 4 * kTileRows);
  uint64_t* empty = full + S;
  uint64_t* acc_full = empty + S;      // [2] MMA -> epilogue
  uint64_t* acc_empty = acc_full + 2;  // [2] epilogue -> MMA
  uint64_t* drainb = acc_empty + 2;    // the MMA issuer's give-up path
  uint32_t* tslot = reinterpret_cast<uint32_t*>(drainb + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t ntiles = (a.n + kTileRows - 1) / kTileRows;
  const int64_t G = gridDim.x;
  const uint32_t all = (1u << a.nrel) - 1u;
  // the relations whose products tile q computes (a relation without a stored row in it is skipped)
  auto rels_of = [&](int64_t q) -> uint32_t {
    if (q >= ntiles) return 0u;
    return a.tmask ? (uint32_t)__ldg(a.tmask + q) & all : all;
  };
  // local node at position m of the order; -1 past the type
  auto node_at = [&](int64_t m) -> int64_t {
    if (m >= a.n) return -1;
    return a.perm ? (int64_t)__ldg(a.perm + m) : m;
  };
  __shared__ int64_t s_row0[kMaxRels];  // gather variant: first CSR row and id of each relation into the type
  __shared__ int s_rel[kMaxRels];
  if constexpr (kGather) {
#pragma unroll
    for (int r = 0; r < kMaxRels; ++r)
      if (threadIdx.x == r) {
        s_row0[r] = a.mrow0[r];
        s_rel[r] = a.rel[r];
      }
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(&full[s], C::kProducers + 1);  // the producer threads and the weight loads' byte count
      mbar_init(&empty[s], 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&acc_full[b], 1);
      mbar_init(&acc_empty[b], C::kEpiThreads);
    }
    mbar_init(drainb, 1);
    fence_mbar_init();
    prefetch_tmap(&tm_Vt);
  }
  if (warp == C::kMmaWarp) tmem_alloc(tslot, C::kTmemCols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;

  auto gather_role = [&]() {
    if constexpr (kGather) {
      // ---- gather producers (the fused mean layer).  The seven warps' fourteen half-warps share
      // the rows of every relation tile: half h takes rows h, h + 14, ...; lane l of a half owns
      // 16-byte chunk l of a row (columns 8 l .. 8 l + 7, in K chunk l / 8), so one pass over a
      // row's runs fills both K chunks' stages (g, g + 1), which are filled together.  Rows above
      // kFuseRuns runs copy their mean from Mlong; rows without in-edges (or past the type) are
      // zero; the other rows are streamed: batches of eight runs in row order, crossing row
      // boundaries (each lane of the batch loads one column or count), and a row is written when
      // the batch reaches the next one.  A row's runs are added one by one into an fp32 sum that
      // starts at 0 and the sum is scaled by 1/deg and rounded to bf16: the streaming row
      // kernel's arithmetic, term for term, so M's rows come out bit for bit.  Thread 0 also
      // loads the two stages' V_r^T hi / lo chunks by TMA.  A thread arrives on both stage
      // barriers once its rows are written and fenced for the async proxy.  Lane i < 10 of a half
      // holds row i's metadata (run bounds, 1/deg, long slot), loaded a relation tile ahead, and
      // the nodes a relation tile further ahead.
      static_assert(D == 128 && KC == 2, "gather variant: d = 128");
      constexpr int kGrp = 2 * C::kGatherWarps;                // half-warps
      constexpr int kRowsPer = (kTileRows + kGrp - 1) / kGrp;  // rows per half and relation tile
      static_assert(kRowsPer <= 15, "rows per half fit the 4-bit batch slots");
      const int half = lane >> 4, hl = lane & 15;
      const int grp = 2 * (warp < C::kMmaWarp ? warp : warp - 1) + half;
      const int hb = half << 4;  // first lane of the half
      const unsigned hmask = 0xffffu << hb;
      const int myrow = grp + kGrp * hl;  // the row whose metadata this lane holds
      const bool mine = hl < kRowsPer && myrow < kTileRows;
      const __nv_bfloat16* Hc = a.H_in + hl * 8;
      const uint32_t stage_s = smem_u32(stage);
      bool ok = true;
      uint32_t g = 0;
      // The relation tiles of this CTA (warp-uniform): tiles blockIdx.x, + G, ..., each with the
      // relations of its mask in ascending order (the MMA warp's order).  Lane k holds the mask of
      // tile wb + G k of a window of 32 tiles.
      int wb = blockIdx.x;
      uint32_t wmask = rels_of(wb + G * lane);
      unsigned wnz = __ballot_sync(0xffffffffu, wmask != 0u);
      int wnext = 0;
      uint32_t rem = 0;
      int ctile = 0;
      // the next relation tile: its tile and relation (r = -1 past the last)
      auto next_rt = [&](int& tile, int& r) {
        r = -1;
        while (rem == 0u) {
          const unsigned later = wnext >= 32 ? 0u : (wnz & (0xffffffffu << wnext));
          if (later == 0u) {
            wb += 32 * (int)G;
            if (wb >= ntiles) return;
            wmask = rels_of(wb + G * lane);
            wnz = __ballot_sync(0xffffffffu, wmask != 0u);
            wnext = 0;
            continue;
          }
          const int k = __ffs(later) - 1;
          wnext = k + 1;
          ctile = wb + (int)G * k;
          rem = __shfl_sync(0xffffffffu, wmask, k);
        }
        r = __ffs(rem) - 1;
        rem &= rem - 1u;
        tile = ctile;
      };
      // this lane's node in tile q (-1: none), and its row's metadata under relation r (r < 0: none)
      auto node_of = [&](int q) -> int { return mine ? (int)node_at((int64_t)q * kTileRows + myrow) : -1; };
      auto meta_of = [&](int r, int j, int& rb, int& re, int& slot, float& sc) {
        rb = re = 0;
        slot = -1;
        sc = 0.f;
        if (r >= 0 && j >= 0) {
          const int64_t row = s_row0[r] + j;
          rb = __ldg(a.agg_ptr + row);
          re = __ldg(a.agg_ptr + row + 1);
          const int l0 = __ldg(a.long_ofs + row), l1 = __ldg(a.long_ofs + row + 1);
          const int e0 = __ldg(a.csr_ptr + row), e1 = __ldg(a.csr_ptr + row + 1);
          if (l1 > l0) slot = l0;
          if (e1 > e0) sc = __fdiv_rn(1.0f, (float)(e1 - e0));
        }
      };
      int tile_c = 0, tile_n = 0, r_c, r_n = -1;
      next_rt(tile_c, r_c);
      const int j_c0 = r_c >= 0 ? node_of(tile_c) : -1;
      if (r_c >= 0) next_rt(tile_n, r_n);
      int j_n = r_n >= 0 ? (tile_n == tile_c ? j_c0 : node_of(tile_n)) : -1;
      int m_rb, m_re, m_slot;
      float m_sc;
      meta_of(r_c, j_c0, m_rb, m_re, m_slot, m_sc);
      while (r_c >= 0) {
        int n_rb, n_re, n_slot;
        float n_sc;
        meta_of(r_n, j_n, n_rb, n_re, n_slot, n_sc);  // in flight during this relation tile
        int tile_nn = 0, r_nn = -1;
        if (r_n >= 0) next_rt(tile_nn, r_nn);
        const int j_nn = r_nn >= 0 ? (tile_nn == tile_n ? j_n : node_of(tile_nn)) : -1;
        // the streamed rows (bit i: row grp + 14 i has runs and is not long)
        unsigned qrows = (__ballot_sync(hmask, mine && m_slot < 0 && m_rb < m_re) >> hb) & 0xffffu;
        int qi = 0, qe = 0, qend = 0;  // queue cursor: row qi, its next run qe and end qend
        // the next eight runs in row order: slot k's row in srow (4 bits each, 15: none); returns the
        // entry this lane loads for them: lanes 0-7 the source column of slot l, lanes 8-15 the
        // count of slot l - 8
        auto fill = [&](uint32_t& srow) -> int {
          srow = 0xffffffffu;
          int e = -1;
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            if (qe >= qend && qrows != 0u) {
              qi = __ffs(qrows) - 1;
              qrows &= qrows - 1u;
              qe = __shfl_sync(hmask, m_rb, hb + qi);
              qend = __shfl_sync(hmask, m_re, hb + qi);
            }
            if (qe < qend) {
              srow = (srow & ~(0xFu << (4 * k))) | ((uint32_t)qi << (4 * k));
              if ((hl & 7) == k) e = qe;
              ++qe;
            }
          }
          return e >= 0 ? __ldg((hl < 8 ? a.agg_col : a.agg_cnt) + e) : 0;
        };
        uint32_t srow;
        int v = fill(srow);  // the first batch's run entries, in flight while the stages are awaited
        // ---- the relation tile's two stages
        const uint32_t s0 = g % S, s1 = (g + 1) % S;
        bool w_ok = true;
        if (g >= (uint32_t)S) w_ok = mbar_wait(&empty[s0], ((g / S) - 1) & 1);
        if (w_ok && g + 1 >= (uint32_t)S) w_ok = mbar_wait(&empty[s1], (((g + 1) / S) - 1) & 1);
        ok = __all_sync(0xffffffffu, w_ok);
        if (!ok) break;
        if (threadIdx.x == 0) {
#pragma unroll
          for (int k = 0; k < 2; ++k) {
            const uint32_t sk = k ? s1 : s0;
            uint8_t* Ak = stage + sk * C::kStage;
            mbar_expect_tx(&full[sk], 2 * C::kB);
            tma_load_2d(Ak + kATile, &tm_Vt, k * 64, 2 * s_rel[r_c] * D, &full[sk]);                // hi
            tma_load_2d(Ak + kATile + C::kB, &tm_Vt, k * 64, (2 * s_rel[r_c] + 1) * D, &full[sk]);  // lo
          }
        }
        // this lane's 16 bytes of row rho in its K chunk's stage
        const uint32_t A = stage_s + ((hl >> 3) ? s1 : s0) * C::kStage;
        auto put = [&](int rho, uint4 v) {
          asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(A + sw128_offset(rho, (hl & 7) * 16)),
                       "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                       : "memory");
        };
        // rows without gathers, by cp.async (awaited before the stages are released): a long row's
        // mean, or zeros
        uint8_t* Ag = stage + ((hl >> 3) ? s1 : s0) * C::kStage;
#pragma unroll
        for (int i = 0; i < kRowsPer; ++i) {
          const int rho = grp + kGrp * i;
          if (rho < kTileRows) {  // the same for the whole half
            const int rb = __shfl_sync(hmask, m_rb, hb + i), re = __shfl_sync(hmask, m_re, hb + i);
            const int slot = __shfl_sync(hmask, m_slot, hb + i);
            if (slot >= 0 || rb == re)
              cp_async16(Ag + sw128_offset(rho, (hl & 7) * 16), a.Mlong + (slot >= 0 ? (int64_t)slot * D + hl * 8 : 0),
                         slot >= 0);
          }
        }
        cp_async_commit();
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        int arow = -1;  // the row being summed
        auto flush = [&]() {
          const float sc = __shfl_sync(hmask, m_sc, hb + arow);
          put(grp + kGrp * arow,
              make_uint4(pack_bf16x2(acc[0] * sc, acc[1] * sc), pack_bf16x2(acc[2] * sc, acc[3] * sc),
                         pack_bf16x2(acc[4] * sc, acc[5] * sc), pack_bf16x2(acc[6] * sc, acc[7] * sc)));
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        };
        while ((srow & 0xFu) != 0xFu) {
          uint4 x[8];
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int c = __shfl_sync(hmask, v, hb + k);
            x[k] = ((srow >> (4 * k)) & 0xFu) != 0xFu ? ldg16(Hc + (int64_t)c * D) : make_uint4(0u, 0u, 0u, 0u);
          }
          // the next batch's run entries, in flight while this batch is added
          uint32_t nsrow;
          const int vn = fill(nsrow);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const int rk = (int)((srow >> (4 * k)) & 0xFu);
            if (rk == 0xF) break;
            if (rk != arow) {
              if (arow >= 0) flush();
              arow = rk;
            }
            const float w = (float)__shfl_sync(hmask, v, hb + 8 + k);
            float f[8];
            unpack(x[k], f, __nv_bfloat16());
#pragma unroll
            for (int q = 0; q < 8; ++q) acc[q] = fmaf(w, f[q], acc[q]);
          }
          srow = nsrow;
          v = vn;
        }
        if (arow >= 0) flush();
        cp_async_wait<0>();  // this thread's copies of the long rows and zero rows
        fence_async_smem();
        mbar_arrive(&full[s0]);
        mbar_arrive(&full[s1]);
        g += 2;
        __syncwarp();
        // the next relation tile
        r_c = r_n;
        tile_c = tile_n;
        m_rb = n_rb;
        m_re = n_re;
        m_slot = n_slot;
        m_sc = n_sc;
        r_n = r_nn;
        tile_n = tile_nn;
        j_n = j_nn;
      }
      if (!ok) {
        if (lane == 0) atomicOr(a.status, kErrTimeout);
        if (threadIdx.x == 0) drain_rounds(full, S, g);
      }
    }
  };
  auto plain_role = [&]() {
    // ---- producers.  Warp w fills rows 64 w .. 64 w + 63 of every A stage from M with cp.async:
    // one instruction copies four whole 128-byte row chunks (lane l: chunk l % 8 of row 4 k + l / 8),
    // into the 128B-swizzled layout the MMA reads; a row past the type or without a stored relation
    // row is zero-filled without a read.  Thread 0 also loads the stage's V_r^T hi / lo chunks by
    // TMA.  A thread releases a stage kLag stages after issuing it: once its own copies have landed
    // (wait_group) and are fenced for the async proxy, it arrives on the stage's barrier.  The
    // nodes of the tile after next and the rows of M of the next tile are loaded while a tile's
    // stages are issued.
    const int t = threadIdx.x;
    const int rbase = warp * 64;
    bool ok = true;
    uint32_t g = 0, done = 0;  // stages issued, stages released
    // nodes of this lane's two rows (rbase + lane, rbase + 32 + lane) of tile q
    auto nodes = [&](int64_t q, int64_t* j) {
#pragma unroll
      for (int h = 0; h < 2; ++h) j[h] = q < ntiles ? node_at(q * kTileRows + rbase + 32 * h + lane) : -1;
    };
    // rows of M of those nodes for each relation of tm (-1: zeros)
    auto mrows = [&](uint32_t tm, const int64_t* j, int32_t (*v)[2]) {
#pragma unroll
      for (int r = 0; r < kMaxRels; ++r)
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          int64_t x = -1;
          if (((tm >> r) & 1u) && j[h] >= 0)
            x = a.mrow ? (int64_t)__ldg(a.mrow + a.mrow0[r] + j[h]) : a.mrow0[r] + j[h];
          v[r][h] = x >= 0 && x < a.msent ? (int32_t)x : -1;
        }
    };
    int64_t tile = blockIdx.x;
    uint32_t tm_c = rels_of(tile), tm_n = rels_of(tile + G);
    int64_t j_c[2], j_n[2];
    int32_t v_c[kMaxRels][2];
    nodes(tile, j_c);
    nodes(tile + G, j_n);
    mrows(tm_c, j_c, v_c);
    for (; tile < ntiles && ok; tile += G) {
      int32_t v_n[kMaxRels][2];
      mrows(tm_n, j_n, v_n);  // the next tile's rows of M (its nodes were loaded a tile ago)
      const uint32_t tm_nn = rels_of(tile + 2 * G);
      int64_t j_nn[2];
      nodes(tile + 2 * G, j_nn);
#pragma unroll
      for (int r = 0; r < kMaxRels; ++r) {
        if (!((tm_c >> r) & 1u) || !ok) continue;
        int32_t vk[16];  // the row this lane copies in instruction k: 4 k + lane / 8
#pragma unroll
        for (int k = 0; k < 16; ++k) vk[k] = __shfl_sync(0xffffffffu, v_c[r][k >> 3], ((4 * k) & 31) + (lane >> 3));
        for (int kc = 0; kc < KC; ++kc, ++g) {
          const uint32_t s = g % S;
          if (g >= (uint32_t)S) ok = mbar_wait(&empty[s], ((g / S) - 1) & 1);
          if (!ok) break;
          uint8_t* A = stage + s * C::kStage;
          if (t == 0) {
            mbar_expect_tx(&full[s], 2 * C::kB);
            tma_load_2d(A + kATile, &tm_Vt, kc * 64, 2 * a.rel[r] * D, &full[s]);                // hi
            tma_load_2d(A + kATile + C::kB, &tm_Vt, kc * 64, (2 * a.rel[r] + 1) * D, &full[s]);  // lo
          }
          const int ch = lane & 7;
#pragma unroll
          for (int k = 0; k < 16; ++k) {
            const int rr = rbase + 4 * k + (lane >> 3);
            cp_async16(A + sw128_offset(rr, ch * 16), a.M + (int64_t)max(vk[k], 0) * D + kc * 64 + ch * 8, vk[k] >= 0);
          }
          cp_async_commit();
          if (g + 1 - done > kLag) {
            cp_async_wait<kLag>();
            fence_async_smem();
            mbar_arrive(&full[done % S]);
            ++done;
          }
        }
      }
      tm_c = tm_n;
      tm_n = tm_nn;
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        j_n[h] = j_nn[h];
#pragma unroll
        for (int r = 0; r < kMaxRels; ++r) v_c[r][h] = v_n[r][h];
      }
    }
    // Every stage issued is released, also on the give-up path: its phase can then complete, and
    // thread 0 waits (bounded) for the weight loads of each stage's last round before the CTA exits.
    cp_async_wait<0>();
    fence_async_smem();
    for (; done < g; ++done) mbar_arrive(&full[done % S]);
    if (!ok) {
      atomicOr(a.status, kErrTimeout);
      if (t == 0) drain_rounds(full, S, g);
    }
  };
  auto mma_role = [&]() {
    // ---- MMA issuer: U_tile = sum_r M_r V_r into accumulator (it & 1), over the tile's relations
    if (lane == 0) {
      const uint32_t idesc = idesc_bf16(128, D, false, false);
      bool ok = true;
      uint32_t g = 0;
      int it = 0;
      uint32_t tm_n = rels_of(blockIdx.x);
      for (int64_t tile = blockIdx.x; tile < ntiles && ok; tile += G, ++it) {
        const uint32_t tm = tm_n;
        tm_n = rels_of(tile + G);  // in flight during this tile
        const int b = it & 1;
        if (it >= 2) ok = mbar_wait(&acc_empty[b], ((it >> 1) - 1) & 1);
        if (!ok) break;
        fence_after_sync();
        const uint32_t acc = tmem + b * C::kAccCols;
        bool first = true;
        for (int r = 0; r < a.nrel && ok; ++r) {
          if (!((tm >> r) & 1u)) continue;
          for (int kc = 0; kc < KC; ++kc, ++g) {
            const uint32_t s = g % S;
            ok = mbar_wait(&full[s], (g / S) & 1);
            if (!ok) break;
            fence_after_sync();
            const uint32_t A = smem_u32(stage + s * C::kStage);
#pragma unroll
            for (int ks = 0; ks < 4; ++ks) {
              const uint64_t ad = desc_sw128(A + ks * 32, 16, 1024);
              mma_bf16(acc, ad, desc_sw128(A + kATile + ks * 32, 16, 1024), idesc, (first && ks == 0) ? 0u : 1u);
              mma_bf16(acc, ad, desc_sw128(A + kATile + C::kB + ks * 32, 16, 1024), idesc, 1u);
            }
            first = false;
            mma_commit(&empty[s]);
          }
        }
        if (!ok) break;
        if (tm != 0) {
          mma_commit(&acc_full[b]);
        } else {
          mbar_arrive(&acc_full[b]);  // no products: the epilogue reads no accumulator
        }
      }
      if (!ok) {
        atomicOr(a.status, kErrTimeout);
        drain_mma(drainb, 0);  // the MMAs issued so far complete before TMEM is released
      }
    }
    __syncwarp();
  };
  auto epi_role = [&]() {
    // ---- epilogue: bias, activation, residual, LayerNorm.  Warp w owns TMEM lanes 32 (w % 4) ..;
    // thread (row, half) handles columns kHalf * half .. + kHalf of its row; the two halves of a
    // row add their partial sums through shared memory (a barrier per pair of warps).
    const int q = warp & 3;
    const int hf = (warp - C::kEpiWarp0) >> 2;
    const int row = q * 32 + lane;
    const int c0 = hf * C::kHalf;
    const float* pb = params;
    const float* pgm = params + D;
    const float* pbe = params + 2 * D;
    for (int c = threadIdx.x - C::kEpiWarp0 * 32; c < D; c += C::kEpiThreads) {
      params[c] = __bfloat162float(a.b[c]);
      params[D + c] = a.ln ? __bfloat162float(a.gamma[c]) : 1.f;
      params[2 * D + c] = a.ln ? __bfloat162float(a.beta[c]) : 0.f;
    }
    asm volatile("bar.sync 1, %0;" ::"n"(C::kEpiThreads) : "memory");  // the epilogue warps
    const uint32_t pair_bar = 2 + q;  // warps q and q + 4 of the epilogue: the two halves of its rows
    // the row's total of v over both halves (the same sum, v0 + v1, in both threads)
    auto pair_sum = [&](float v, int which) -> float {
      red[(which * 2 + hf) * kTileRows + row] = v;
      asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory");
      return v + red[(which * 2 + (hf ^ 1)) * kTileRows + row];
    };
    // Row transfers between global memory and the warp's 32 rows (its column half) of a
    // 128B-swizzled tile: lane l moves 16-byte chunk l % kCh of row kRpi k + l / kCh, the row's
    // node taken from the lane that owns it.
    constexpr int kCh = C::kHalf / 8, kRpi = 32 / kCh;
    auto chunk_at = [&](uint8_t* t, int rr, int ch) {  // rr: row within the warp's 32
      const int cg = hf * kCh + ch;                     // chunk within the full row
      return t + (cg >> 3) * kATile + sw128_offset(q * 32 + rr, (cg & 7) * 16);
    };
    // the residual of the warp's rows (nodes jw, per lane) into buffer hb; one commit group per call
    auto fetch_h = [&](int64_t jw, int hb) {
      if constexpr (C::kHTile) {
        uint8_t* t = htile + hb * C::kH;
#pragma unroll
        for (int k = 0; k < 32 / kRpi; ++k) {
          const int rr = kRpi * k + lane / kCh, ch = lane % kCh;
          const int64_t jj = __shfl_sync(0xffffffffu, jw, rr);
          if (jj >= 0) cp_async16(chunk_at(t, rr, ch), a.H_in + (a.off + jj) * D + c0 + ch * 8, true);
        }
        cp_async_commit();
      }
    };
    // the warp's rows of tile buffer t to out (the rows of nodes jw)
    auto store_rows = [&](uint8_t* t, int64_t jw, __nv_bfloat16* out) {
#pragma unroll
      for (int k = 0; k < 32 / kRpi; ++k) {
        const int rr = kRpi * k + lane / kCh, ch = lane % kCh;
        const int64_t jj = __shfl_sync(0xffffffffu, jw, rr);
        if (jj >= 0) st16(out + (a.off + jj) * D + c0 + ch * 8, *reinterpret_cast<const uint4*>(chunk_at(t, rr, ch)));
      }
    };
    bool ok = true;
    int it = 0;
    int64_t j_c = node_at((int64_t)blockIdx.x * kTileRows + row);  // this tile's node at the row
    int64_t j_n = node_at(((int64_t)blockIdx.x + G) * kTileRows + row);  // the next tile's
    bool has_n = rels_of(blockIdx.x) != 0;
    fetch_h(j_c, 0);
    for (int64_t tile = blockIdx.x; tile < ntiles && ok; tile += G, ++it) {
      const int b = it & 1;
      const int64_t j = j_c;
      const bool live = j >= 0;
      const int64_t node = a.off + (live ? j : 0);
      const bool has = has_n;  // else U = 0 without an accumulator
      has_n = rels_of(tile + G) != 0;
      fetch_h(j_n, b ^ 1);  // the next tile's residual rows, in flight during this tile
      const int64_t j_nn = node_at((tile + 2 * G) * kTileRows + row);
      ok = mbar_wait(&acc_full[b], (it >> 1) & 1);
      ok = bar_and(pair_bar, 64, ok);  // both halves of a row give up together (no lone pair barrier)
      if (!ok) break;
      fence_after_sync();
      if constexpr (C::kHTile) {
        cp_async_wait<1>();  // this tile's residual rows have landed (this lane's copies) ...
        __syncwarp();        // ... and the other lanes'
      }
      const uint32_t trow = tmem + b * C::kAccCols + ((uint32_t)(q * 32) << 16);
      uint8_t* ht = htile + b * C::kH;
      // U_s = bf16(acc) for columns c .. c+15 (acc already in u when preloaded), stored to global
      // memory when store_g; returned as U_s + b in u, and packed in up
      auto u16 = [&](int c, float* u, uint32_t* up, bool store_g, bool preloaded = false) {
        if (!preloaded) {
          if (has) {
            tmem_ld16(trow + c, u);
          } else {
#pragma unroll
            for (int i = 0; i < 16; ++i) u[i] = 0.f;
          }
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) up[i] = pack_bf16x2(u[2 * i], u[2 * i + 1]);
        if (store_g && live) {
          st16(a.U + node * D + c, make_uint4(up[0], up[1], up[2], up[3]));
          st16(a.U + node * D + c + 8, make_uint4(up[4], up[5], up[6], up[7]));
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          u[2 * i] = __uint_as_float(up[i] << 16) + pb[c + 2 * i];
          u[2 * i + 1] = __uint_as_float(up[i] & 0xFFFF0000u) + pb[c + 2 * i + 1];
        }
      };
      auto h16 = [&](int c, float* h) {  // residual row, columns c .. c+15
        if constexpr (C::kHTile) {  // from the 128B-swizzled tile
          const uint8_t* t = ht + (c >> 6) * kATile;
          const uint32_t cb = (uint32_t)(c & 63) * 2;
          unpack(*reinterpret_cast<const uint4*>(t + sw128_offset(row, cb)), h, __nv_bfloat16());
          unpack(*reinterpret_cast<const uint4*>(t + sw128_offset(row, cb + 16)), h + 8, __nv_bfloat16());
        } else {
          load16_bf16(a.H_in + node * D + c, h);
        }
      };
      auto put16 = [&](int c, const uint32_t* up) {  // 16 packed columns into this thread's tile row
        uint8_t* t = ht + (c >> 6) * kATile;
        const uint32_t cb = (uint32_t)(c & 63) * 2;
        *reinterpret_cast<uint4*>(t + sw128_offset(row, cb)) = make_uint4(up[0], up[1], up[2], up[3]);
        *reinterpret_cast<uint4*>(t + sw128_offset(row, cb + 16)) = make_uint4(up[4], up[5], up[6], up[7]);
      };
      auto out16 = [&](int c, const float* y, float mean, float rstd, uint32_t* up) {  // H_out, c .. c+15
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          const int k0 = 2 * i, k1 = k0 + 1;
          const float o0 = a.ln ? (y[k0] - mean) * rstd * pgm[c + k0] + pbe[c + k0] : y[k0];
          const float o1 = a.ln ? (y[k1] - mean) * rstd * pgm[c + k1] + pbe[c + k1] : y[k1];
          up[i] = pack_bf16x2(o0, o1);
        }
      };
      if constexpr (C::kHTile) {
        // the half row in registers: one pass over TMEM.  U_s replaces the residual in the tile row
        // once read, then H_out; each leaves as whole row chunks per instruction.
        float y[C::kHalf];
        float sum = 0.f;
#pragma unroll
        for (int cc = 0; cc < C::kHalf; cc += 32) {
          float u[32];
          if (has) {
            tmem_ld32(trow + c0 + cc, u);
          } else {
#pragma unroll
            for (int i = 0; i < 32; ++i) u[i] = 0.f;
          }
#pragma unroll
          for (int hh = 0; hh < 32; hh += 16) {
            float h[16];
            uint32_t up[8];
            h16(c0 + cc + hh, h);
            u16(c0 + cc + hh, u + hh, up, false, true);
            put16(c0 + cc + hh, up);
#pragma unroll
            for (int i = 0; i < 16; ++i) {
              y[cc + hh + i] = act_apply(u[hh + i], a.act) + h[i];
              sum += y[cc + hh + i];
            }
          }
        }
        fence_before_sync();
        mbar_arrive(&acc_empty[b]);  // the accumulator is read: the MMAs of tile it + 2 may start
        __syncwarp();
        store_rows(ht, j, a.U);
        const float mean = pair_sum(sum, 0) * (1.f / D);
        float qq = 0.f;
#pragma unroll
        for (int i = 0; i < C::kHalf; ++i) qq += (y[i] - mean) * (y[i] - mean);
        const float rstd = rsqrtf(pair_sum(qq, 1) * (1.f / D) + a.eps);
        __syncwarp();  // every lane has read U_s from the tile
#pragma unroll
        for (int cc = 0; cc < C::kHalf; cc += 16) {
          uint32_t up[8];
          out16(c0 + cc, y + cc, mean, rstd, up);
          put16(c0 + cc, up);
        }
        __syncwarp();
        store_rows(ht, j, a.H_out);
        if (a.ln && live && hf == 0) a.stats[node] = make_float2(mean, rstd);
        __syncwarp();  // the tile buffer is refilled two tiles on
      } else {
        // three passes over TMEM and the residual (row sum, centred sum of squares, output)
        auto y16 = [&](int c, float* y, bool store) {
          float u[16], h[16];
          uint32_t up[8];
          u16(c, u, up, store);
          h16(c, h);
#pragma unroll
          for (int i = 0; i < 16; ++i) y[i] = act_apply(u[i], a.act) + h[i];
        };
        float sum = 0.f;
#pragma unroll 1
        for (int cc = 0; cc < C::kHalf; cc += 16) {
          float y[16];
          y16(c0 + cc, y, true);
#pragma unroll
          for (int i = 0; i < 16; ++i) sum += y[i];
        }
        const float mean = pair_sum(sum, 0) * (1.f / D);
        float qq = 0.f;
#pragma unroll 1
        for (int cc = 0; cc < C::kHalf; cc += 16) {
          float y[16];
          y16(c0 + cc, y, false);
#pragma unroll
          for (int i = 0; i < 16; ++i) qq += (y[i] - mean) * (y[i] - mean);
        }
        const float rstd = rsqrtf(pair_sum(qq, 1) * (1.f / D) + a.eps);
#pragma unroll 1
        for (int cc = 0; cc < C::kHalf; cc += 16) {
          float y[16];
          uint32_t up[8];
          y16(c0 + cc, y, false);
          out16(c0 + cc, y, mean, rstd, up);
          if (live) {
            st16(a.H_out + node * D + c0 + cc, make_uint4(up[0], up[1], up[2], up[3]));
            st16(a.H_out + node * D + c0 + cc + 8, make_uint4(up[4], up[5], up[6], up[7]));
          }
        }
        if (a.ln && live && hf == 0) a.stats[node] = make_float2(mean, rstd);
        fence_before_sync();
        mbar_arrive(&acc_empty[b]);
      }
      j_c = j_n;
      j_n = j_nn;
    }
    if constexpr (C::kHTile) cp_async_wait<0>();  // no residual copy outlives the kernel
    if (!ok) atomicOr(a.status, kErrTimeout);
  };
  if constexpr (kGather) {
    // warpgroups 0-1 (the gather warps and the MMA warp) give registers to 2-3 (the epilogue)
    if (warp < 8) {
      setmaxnreg_dec<C::kLowRegs>();
      if (warp == C::kMmaWarp) {
        mma_role();
      } else {
        gather_role();
      }
    } else {
      setmaxnreg_inc<C::kHighRegs>();
      epi_role();
    }
  } else {
    if (warp < C::kMmaWarp) {
      plain_role();
    } else if (warp == C::kMmaWarp) {
      mma_role();
    } else {
      epi_role();
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == C::kMmaWarp) tmem_dealloc(tmem, C::kTmemCols);
}

template <int D>
__global__ void __launch_bounds__(FwdCfg<D>::kThreads, 1)
    proj_fwd_tc(const __grid_constant__ CUtensorMap tm_Vt, TcFwdArgs a) {
  proj_fwd_body<D, false>(tm_Vt, a);
}

template <int D>
__global__ void __launch_bounds__(FwdCfg<D, true>::kThreads, 1)
    proj_fwd_gather_tc(const __grid_constant__ CUtensorMap tm_Vt, TcFwdArgs a) {
  if constexpr (D == 128) proj_fwd_body<D, true>(tm_Vt, a);
}

// Fused weights V_r = W_r W_agg[t_r] accumulated in fp64 (exact for bf16 factors of these sizes),
// written as the pair V_hi = bf16(V_r), V_lo = bf16(V_r - V_hi): V holds [relation][hi, lo][D][D]
// and Vt the transposes in the same order.  Grid (D/32, D/32, relations): a
// block computes a 32 x 32 tile from 32-wide K slices staged in shared memory; thread (ty, tx)
// owns rows ty, ty + 8, ty + 16, ty + 24 of column tx.
template <int D>
__global__ void __launch_bounds__(256) fuse_weights(const __nv_bfloat16* __restrict__ W_rel,
                                                    const __nv_bfloat16* __restrict__ W_agg, RelDst rel_dst,
                                                    int num_rels, __nv_bfloat16* __restrict__ V,
                                                    __nv_bfloat16* __restrict__ Vt) {
  __shared__ double As[32][33];
  __shared__ double Bs[32][33];
  const int r = blockIdx.z, i0 = blockIdx.y * 32, j0 = blockIdx.x * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  const __nv_bfloat16* W = W_rel + (int64_t)r * D * D;
  const __nv_bfloat16* G = W_agg + (int64_t)rel_dst.v[r] * D * D;
  double acc[4] = {0.0, 0.0, 0.0, 0.0};
  for (int k0 = 0; k0 < D; k0 += 32) {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      const int rr = ty + 8 * q;
      As[rr][tx] = (double)__bfloat162float(W[(int64_t)(i0 + rr) * D + k0 + tx]);
      Bs[rr][tx] = (double)__bfloat162float(G[(int64_t)(k0 + rr) * D + j0 + tx]);
    }
    __syncthreads();
#pragma unroll 8
    for (int k = 0; k < 32; ++k) {
      const double bv = Bs[k][tx];
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[q] = fma(As[ty + 8 * q][k], bv, acc[q]);
    }
    __syncthreads();
  }
#pragma unroll
  for (int q = 0; q < 4; ++q) {
    const int i = i0 + ty + 8 * q, j = j0 + tx;
    const __nv_bfloat16 hi = __float2bfloat16_rn(__double2float_rn(acc[q]));
    const __nv_bfloat16 lo = __float2bfloat16_rn(__double2float_rn(acc[q] - (double)__bfloat162float(hi)));
    const int64_t base = (int64_t)2 * r * D * D;
    V[base + (int64_t)i * D + j] = hi;
    V[base + (int64_t)D * D + (int64_t)i * D + j] = lo;
    Vt[base + (int64_t)j * D + i] = hi;
    Vt[base + (int64_t)D * D + (int64_t)j * D + i] = lo;
  }
}

// dW_r = G_r W_agg[t_r]^T and dW_agg[t] = sum over r -> t (ascending) of W_r^T G_r, fp32, where
// G_r = M_r^T dU_{t_r}; types without relations get zero.  Grid (D/32, D/32, relations + types),
// 32 x 32 output tiles from 32-wide K slices in shared memory (thread layout as fuse_weights).
template <int D>
__global__ void __launch_bounds__(256) wgrad_finish(const float* __restrict__ G, const __nv_bfloat16* __restrict__ W_rel,
                                                    const __nv_bfloat16* __restrict__ W_agg, RelDst rel_dst,
                                                    int num_rels, int num_types, float* __restrict__ dW_rel,
                                                    float* __restrict__ dW_agg) {
  __shared__ float As[32][33];
  __shared__ float Bs[32][33];
  const int z = blockIdx.z, i0 = blockIdx.y * 32, j0 = blockIdx.x * 32;
  const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
  float acc[4] = {0.f, 0.f, 0.f, 0.f};
  auto mac = [&]() {
#pragma unroll 8
    for (int k = 0; k < 32; ++k) {
      const float bv = Bs[k][tx];
#pragma unroll
      for (int q = 0; q < 4; ++q) acc[q] = fmaf(As[ty + 8 * q][k], bv, acc[q]);
    }
  };
  if (z < num_rels) {  // dW_r[i][j] = sum_k G_r[i][k] W_agg[t][j][k]
    const float* Gr = G + (int64_t)z * D * D;
    const __nv_bfloat16* Wa = W_agg + (int64_t)rel_dst.v[z] * D * D;
    for (int k0 = 0; k0 < D; k0 += 32) {
#pragma unroll
      for (int q = 0; q < 4; ++q) {
        const int rr = ty + 8 * q;
        As[rr][tx] = Gr[(int64_t)(i0 + rr) * D + k0 + tx];
        Bs[tx][rr] = __bfloat162float(Wa[(int64_t)(j0 + rr) * D + k0 + tx]);
      }
      __syncthreads();
      mac();
      __syncthreads();
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) dW_rel[(int64_t)z * D * D + (int64_t)(i0 + ty + 8 * q) * D + j0 + tx] = acc[q];
  } else {  // dW_agg[t][i][j] = sum_{r -> t} sum_k W_r[k][i] G_r[k][j]
    const int t = z - num_rels;
    for (int r = 0; r < num_rels; ++r) {
      if (rel_dst.v[r] != t) continue;
      const __nv_bfloat16* Wr = W_rel + (int64_t)r * D * D;
      const float* Gr = G + (int64_t)r * D * D;
      for (int k0 = 0; k0 < D; k0 += 32) {
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          const int rr = ty + 8 * q;
          As[tx][rr] = __bfloat162float(Wr[(int64_t)(k0 + rr) * D + i0 + tx]);
          Bs[rr][tx] = Gr[(int64_t)(k0 + rr) * D + j0 + tx];
        }
        __syncthreads();
        mac();
        __syncthreads();
      }
    }
#pragma unroll
    for (int q = 0; q < 4; ++q) dW_agg[(int64_t)t * D * D + (int64_t)(i0 + ty + 8 * q) * D + j0 + tx] = acc[q];
  }
}

// ln_act_bwd: rows per warp whose loads are in flight together, and resident blocks per SM (the
// register budget that keeps them without spills)
template <int D>
struct LnCfg {
  static constexpr int kRows = D == 256 ? 2 : (D == 128 ? 3 : 4);
  static constexpr int kBlocks = D == 256 ? 1 : (D == 128 ? 3 : 4);
};

// LayerNorm / activation backward, one warp per row (coalesced rows, D / 32 columns per lane):
// U = stored U_s + b (as in the forward), dY = rstd (dXh - mean(dXh) - Xh mean(dXh Xh)),
// dXh = dH_out gamma, dU = dY act'(U); per-block
// column partials part[block] = {sum dU, sum dH_out Xh, sum dH_out} over the block's rows.
template <int D>
__global__ void __launch_bounds__(256, LnCfg<D>::kBlocks) ln_act_bwd(TcBwdArgs a) {
  constexpr int E = D / 32;
  constexpr int kLnRows = LnCfg<D>::kRows;
  __shared__ float red[8][3][D];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int c0 = lane * E;
  float g[E], bias[E];
#pragma unroll
  for (int i = 0; i < E; ++i) {
    g[i] = a.ln ? __bfloat162float(a.gamma[c0 + i]) : 1.f;
    bias[i] = __bfloat162float(a.b[c0 + i]);
  }
  float pdb[E], pdg[E], pdbe[E];
#pragma unroll
  for (int i = 0; i < E; ++i) pdb[i] = pdg[i] = pdbe[i] = 0.f;
  auto store = [&](__nv_bfloat16* p, const float* v) {
    if constexpr (E == 2) {
      *reinterpret_cast<uint32_t*>(p) = pack_bf16x2(v[0], v[1]);
    } else if constexpr (E == 4) {
      *reinterpret_cast<uint2*>(p) = make_uint2(pack_bf16x2(v[0], v[1]), pack_bf16x2(v[2], v[3]));
    } else {
      st16(p, pack(v, __nv_bfloat16()));
    }
  };
  // kLnRows rows per iteration: all their loads are in flight before any is computed (held as the
  // raw bf16 words, E / 2 registers per tensor and row)
  using Raw = typename std::conditional<E == 2, uint32_t, typename std::conditional<E == 4, uint2, uint4>::type>::type;
  auto unpack_raw = [&](const Raw& w, float* v) {
    if constexpr (E == 2) {
      v[0] = __uint_as_float(w << 16);
      v[1] = __uint_as_float(w & 0xFFFF0000u);
    } else if constexpr (E == 4) {
      v[0] = __uint_as_float(w.x << 16);
      v[1] = __uint_as_float(w.x & 0xFFFF0000u);
      v[2] = __uint_as_float(w.y << 16);
      v[3] = __uint_as_float(w.y & 0xFFFF0000u);
    } else {
      unpack(w, v, __nv_bfloat16());
    }
  };
  const int64_t step = (int64_t)gridDim.x * 8;
  for (int64_t row0 = (int64_t)blockIdx.x * 8 + warp; row0 < a.n; row0 += kLnRows * step) {
    Raw rd[kLnRows], ru[kLnRows], rh[kLnRows];
    float2 st[kLnRows];
#pragma unroll
    for (int k = 0; k < kLnRows; ++k) {
      const int64_t row = row0 + k * step;
      const int64_t o = (a.off + (row < a.n ? row : row0)) * D + c0;
      rd[k] = *reinterpret_cast<const Raw*>(a.dH_out + o);
      ru[k] = *reinterpret_cast<const Raw*>(a.U + o);
      rh[k] = *reinterpret_cast<const Raw*>(a.H_in + o);
      st[k] = a.ln ? a.stats[a.off + (row < a.n ? row : row0)] : make_float2(0.f, 1.f);
    }
#pragma unroll
    for (int k = 0; k < kLnRows; ++k) {
      const int64_t row = row0 + k * step;
      if (row >= a.n) continue;
      float dv[E], uv[E], hv[E], dy[E], du[E], xh[E];
      unpack_raw(rd[k], dv);
      unpack_raw(ru[k], uv);
      unpack_raw(rh[k], hv);
#pragma unroll
      for (int i = 0; i < E; ++i) uv[i] += bias[i];
      if (a.ln) {
        float s1 = 0.f, s2 = 0.f;
#pragma unroll
        for (int i = 0; i < E; ++i) {
          xh[i] = (act_apply(uv[i], a.act) + hv[i] - st[k].x) * st[k].y;
          const float dxh = dv[i] * g[i];
          s1 += dxh;
          s2 += dxh * xh[i];
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          s1 += __shfl_xor_sync(0xffffffffu, s1, o);
          s2 += __shfl_xor_sync(0xffffffffu, s2, o);
        }
        const float mean1 = s1 * (1.f / D), mean2 = s2 * (1.f / D);
#pragma unroll
        for (int i = 0; i < E; ++i) dy[i] = st[k].y * (dv[i] * g[i] - mean1 - xh[i] * mean2);
      } else {
#pragma unroll
        for (int i = 0; i < E; ++i) {
          dy[i] = dv[i];
          xh[i] = 0.f;
        }
      }
#pragma unroll
      for (int i = 0; i < E; ++i) {
        du[i] = __bfloat162float(__float2bfloat16_rn(dy[i] * act_grad(uv[i], a.act)));
        pdb[i] += du[i];
        pdg[i] += dv[i] * xh[i];
        pdbe[i] += dv[i];
      }
      const int64_t o = (a.off + row) * D + c0;
      store(a.dY + o, dy);
      store(a.dU + o, du);
    }
  }
#pragma unroll
  for (int i = 0; i < E; ++i) {
    red[warp][0][c0 + i] = pdb[i];
    red[warp][1][c0 + i] = pdg[i];
    red[warp][2][c0 + i] = pdbe[i];
  }
  __syncthreads();
  for (int k = threadIdx.x; k < 3 * D; k += blockDim.x) {
    const int q = k / D, c = k % D;
    float s = 0.f;
#pragma unroll
    for (int w = 0; w < 8; ++w) s += red[w][q][c];
    a.part[((int64_t)blockIdx.x * 3 + q) * D + c] = s;
  }
}

// ---------------------------------------------------------------------------------------------
// backward, row side
// ---------------------------------------------------------------------------------------------
template <int D>
struct BwdCfg {
  static constexpr int kStages = D == 64 ? 4 : (D == 128 ? 3 : 2);  // ring of V_r chunks (hi and lo)
  static constexpr int kB = D * 128;                    // D rows x 64 columns, one half of the pair
  static constexpr int kBStage = 2 * kB;
  static constexpr int kT = kTileRows * D * 2;          // gathered dU operand tile (KC x 16 KB)
  static constexpr int kABuf = D == 256 ? 1 : 2;        // dU tiles in flight (shared memory allowing)
  static constexpr int kAcc = D < 32 ? 32 : D;
  static constexpr int kNumAcc = 512 / kAcc < 4 ? 512 / kAcc : 4;  // ring of TMEM accumulators
  static constexpr int kTmemCols = kNumAcc * kAcc;
  static constexpr int kEpiGroups = 2;  // epilogue warp groups, taking alternate accumulators
  static constexpr int kIdx = kTileRows * 4;
  static constexpr int kSmem = kStages * kBStage + kABuf * kT + kIdx + 512 + 1024;
  static constexpr int kThreads = 64 + kEpiGroups * 128;
  static_assert(kSmem <= 227 * 1024, "shared memory of proj_bwd_tc");
};

// one tensor map per relation (used by the weight-gradient kernel's operands)
struct RelMaps {
  CUtensorMap m[kMaxRels];
};

// The jobs of proj_bwd_tc: 128 rows of one relation's stored rows each, relation by relation.
struct BwdJobs {
  int nrel;
  int64_t base[kMaxRels];   // first stored row of relation j (compact index, or 0 by CSR row)
  int64_t count[kMaxRels];  // its stored rows
  int64_t first[kMaxRels + 1];  // first job of relation j; first[nrel] = the number of jobs
  __device__ __forceinline__ void init(const TcBwdArgs& a) {  // one thread
    nrel = a.nrel;
    first[0] = 0;
    for (int j = 0; j < a.nrel; ++j) {
      base[j] = a.mlist ? (int64_t)a.mbase[a.rel[j]] : 0;
      count[j] = a.mlist ? (int64_t)a.mbase[a.rel[j] + 1] - base[j] : a.n;
      first[j + 1] = first[j] + (count[j] + kTileRows - 1) / kTileRows;
    }
  }
  __device__ __forceinline__ int rel_of(int64_t job) const {
    int j = 0;
    while (j + 1 < nrel && job >= first[j + 1]) ++j;
    return j;
  }
};

// dMs_r = (dU V_r^T) / deg_r for the stored rows of every relation r into this type (the non-empty
// CSR rows, in compact order; or every CSR row without a compact list).  Persistent, one CTA per
// SM, one job = 128 stored rows of one relation: warp 0 gathers the rows' dU (TMA gathers by the
// rows' destination nodes) and streams V_r chunks (hi and lo halves), warp 1 issues the job's MMA
// chain into a ring of TMEM accumulators, and two groups of four warps (2-5, 6-9) scale alternate
// jobs by 1/deg and store them, so the stores of one job overlap the products of the next.
template <int D>
__global__ void __launch_bounds__(BwdCfg<D>::kThreads, 1)
    proj_bwd_tc(const __grid_constant__ CUtensorMap tm_dU, const __grid_constant__ CUtensorMap tm_V, TcBwdArgs a) {
  using C = BwdCfg<D>;
  constexpr int S = C::kStages;
  constexpr int NB = C::kNumAcc;
  constexpr int NA = C::kABuf;
  constexpr int KC = D / 64;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint8_t* bstage = smem;                  // S x (B_hi | B_lo) chunk
  uint8_t* tiles = smem + S * C::kBStage;  // NA x (KC x 16 KB)
  uint64_t* b_full = reinterpret_cast<uint64_t*>(tiles + NA * C::kT + C::kIdx);
  uint64_t* b_empty = b_full + S;
  uint64_t* a_full = b_empty + S;       // [NA] dU tile gathered
  uint64_t* a_empty = a_full + 2;       // [NA] the job's products done
  uint64_t* acc_full = a_empty + 2;     // [NB]
  uint64_t* acc_empty = acc_full + NB;  // [NB]
  uint64_t* drainb = acc_empty + NB;    // the MMA issuer's give-up path
  uint32_t* tslot = reinterpret_cast<uint32_t*>(drainb + 1);

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  __shared__ BwdJobs J;
  if (threadIdx.x == 0) {
    J.init(a);
    for (int s = 0; s < S; ++s) {
      mbar_init(&b_full[s], 1);
      mbar_init(&b_empty[s], 1);
    }
    for (int b = 0; b < NA; ++b) {
      mbar_init(&a_full[b], 1);
      mbar_init(&a_empty[b], 1);
    }
    for (int k = 0; k < NB; ++k) {
      mbar_init(&acc_full[k], 1);
      mbar_init(&acc_empty[k], kTileRows);
    }
    mbar_init(drainb, 1);
    fence_mbar_init();
    prefetch_tmap(&tm_dU);
    prefetch_tmap(&tm_V);
  }
  if (warp == 1) tmem_alloc(tslot, C::kTmemCols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  const int64_t njobs = J.first[J.nrel];

  if (warp == 0) {  // ---- producer: lane q gathers the job's dU rows 4q .. 4q + 3, lane 0 streams V_r
    bool ok = true;
    uint32_t g = 0, a_issued = 0;
    int it = 0;
    for (int64_t job = blockIdx.x; job < njobs && ok; job += gridDim.x, ++it) {
      const int j = J.rel_of(job);
      const int64_t i0 = (job - J.first[j]) * kTileRows;  // first row of the job within the relation
      int c[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int64_t k = i0 + 4 * lane + i;
        int64_t local = a.n;  // past the relation's rows: zeros
        if (k < J.count[j]) local = a.mlist ? (int64_t)__ldg(a.mlist + J.base[j] + k) - a.mrow0[j] : k;
        c[i] = (int)local;
      }
      const int ab = it % NA;
      if (lane == 0) {
        if (it >= NA) ok = mbar_wait(&a_empty[ab], ((it / NA) - 1) & 1);
        if (ok) mbar_expect_tx(&a_full[ab], C::kT);
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
      if (ok) {
        uint8_t* A = tiles + ab * C::kT;
        for (int kc = 0; kc < KC; ++kc)
          tma_gather4(A + kc * kATile + lane * 512, &tm_dU, kc * 64, c[0], c[1], c[2], c[3], &a_full[ab]);
        ++a_issued;
      }
      if (lane == 0) {
        for (int kc = 0; kc < KC && ok; ++kc, ++g) {
          const uint32_t s = g % S;
          if (g >= (uint32_t)S) ok = mbar_wait(&b_empty[s], ((g / S) - 1) & 1);
          if (!ok) break;
          mbar_expect_tx(&b_full[s], C::kBStage);
          tma_load_2d(bstage + s * C::kBStage, &tm_V, kc * 64, 2 * a.rel[j] * D, &b_full[s]);
          tma_load_2d(bstage + s * C::kBStage + C::kB, &tm_V, kc * 64, (2 * a.rel[j] + 1) * D, &b_full[s]);
        }
      }
      ok = __shfl_sync(0xffffffffu, ok, 0);
    }
    if (lane == 0 && !ok) {
      atomicOr(a.status, kErrTimeout);
      drain_rounds(a_full, NA, a_issued);  // no gather or weight load still writes shared memory
      drain_rounds(b_full, S, g);
    }
    __syncwarp();
  } else if (warp == 1) {
    if (lane == 0) {  // ---- MMA issuer: one chain per job into accumulator (job count mod NB)
      const uint32_t idesc = idesc_bf16(128, D, false, false);
      bool ok = true;
      uint32_t g = 0, jb = 0;
      int it = 0;
      for (int64_t job = blockIdx.x; job < njobs && ok; job += gridDim.x, ++it, ++jb) {
        const int ab = it % NA;
        ok = mbar_wait(&a_full[ab], (it / NA) & 1);
        if (!ok) break;
        const uint32_t k = jb % NB;
        if (jb >= (uint32_t)NB) ok = mbar_wait(&acc_empty[k], ((jb / NB) - 1) & 1);
        if (!ok) break;
        fence_after_sync();
        const uint32_t acc = tmem + k * C::kAcc;
        const uint32_t A0 = smem_u32(tiles + ab * C::kT);
        for (int kc = 0; kc < KC && ok; ++kc, ++g) {
          const uint32_t s = g % S;
          ok = mbar_wait(&b_full[s], (g / S) & 1);
          if (!ok) break;
          fence_after_sync();
          const uint32_t A = A0 + kc * kATile;
          const uint32_t B = smem_u32(bstage + s * C::kBStage);
#pragma unroll
          for (int ks = 0; ks < 4; ++ks) {
            const uint64_t ad = desc_sw128(A + ks * 32, 16, 1024);
            mma_bf16(acc, ad, desc_sw128(B + ks * 32, 16, 1024), idesc, (kc > 0 || ks > 0) ? 1u : 0u);
            mma_bf16(acc, ad, desc_sw128(B + C::kB + ks * 32, 16, 1024), idesc, 1u);
          }
          mma_commit(&b_empty[s]);
        }
        mma_commit(&acc_full[k]);
        mma_commit(&a_empty[ab]);
      }
      if (!ok) {
        atomicOr(a.status, kErrTimeout);
        drain_mma(drainb, 0);
      }
    }
    __syncwarp();
  } else {  // ---- epilogue: scale by 1 / deg_r and store the job's dMs rows
    const int q = warp & 3;
    const int row = q * 32 + lane;
    const uint32_t grp = (uint32_t)(warp - 2) / 4;  // this group takes jobs jb = grp mod kEpiGroups
    bool ok = true;
    uint32_t jb = 0;
    for (int64_t job = blockIdx.x; job < njobs && ok; job += gridDim.x, ++jb) {
      if (jb % C::kEpiGroups != grp) continue;
      const int j = J.rel_of(job);
      const int64_t kr = (job - J.first[j]) * kTileRows + row;  // row within the relation's stored rows
      const bool live = kr < J.count[j];
      const int64_t crow = !live ? 0 : (a.mlist ? (int64_t)a.mlist[J.base[j] + kr] : a.mrow0[j] + kr);
      const int64_t out = a.mlist ? J.base[j] + kr : crow;  // compact row, or CSR row
      const int deg = live && a.csr_ptr ? a.csr_ptr[crow + 1] - a.csr_ptr[crow] : 0;
      const float sc = !a.csr_ptr ? 1.f : (deg > 0 ? __fdiv_rn(1.0f, (float)deg) : 0.f);
      const uint32_t k = jb % NB;
      ok = mbar_wait(&acc_full[k], (jb / NB) & 1);
      if (!ok) break;
      fence_after_sync();
      const uint32_t trow = tmem + k * C::kAcc + ((uint32_t)(q * 32) << 16);
#pragma unroll
      for (int c = 0; c < D; c += 32) {
        float v[32];
        tmem_ld32(trow + c, v);
#pragma unroll
        for (int i = 0; i < 32; ++i) v[i] *= sc;
        if (live) {
          store16_bf16(a.dMs + out * D + c, v);
          store16_bf16(a.dMs + out * D + c + 16, v + 16);
        }
      }
      fence_before_sync();
      mbar_arrive(&acc_empty[k]);
    }
    if (!ok) atomicOr(a.status, kErrTimeout);
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 1) tmem_dealloc(tmem, C::kTmemCols);
}

// ---------------------------------------------------------------------------------------------
// weight gradients: part[split][i][j] = sum over the split's rows k of X[k][i] Y[k][j]
// ---------------------------------------------------------------------------------------------
template <int D>
struct WgCfg {
  static constexpr int kA = 2 * 8192;                  // 64 rows x 128 columns (two 64-wide blocks)
  static constexpr int kB = (D < 64 ? 64 : D) * 128;   // 64 rows x D columns
  static constexpr int kAcc = D;                       // TMEM columns of one accumulator
  static constexpr int kMaxR = D == 64 ? 5 : (D == 128 ? 4 : 2);  // relations per launch
  static constexpr int kSmem = 227 * 1024;             // stages sized at run time within this
  static constexpr int kThreads = 128;
};

// G_r = X_r^T Y for up to kMaxR relations r that share the operand Y (the dU rows of their common
// destination type; X_r = the relation means M_r): each 64-row chunk of Y is loaded once and used
// by the MMAs of every relation, each accumulating into its own TMEM region.  Grid (M tiles of 128
// output rows, splits); part[r][split][D][D].
template <int D>
__global__ void __launch_bounds__(WgCfg<D>::kThreads, 1)
    wgrad_tc(const __grid_constant__ RelMaps tm_X, const __grid_constant__ CUtensorMap tm_Y, int R, int S,
             int64_t n, int chunks_per_split, float* __restrict__ part, int* __restrict__ status) {
  using C = WgCfg<D>;
  constexpr int NB = D / 64;  // 64-wide column blocks of Y
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  const int stage_bytes = R * C::kA + NB * 8192;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * stage_bytes);
  uint64_t* empty = full + S;
  uint64_t* accb = empty + S;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x;  // 128-wide block of X's columns (output rows)
  const int64_t nchunks = (n + 63) / 64;
  const int64_t c0 = (int64_t)blockIdx.y * chunks_per_split;
  const int64_t c1 = min(nchunks, c0 + chunks_per_split);
  const int CT = (int)max((int64_t)0, c1 - c0);
  uint32_t ncols = 32;
  while (ncols < (uint32_t)(R * C::kAcc)) ncols <<= 1;
  if (threadIdx.x == 0) {
    for (int st = 0; st < S; ++st) {
      mbar_init(&full[st], 1);
      mbar_init(&empty[st], 1);
    }
    mbar_init(accb, 1);
    fence_mbar_init();
    for (int r = 0; r < R; ++r) prefetch_tmap(&tm_X.m[r]);
    prefetch_tmap(&tm_Y);
  }
  if (warp == 0) tmem_alloc(tslot, ncols);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  if (warp == 0) {
    if (lane == 0) {
      uint32_t issued = 0;
      auto issue_load = [&](int g) {
        const int st = g % S;
        uint8_t* stage = smem + st * stage_bytes;
        uint8_t* B = stage + R * C::kA;
        const int y = (int)((c0 + g) * 64);
        ++issued;
        mbar_expect_tx(&full[st], stage_bytes);
        for (int r = 0; r < R; ++r) {
          tma_load_2d(stage + r * C::kA, &tm_X.m[r], mt * 128, y, &full[st]);
          tma_load_2d(stage + r * C::kA + 8192, &tm_X.m[r], mt * 128 + 64, y, &full[st]);
        }
        for (int j = 0; j < NB; ++j) tma_load_2d(B + j * 8192, &tm_Y, j * 64, y, &full[st]);
      };
      const uint32_t idesc = idesc_bf16(128, D, true, true);
      bool ok = true;
      for (int g = 0; g < S && g < CT; ++g) issue_load(g);
      for (int g = 0; g < CT && ok; ++g) {
        const int st = g % S;
        ok = mbar_wait(&full[st], (g / S) & 1);
        if (!ok) break;
        fence_after_sync();
        const uint32_t A0 = smem_u32(smem + st * stage_bytes);
        const uint32_t B = A0 + R * C::kA;
        for (int r = 0; r < R; ++r) {
#pragma unroll
          for (int ks = 0; ks < 4; ++ks)
            mma_bf16(tmem + r * C::kAcc, desc_sw128(A0 + r * C::kA + ks * 2048, 8192, 1024),
                     desc_sw128(B + ks * 2048, 8192, 1024), idesc, (g > 0 || ks > 0) ? 1u : 0u);
        }
        mma_commit(&empty[st]);
        if (g + S < CT) {
          ok = mbar_wait(&empty[st], (g / S) & 1);
          if (ok) issue_load(g + S);
        }
      }
      if (!ok) {
        atomicOr(status, kErrTimeout);
        drain_rounds(full, S, issued);  // no load still writes shared memory
      }
      mma_commit(accb);  // the MMAs issued complete before TMEM is read and released
    }
    __syncwarp();
  }
  if (!mbar_wait(accb, 0)) atomicOr(status, kErrTimeout);
  fence_after_sync();
  const int orow = mt * 128 + warp * 32 + lane;  // output row i (column of X)
  for (int r = 0; r < R; ++r) {
    float* out = part + ((int64_t)r * gridDim.y + blockIdx.y) * D * D;
#pragma unroll 1
    for (int c = 0; c < D; c += 16) {
      float v[16];
      if (CT > 0) {
        tmem_ld16(tmem + r * C::kAcc + ((uint32_t)(warp * 32) << 16) + c, v);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
      }
      if (orow < D) {
#pragma unroll
        for (int i = 0; i < 16; i += 4)
          *reinterpret_cast<float4*>(out + (int64_t)orow * D + c + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
      }
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 0) tmem_dealloc(tmem, ncols);
}

// G_r = M_r^T dU over the stored (non-empty) rows of one relation r: row k of the relation's compact
// range of M pairs with the dU row of its destination node.  Warps 0-3 copy each 64-row chunk of
// both operands with cp.async into MN-major 128B-swizzled tiles (one instruction: four whole
// 128-byte row blocks; rows past the relation's count, and X columns past D, are zero-filled without
// a read), releasing a stage kLag chunks after issuing it (wait_group, proxy fence, arrive); warp
// 4's lane 0 issues the MMAs; warps 0-3 then read the accumulator.  The chunks are shared among the
// grid's splits by the count read on the device.  Grid (M tiles of 128 output rows, splits);
// part[split][D][D].
template <int D>
struct WgRowsCfg {
  static constexpr int kStages = 4;
  static constexpr int kA = 2 * 8192;        // 64 rows x 128 columns of X (two 64-wide blocks)
  static constexpr int kB = D / 64 * 8192;   // 64 rows x D columns of Y
  static constexpr int kStage = kA + kB;
  static constexpr int kSmem = kStages * kStage + 256 + 1024;
  static_assert(kSmem <= 227 * 1024, "shared memory of wgrad_rows_tc");
  static constexpr int kThreads = 160;
};

template <int D>
__global__ void __launch_bounds__(WgRowsCfg<D>::kThreads, 1)
    wgrad_rows_tc(const __nv_bfloat16* __restrict__ X, const __nv_bfloat16* __restrict__ Y,
                  const int32_t* __restrict__ mlist, const int32_t* __restrict__ mbase, int rel, int64_t row0,
                  int64_t ny, float* __restrict__ part, int* __restrict__ status) {
  using C = WgRowsCfg<D>;
  constexpr int S = C::kStages;
  constexpr uint32_t kLag = S - 1;
  constexpr int NB = D / 64;  // 64-wide column blocks of Y
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * C::kStage);
  uint64_t* empty = full + S;
  uint64_t* accb = empty + S;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int mt = blockIdx.x;  // 128-wide block of X's columns (output rows)
  const int64_t base = mbase[rel], count = (int64_t)mbase[rel + 1] - base;
  const int64_t nchunks = (count + 63) / 64;
  const int64_t cps = (nchunks + gridDim.y - 1) / gridDim.y;
  const int64_t c0 = (int64_t)blockIdx.y * cps;
  const int CT = (int)max((int64_t)0, min(nchunks, c0 + cps) - c0);
  if (threadIdx.x == 0) {
    for (int st = 0; st < S; ++st) {
      mbar_init(&full[st], 128);  // the four producer warps
      mbar_init(&empty[st], 1);
    }
    mbar_init(accb, 1);
    fence_mbar_init();
  }
  if (warp == 4) tmem_alloc(tslot, D);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  if (warp < 4) {
    // ---- producers: warp w copies chunk rows 16 w .. 16 w + 15, lane l chunk l % 8 of a 64-wide
    // block of row 16 w + 4 i + l / 8
    bool ok = true;
    uint32_t done = 0, issued = 0;
    const int ch = lane & 7;
    // rows of X (compact index) and Y (local destination) of this lane's four rows of chunk g; -1: zeros
    auto rows_of = [&](int g, int64_t* xr, int64_t* yr) {
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int64_t k = (c0 + g) * 64 + 16 * warp + 4 * i + (lane >> 3);
        const bool in = g < CT && k < count;
        xr[i] = in ? base + k : -1;
        yr[i] = in ? (int64_t)__ldg(mlist + base + k) - row0 : -1;
        if (yr[i] >= ny) yr[i] = -1;
      }
    };
    int64_t xr[4], yr[4], xn[4], yn[4];
    rows_of(0, xr, yr);
    for (int g = 0; g < CT && ok; ++g) {
      rows_of(g + 1, xn, yn);  // the next chunk's rows, in flight while these are issued
      const int st = g % S;
      if (g >= S) ok = mbar_wait(&empty[st], ((g / S) - 1) & 1);
      if (!ok) break;
      uint8_t* stage = smem + st * C::kStage;
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int kr = 16 * warp + 4 * i + (lane >> 3);  // row of the chunk (K index)
#pragma unroll
        for (int b = 0; b < 2; ++b) {  // X columns mt * 128 + 64 b ..
          const int col = mt * 128 + b * 64 + ch * 8;
          const bool v = xr[i] >= 0 && col < D;
          cp_async16(stage + b * 8192 + sw128_offset(kr, ch * 16), X + (v ? xr[i] * D + col : 0), v);
        }
#pragma unroll
        for (int b = 0; b < NB; ++b) {
          const bool v = yr[i] >= 0;
          cp_async16(stage + C::kA + b * 8192 + sw128_offset(kr, ch * 16), Y + (v ? yr[i] * D + b * 64 + ch * 8 : 0), v);
        }
      }
      cp_async_commit();
      ++issued;
      if (issued - done > kLag) {
        cp_async_wait<kLag>();
        fence_async_smem();
        mbar_arrive(&full[done % S]);
        ++done;
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        xr[i] = xn[i];
        yr[i] = yn[i];
      }
    }
    // every chunk issued is released, also on the give-up path (nothing else is in flight)
    cp_async_wait<0>();
    fence_async_smem();
    for (; done < issued; ++done) mbar_arrive(&full[done % S]);
    if (!ok && lane == 0) atomicOr(status, kErrTimeout);
  } else if (lane == 0) {  // ---- MMA issuer
    const uint32_t idesc = idesc_bf16(128, D, true, true);
    bool ok = true;
    for (int g = 0; g < CT && ok; ++g) {
      const int st = g % S;
      ok = mbar_wait(&full[st], (g / S) & 1);
      if (!ok) break;
      fence_after_sync();
      const uint32_t A0 = smem_u32(smem + st * C::kStage);
      const uint32_t B = A0 + C::kA;
#pragma unroll
      for (int ks = 0; ks < 4; ++ks)
        mma_bf16(tmem, desc_sw128(A0 + ks * 2048, 8192, 1024), desc_sw128(B + ks * 2048, 8192, 1024), idesc,
                 (g > 0 || ks > 0) ? 1u : 0u);
      mma_commit(&empty[st]);
    }
    if (!ok) atomicOr(status, kErrTimeout);
    mma_commit(accb);  // also on the give-up path: the MMAs issued complete before TMEM is released
  }
  __syncwarp();
  if (!mbar_wait(accb, 0)) atomicOr(status, kErrTimeout);
  fence_after_sync();
  if (warp < 4) {
    const int orow = mt * 128 + warp * 32 + lane;  // output row i (column of X)
    float* out = part + (int64_t)blockIdx.y * D * D;
#pragma unroll 1
    for (int c = 0; c < D; c += 16) {
      float v[16];
      if (CT > 0) {
        tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + c, v);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
      }
      if (orow < D) {
#pragma unroll
        for (int i = 0; i < 16; i += 4)
          *reinterpret_cast<float4*>(out + (int64_t)orow * D + c + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
      }
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == 4) tmem_dealloc(tmem, D);
}

// The fused mean layer's weight gradient (d = 128): G_r = M_r^T dU over relation `rel`'s stored rows
// as wgrad_rows_tc computes it, with each row of M_r summed from H over its CSR runs on the way
// in instead of read back (a row above kFuseRuns runs reads its mean from Mlong).  Warps 0-15
// (32 half-warps, two rows of a 64-row chunk each) stream a row's runs as the fused
// projection does (same terms, same order: the rows come out bit for bit as the forward's) into
// the MN-major X stage, and copy the rows' dU by cp.async into the Y stage; a stage is released
// kLag chunks after it was filled (wait_group, proxy fence, arrive).  Warp 16's lane 0 issues the
// MMAs; warps 0-3 then read the accumulator.  Grid (1, splits) with the plain kernel's split-K
// partition; part[split][D][D].
struct WgGatherCfg {
  static constexpr int kStages = 4;
  static constexpr int kA = 2 * 8192;  // 64 rows x 128 columns of X
  static constexpr int kB = 2 * 8192;  // 64 rows x 128 columns of Y
  static constexpr int kStage = kA + kB;
  static constexpr int kSmem = kStages * kStage + 256 + 1024;
  static_assert(kSmem <= 227 * 1024, "shared memory of wgrad_gather_tc");
  static constexpr int kProdWarps = 16;
  static constexpr int kRowsPer = 64 / (2 * kProdWarps);  // rows of a chunk per half-warp
  static constexpr int kThreads = 32 * (kProdWarps + 1);
};

__global__ void __launch_bounds__(WgGatherCfg::kThreads, 1)
    wgrad_gather_tc(const __nv_bfloat16* __restrict__ H, const __nv_bfloat16* __restrict__ Mlong,
                    const int32_t* __restrict__ agg_ptr, const int32_t* __restrict__ agg_col,
                    const int32_t* __restrict__ agg_cnt, const int32_t* __restrict__ csr_ptr,
                    const int32_t* __restrict__ long_ofs, const __nv_bfloat16* __restrict__ Y,
                    const int32_t* __restrict__ mlist, const int32_t* __restrict__ mbase, int rel, int64_t row0,
                    int64_t ny, float* __restrict__ part, int* __restrict__ status) {
  constexpr int D = 128;
  using C = WgGatherCfg;
  constexpr int S = C::kStages;
  constexpr uint32_t kLag = S - 1;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = align1024(smem_raw);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem + S * C::kStage);
  uint64_t* empty = full + S;
  uint64_t* accb = empty + S;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(accb + 1);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t base = mbase[rel], count = (int64_t)mbase[rel + 1] - base;
  const int64_t nchunks = (count + 63) / 64;
  const int64_t cps = (nchunks + gridDim.y - 1) / gridDim.y;
  const int64_t c0 = (int64_t)blockIdx.y * cps;
  const int CT = (int)max((int64_t)0, min(nchunks, c0 + cps) - c0);
  if (threadIdx.x == 0) {
    for (int st = 0; st < S; ++st) {
      mbar_init(&full[st], 32 * C::kProdWarps);
      mbar_init(&empty[st], 1);
    }
    mbar_init(accb, 1);
    fence_mbar_init();
  }
  if (warp == C::kProdWarps) tmem_alloc(tslot, D);
  fence_before_sync();
  __syncthreads();
  fence_after_sync();
  const uint32_t tmem = *tslot;
  if (warp < C::kProdWarps) {
    // ---- producers: half-warp h takes rows h, h + 32 of every chunk; lane l of the half owns
    // 16-byte chunk l of a row (64-wide block l / 8).  Lane i < kRowsPer of a half holds row i's
    // metadata: its dU row (-1: none), run bounds, 1/deg and long slot.
    constexpr int kHalves = 2 * C::kProdWarps;
    const int half = lane >> 4, hl = lane & 15;
    const int grp = 2 * warp + half;
    const int hb = half << 4;
    const unsigned hmask = 0xffffu << hb;
    const __nv_bfloat16* Hc = H + hl * 8;
    const uint32_t smem_s = smem_u32(smem);
    bool ok = true;
    uint32_t done = 0, issued = 0;
    // the CSR row of this lane's row of chunk q (-1: none)
    auto row_of = [&](int q) -> int {
      const int64_t k = (c0 + q) * 64 + grp + kHalves * hl;
      return hl < C::kRowsPer && q < CT && k < count ? __ldg(mlist + base + k) : -1;
    };
    auto meta_of = [&](int row, int& yr, int& rb, int& re, int& slot, float& sc) {
      yr = -1;
      rb = re = 0;
      slot = -1;
      sc = 0.f;
      if (row >= 0) {
        const int64_t y = (int64_t)row - row0;
        yr = y < ny ? (int)y : -1;
        rb = __ldg(agg_ptr + row);
        re = __ldg(agg_ptr + row + 1);
        const int l0 = __ldg(long_ofs + row), l1 = __ldg(long_ofs + row + 1);
        const int e0 = __ldg(csr_ptr + row), e1 = __ldg(csr_ptr + row + 1);
        if (l1 > l0) slot = l0;
        if (e1 > e0) sc = __fdiv_rn(1.0f, (float)(e1 - e0));
      }
    };
    int m_yr, m_rb, m_re, m_slot;
    float m_sc;
    meta_of(row_of(0), m_yr, m_rb, m_re, m_slot, m_sc);
    int row_n = row_of(1);
    for (int g = 0; g < CT && ok; ++g) {
      int n_yr, n_rb, n_re, n_slot;
      float n_sc;
      meta_of(row_n, n_yr, n_rb, n_re, n_slot, n_sc);  // the next chunk's rows, in flight
      const int row_nn = row_of(g + 2);
      const int st = g % S;
      if (g >= S) ok = __all_sync(0xffffffffu, mbar_wait(&empty[st], ((g / S) - 1) & 1));
      if (!ok) break;
      const uint32_t X = smem_s + st * C::kStage + (hl >> 3) * 8192;  // this lane's 64-wide block of X
      uint8_t* Xg = smem + st * C::kStage + (hl >> 3) * 8192;
      uint8_t* Ys = smem + st * C::kStage + C::kA;
      auto put = [&](int kr, uint4 v) {
        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(X + sw128_offset(kr, (hl & 7) * 16)),
                     "r"(v.x), "r"(v.y), "r"(v.z), "r"(v.w)
                     : "memory");
      };
      // dU rows (zeros for rows past the relation's count) and the rows without gathers (a long row's
      // mean, or zeros), by cp.async
#pragma unroll
      for (int i = 0; i < C::kRowsPer; ++i) {
        const int kr = grp + kHalves * i;
        const int yr = __shfl_sync(hmask, m_yr, hb + i);
        cp_async16(Ys + (hl >> 3) * 8192 + sw128_offset(kr, (hl & 7) * 16),
                   Y + (yr >= 0 ? (int64_t)yr * D + hl * 8 : 0), yr >= 0);
        const int rb = __shfl_sync(hmask, m_rb, hb + i), re = __shfl_sync(hmask, m_re, hb + i);
        const int slot = __shfl_sync(hmask, m_slot, hb + i);
        if (slot >= 0 || rb == re)
          cp_async16(Xg + sw128_offset(kr, (hl & 7) * 16), Mlong + (slot >= 0 ? (int64_t)slot * D + hl * 8 : 0),
                     slot >= 0);
      }
      cp_async_commit();
      // the streamed rows
      unsigned qrows = (__ballot_sync(hmask, hl < C::kRowsPer && m_slot < 0 && m_rb < m_re) >> hb) &
                       ((1u << C::kRowsPer) - 1u);
      int qi = 0, qe = 0, qend = 0;
      auto fill = [&](uint32_t& srow) -> int {
        srow = 0xffffffffu;
        int e = -1;
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          if (qe >= qend && qrows != 0u) {
            qi = __ffs(qrows) - 1;
            qrows &= qrows - 1u;
            qe = __shfl_sync(hmask, m_rb, hb + qi);
            qend = __shfl_sync(hmask, m_re, hb + qi);
          }
          if (qe < qend) {
            srow = (srow & ~(0xFu << (4 * k))) | ((uint32_t)qi << (4 * k));
            if ((hl & 7) == k) e = qe;
            ++qe;
          }
        }
        return e >= 0 ? __ldg((hl < 8 ? agg_col : agg_cnt) + e) : 0;
      };
      float acc[8];
#pragma unroll
      for (int q = 0; q < 8; ++q) acc[q] = 0.f;
      int arow = -1;
      auto flush = [&]() {
        const float sc = __shfl_sync(hmask, m_sc, hb + arow);
        put(grp + kHalves * arow,
            make_uint4(pack_bf16x2(acc[0] * sc, acc[1] * sc), pack_bf16x2(acc[2] * sc, acc[3] * sc),
                       pack_bf16x2(acc[4] * sc, acc[5] * sc), pack_bf16x2(acc[6] * sc, acc[7] * sc)));
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
      };
      uint32_t srow;
      int v = fill(srow);
      while ((srow & 0xFu) != 0xFu) {
        uint4 x[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int c = __shfl_sync(hmask, v, hb + k);
          x[k] = ((srow >> (4 * k)) & 0xFu) != 0xFu ? ldg16(Hc + (int64_t)c * D) : make_uint4(0u, 0u, 0u, 0u);
        }
        uint32_t nsrow;
        const int vn = fill(nsrow);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int rk = (int)((srow >> (4 * k)) & 0xFu);
          if (rk == 0xF) break;
          if (rk != arow) {
            if (arow >= 0) flush();
            arow = rk;
          }
          const float w = (float)__shfl_sync(hmask, v, hb + 8 + k);
          float f[8];
          unpack(x[k], f, __nv_bfloat16());
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[q] = fmaf(w, f[q], acc[q]);
        }
        srow = nsrow;
        v = vn;
      }
      if (arow >= 0) flush();
      ++issued;
      if (issued - done > kLag) {
        cp_async_wait<kLag>();
        fence_async_smem();
        mbar_arrive(&full[done % S]);
        ++done;
      }
      __syncwarp();
      m_yr = n_yr;
      m_rb = n_rb;
      m_re = n_re;
      m_slot = n_slot;
      m_sc = n_sc;
      row_n = row_nn;
    }
    // every chunk filled is released, also on the give-up path (nothing else is in flight)
    cp_async_wait<0>();
    fence_async_smem();
    for (; done < issued; ++done) mbar_arrive(&full[done % S]);
    if (!ok && lane == 0) atomicOr(status, kErrTimeout);
  } else if (lane == 0) {  // ---- MMA issuer
    const uint32_t idesc = idesc_bf16(128, D, true, true);
    bool ok = true;
    for (int g = 0; g < CT && ok; ++g) {
      const int st = g % S;
      ok = mbar_wait(&full[st], (g / S) & 1);
      if (!ok) break;
      fence_after_sync();
      const uint32_t A0 = smem_u32(smem + st * C::kStage);
      const uint32_t B = A0 + C::kA;
#pragma unroll
      for (int ks = 0; ks < 4; ++ks)
        mma_bf16(tmem, desc_sw128(A0 + ks * 2048, 8192, 1024), desc_sw128(B + ks * 2048, 8192, 1024), idesc,
                 (g > 0 || ks > 0) ? 1u : 0u);
      mma_commit(&empty[st]);
    }
    if (!ok) atomicOr(status, kErrTimeout);
    mma_commit(accb);  // also on the give-up path: the MMAs issued complete before TMEM is released
  }
  __syncwarp();
  if (!mbar_wait(accb, 0)) atomicOr(status, kErrTimeout);
  fence_after_sync();
  if (warp < 4) {
    const int orow = warp * 32 + lane;  // output row i (column of X)
    float* out = part + (int64_t)blockIdx.y * D * D;
#pragma unroll 1
    for (int c = 0; c < D; c += 16) {
      float v[16];
      if (CT > 0) {
        tmem_ld16(tmem + ((uint32_t)(warp * 32) << 16) + c, v);
      } else {
#pragma unroll
        for (int i = 0; i < 16; ++i) v[i] = 0.f;
      }
#pragma unroll
      for (int i = 0; i < 16; i += 4)
        *reinterpret_cast<float4*>(out + (int64_t)orow * D + c + i) = make_float4(v[i], v[i + 1], v[i + 2], v[i + 3]);
    }
  }
  fence_before_sync();
  __syncthreads();
  if (warp == C::kProdWarps) tmem_dealloc(tmem, D);
}

// ---------------------------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------------------------
template <int D>
static hg_status smem_attr_once() {
  static bool done = false;
  if (!done) {
    HG_CUDA(cudaFuncSetAttribute(proj_fwd_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, FwdCfg<D>::kSmem));
    HG_CUDA(cudaFuncSetAttribute(proj_bwd_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, BwdCfg<D>::kSmem));
    HG_CUDA(cudaFuncSetAttribute(wgrad_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, WgCfg<D>::kSmem));
    HG_CUDA(cudaFuncSetAttribute(wgrad_rows_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, WgRowsCfg<D>::kSmem));
    done = true;
  }
  return HG_OK;
}


template <int D>
static hg_status tc_fuse_t(const void* W_rel, const void* W_agg, RelDst rd, int num_rels, void* V, void* Vt,
                           cudaStream_t s) {
  if (num_rels == 0) return HG_OK;
  return launch("fuse_weights", fuse_weights<D>, dim3(D / 32, D / 32, num_rels), dim3(256), 0, s,
                (const __nv_bfloat16*)W_rel, (const __nv_bfloat16*)W_agg, rd, num_rels, (__nv_bfloat16*)V,
                (__nv_bfloat16*)Vt);
}

template <int D>
static hg_status tc_fwd_t(const TcFwdArgs& a0, const void* M, int64_t m_rows, const void* Vt, int num_rels,
                          cudaStream_t s) {
  HG_TRY(smem_attr_once<D>());
  TcFwdArgs a = a0;
  a.M = (const __nv_bfloat16*)M;
  a.msent = m_rows;
  CUtensorMap tm_V;
  HG_TRY(make_tmap_bf16(&tm_V, Vt, (uint64_t)2 * num_rels * D, D, D));
  int sms = 0, dev = 0;
  HG_CUDA(cudaGetDevice(&dev));
  HG_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(a.n, kTileRows), sms));
  return launch("proj_fwd_tc", proj_fwd_tc<D>, dim3(grid), dim3(FwdCfg<D>::kThreads), FwdCfg<D>::kSmem, s, tm_V,
                a);
}

template <int D>
static hg_status tc_fwd_gather_t(const TcFwdArgs& a, const void* Vt, int num_rels, cudaStream_t s) {
  if constexpr (D != 128) {
    set_error("the fused mean layer needs d = 128 (d = %d)", D);
    return HG_ERR_UNSUPPORTED;
  } else {
    static bool attr = false;
    if (!attr) {
      HG_CUDA(cudaFuncSetAttribute(proj_fwd_gather_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   FwdCfg<D, true>::kSmem));
      attr = true;
    }
    CUtensorMap tm_V;
    HG_TRY(make_tmap_bf16(&tm_V, Vt, (uint64_t)2 * num_rels * D, D, D));
    int sms = 0, dev = 0;
    HG_CUDA(cudaGetDevice(&dev));
    HG_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(ceil_div(a.n, kTileRows), sms));
    return launch("proj_fwd_gather_tc", proj_fwd_gather_tc<D>, dim3(grid), dim3(FwdCfg<D, true>::kThreads),
                  FwdCfg<D, true>::kSmem, s, tm_V, a);
  }
}

template <int D>
static hg_status tc_ln_act_t(const TcBwdArgs& a, int* blocks, cudaStream_t s) {
  // one wave of resident blocks: fewer column partials to reduce afterwards
  static int resident = 0;
  if (resident == 0) {
    int dev = 0, sms = 0, per_sm = 0;
    HG_CUDA(cudaGetDevice(&dev));
    HG_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    HG_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, ln_act_bwd<D>, 256, 0));
    resident = std::max(1, sms * per_sm);
  }
  const int g = (int)std::max<int64_t>(1, std::min<int64_t>(ceil_div(a.n, 8), std::min(resident, 152 * 8)));
  *blocks = g;
  return launch("ln_act_bwd", ln_act_bwd<D>, dim3(g), dim3(256), 0, s, a);
}

template <int D>
static hg_status tc_bwd_t(const TcBwdArgs& a, const void* V, int num_rels, cudaStream_t s) {
  HG_TRY(smem_attr_once<D>());
  if (a.nrel == 0) return HG_OK;
  CUtensorMap tm_dU, tm_V;
  HG_TRY(make_tmap_bf16(&tm_dU, a.dU + a.off * D, (uint64_t)a.n, D, 1));  // one-row box: gathers
  HG_TRY(make_tmap_bf16(&tm_V, V, (uint64_t)2 * num_rels * D, D, D));
  int sms = 0, dev = 0;
  HG_CUDA(cudaGetDevice(&dev));
  HG_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  // the jobs (128 stored rows of one relation) are counted on the device; at most this many
  const int64_t cap = (int64_t)a.nrel * ceil_div(a.n, kTileRows);
  const unsigned grid = (unsigned)std::max<int64_t>(1, std::min<int64_t>(cap, sms));
  return launch("proj_bwd_tc", proj_bwd_tc<D>, dim3(grid), dim3(BwdCfg<D>::kThreads), BwdCfg<D>::kSmem, s, tm_dU,
                tm_V, a);
}

int wgrad_tc_splits(int64_t n, int d) {
  const int mtiles = d > 128 ? d / 128 : 1;
  const int64_t chunks = std::max<int64_t>(1, ceil_div(n, 64));
  return (int)std::max<int64_t>(1, std::min<int64_t>(chunks, 152 / mtiles));  // one wave, one CTA per SM
}

template <int D>
static hg_status tc_wgrad_t(const void* X, const int64_t* x0, int R, const void* Y, int64_t y0, int64_t n,
                            float* part, float* const* outs, float* tmp, cudaStream_t s) {
  HG_TRY(smem_attr_once<D>());
  if (R < 1 || R > WgCfg<D>::kMaxR) {
    set_error("tc_weight_grad: %d relations per launch (at most %d at d=%d)", R, WgCfg<D>::kMaxR, D);
    return HG_ERR_UNSUPPORTED;
  }
  if (n == 0) {
    for (int r = 0; r < R; ++r) HG_CUDA(cudaMemsetAsync(outs[r], 0, (size_t)D * D * sizeof(float), s));
    return HG_OK;
  }
  const int mtiles = D > 128 ? D / 128 : 1;
  const int splits = wgrad_tc_splits(n, D);
  const int64_t chunks = std::max<int64_t>(1, ceil_div(n, 64));
  const int cps = (int)ceil_div(chunks, splits);
  const int stage_bytes = R * WgCfg<D>::kA + (D / 64) * 8192;
  const int stages = std::min(4, (WgCfg<D>::kSmem - 1024 - 256) / stage_bytes);
  RelMaps tm_X;
  std::memset(&tm_X, 0, sizeof(tm_X));
  for (int r = 0; r < R; ++r)
    HG_TRY(make_tmap_bf16(&tm_X.m[r], (const __nv_bfloat16*)X + x0[r] * D, (uint64_t)n, D, 64));
  CUtensorMap tm_Y;
  HG_TRY(make_tmap_bf16(&tm_Y, (const __nv_bfloat16*)Y + y0 * D, (uint64_t)n, D, 64));
  HG_TRY(launch("wgrad_tc", wgrad_tc<D>, dim3(mtiles, splits), dim3(WgCfg<D>::kThreads),
                (size_t)stages * stage_bytes + 256 + 1024, s, tm_X, tm_Y, R, stages, n, cps, part,
                device_status_ptr()));
  for (int r = 0; r < R; ++r)
    HG_TRY(reduce_partials(part + (size_t)r * splits * D * D, (int64_t)D * D, splits, (int64_t)D * D, outs[r], tmp,
                           s));
  return HG_OK;
}

template <int D>
static hg_status tc_wgrad_rows_t(const void* M, int64_t m_rows, const int32_t* mlist, const int32_t* mbase, int rel,
                                 int64_t row0, const void* dU, int64_t y0, int64_t n, float* part, float* out,
                                 float* tmp, cudaStream_t s) {
  HG_TRY(smem_attr_once<D>());
  if (n == 0) {
    HG_CUDA(cudaMemsetAsync(out, 0, (size_t)D * D * sizeof(float), s));
    return HG_OK;
  }
  const int mtiles = D > 128 ? D / 128 : 1;
  const int splits = wgrad_tc_splits(n, D);  // the stored rows (at most n) are split on the device
  (void)m_rows;
  HG_TRY(launch("wgrad_tc", wgrad_rows_tc<D>, dim3(mtiles, splits), dim3(WgRowsCfg<D>::kThreads),
                (size_t)WgRowsCfg<D>::kSmem, s, (const __nv_bfloat16*)M, (const __nv_bfloat16*)dU + y0 * D, mlist,
                mbase, rel, row0, n, part, device_status_ptr()));
  return reduce_partials(part, (int64_t)D * D, splits, (int64_t)D * D, out, tmp, s);
}

template <int D>
static hg_status tc_wgrad_gather_t(const hg_graph* g, const void* H, const void* Mlong, int rel, int64_t row0,
                                  const void* dU, int64_t y0, int64_t n, float* part, float* out, float* tmp,
                                  cudaStream_t s) {
  if constexpr (D != 128) {
    set_error("the fused mean layer needs d = 128 (d = %d)", D);
    return HG_ERR_UNSUPPORTED;
  } else {
    static bool attr = false;
    if (!attr) {
      HG_CUDA(cudaFuncSetAttribute(wgrad_gather_tc, cudaFuncAttributeMaxDynamicSharedMemorySize, WgGatherCfg::kSmem));
      attr = true;
    }
    if (n == 0) {
      HG_CUDA(cudaMemsetAsync(out, 0, (size_t)D * D * sizeof(float), s));
      return HG_OK;
    }
    // the split-K partition of the plain kernel (the stored rows, at most n, split on the device),
    // so that the partial sums and their fixed-order reduction are the same
    const int splits = wgrad_tc_splits(n, D);
    HG_TRY(launch("wgrad_gather_tc", wgrad_gather_tc, dim3(1, splits), dim3(WgGatherCfg::kThreads),
                  (size_t)WgGatherCfg::kSmem, s, (const __nv_bfloat16*)H, (const __nv_bfloat16*)Mlong,
                  (const int32_t*)g->agg_ptr, (const int32_t*)g->agg_col, (const int32_t*)g->agg_cnt,
                  (const int32_t*)g->csr_ptr, (const int32_t*)g->long_ofs, (const __nv_bfloat16*)dU + y0 * D,
                  (const int32_t*)g->mlist, (const int32_t*)g->mbase, rel, row0, n, part, device_status_ptr()));
    return reduce_partials(part, (int64_t)D * D, splits, (int64_t)D * D, out, tmp, s);
  }
}

template <int D>
static hg_status tc_finish_t(const float* G, const void* W_rel, const void* W_agg, RelDst rd, int num_rels,
                             int num_types, float* dW_rel, float* dW_agg, cudaStream_t s) {
  return launch("wgrad_finish", wgrad_finish<D>, dim3(D / 32, D / 32, num_rels + num_types), dim3(256),
                0, s, G, (const __nv_bfloat16*)W_rel, (const __nv_bfloat16*)W_agg, rd, num_rels, num_types, dW_rel,
                dW_agg);
}

#define HG_TC_DISPATCH(d, FN, ...)                  \
  do {                                              \
    if (d == 64) return FN<64>(__VA_ARGS__);        \
    if (d == 128) return FN<128>(__VA_ARGS__);      \
    if (d == 256) return FN<256>(__VA_ARGS__);      \
    set_error("unsupported feature width %d", d);   \
    return HG_ERR_UNSUPPORTED;                      \
  } while (0)

hg_status tc_fuse_weights(int d, const void* W_rel, const void* W_agg, RelDst rd, int num_rels, void* V, void* Vt,
                          cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_fuse_t, W_rel, W_agg, rd, num_rels, V, Vt, s);
}
hg_status tc_proj_forward(int d, const TcFwdArgs& a, const void* M, int64_t m_rows, const void* Vt, int num_rels,
                          cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_fwd_t, a, M, m_rows, Vt, num_rels, s);
}
hg_status tc_proj_forward_gather(int d, const TcFwdArgs& a, const void* Vt, int num_rels, cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_fwd_gather_t, a, Vt, num_rels, s);
}
hg_status tc_ln_act_backward(int d, const TcBwdArgs& a, int* blocks, cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_ln_act_t, a, blocks, s);
}
hg_status tc_proj_backward(int d, const TcBwdArgs& a, const void* V, int num_rels, cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_bwd_t, a, V, num_rels, s);
}
hg_status tc_weight_grad(int d, const void* X, const int64_t* x0, int R, const void* Y, int64_t y0, int64_t n,
                         float* part, float* const* outs, float* tmp, cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_wgrad_t, X, x0, R, Y, y0, n, part, outs, tmp, s);
}
hg_status tc_weight_grad_rows(int d, const void* M, int64_t m_rows, const int32_t* mlist, const int32_t* mbase, int rel,
                              int64_t row0, const void* dU, int64_t y0, int64_t n, float* part, float* out, float* tmp,
                              cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_wgrad_rows_t, M, m_rows, mlist, mbase, rel, row0, dU, y0, n, part, out, tmp, s);
}
hg_status tc_weight_grad_gather(int d, const hg_graph* g, const void* H, const void* Mlong, int rel, int64_t row0,
                                const void* dU, int64_t y0, int64_t n, float* part, float* out, float* tmp,
                                cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_wgrad_gather_t, g, H, Mlong, rel, row0, dU, y0, n, part, out, tmp, s);
}
int wgrad_tc_max_rels(int d) { return d == 64 ? WgCfg<64>::kMaxR : (d == 128 ? WgCfg<128>::kMaxR : WgCfg<256>::kMaxR); }
hg_status tc_wgrad_finish(int d, const float* G, const void* W_rel, const void* W_agg, RelDst rd, int num_rels,
                          int num_types, float* dW_rel, float* dW_agg, cudaStream_t s) {
  HG_TC_DISPATCH(d, tc_finish_t, G, W_rel, W_agg, rd, num_rels, num_types, dW_rel, dW_agg, s);
}

}  // namespace hg
