// H2O sparse SDPA for one chunk, with summed attention weights.
//
// What it computes (§3.1 Eq. 2, mask of §3.3.1, summed weights of §3.3.1 and
// §A.6.1): for every (b, query head hq) and chunk row i,
//   lambda_i  = log sum_{j visible} exp(scale * q_i . k_j)
//   out_i     = sum_j exp(scale * q_i . k_j - lambda_i) v_j
//   score_inc[b, hq, j] += sum_i exp(scale * q_i . k_j - lambda_i)
// over the key columns j = cache slots 0..M-1 then chunk tokens 0..S-1.
//
// Design (one CTA per 128 query rows of one KV-head group; GQA heads of the
// group are packed into the rows when S <= 128):
//  * §A.6.1 notes that column sums need each row's final normaliser before
//    they can be reduced.  The CTA therefore makes two passes over its key
//    tiles: pass 1 computes lambda (Q K^T + online max/sum), pass 2 recomputes
//    Q K^T, forms P = exp2(S log2e scale - lambda log2e) in fp32, reduces P's
//    columns into score_inc and accumulates P V.  Because lambda is final in
//    pass 2, the P V accumulator never needs rescaling.
//  * d = 128 runs on CTA pairs (a cluster of two CTAs, adjacent row tiles of
//    the same group) with the 2-SM tcgen05 MMA (M = 256): each CTA loads only
//    half of every K tile (64 keys) and half of every V tile (64 of the d
//    columns), which halves the L2-to-SM traffic per MMA.  The even CTA
//    issues all MMAs; the odd CTA's softmax warps signal it through its
//    barriers.  Both CTAs walk the union of their key-tile lists; a tile only
//    the other CTA can see is fully masked here.  d = 64 runs one CTA per row
//    tile with the 1-SM MMA.
//  * Warp roles: warp 0 issues TMA loads (Q once, then K tiles through ring A
//    and V tiles through ring B of shared-memory slots); warps 1 and 3 issue
//    the Q K^T MMAs of the even and the odd tiles of each pass and warp 2 every
//    P V, so that the tensor pipe keeps working while an issuing thread waits
//    on a barrier or commits; warps 4-19 form four softmax warpgroups.  In
//    pass 1 the warpgroups form two teams that take alternate tiles (a team's
//    two warpgroups own key columns 0-63 and 64-127); in pass 2 every
//    warpgroup takes every tile, warpgroup w its key columns 32w .. 32w+31.
//  * TMEM: pass 1 uses four fp32 S buffers; pass 2 three S buffers and the O
//    accumulator.  In pass 2 the bf16 P of a tile is written over the S
//    columns it came from (each warpgroup over its own), and the P V MMA reads
//    it there, so storing P never waits for an earlier P V.
//  * Column sums use the fp32 P (not the bf16 copy fed to the MMA).  Pass 2
//    reads S in TMEM's 16x256b layout, where a thread holds 4 rows x 8
//    columns: it adds its 4 rows, a 3-step warp reduce-scatter leaves one
//    column sum (over the warp's 32 rows) per lane and 32-column block, the
//    last of the four warps of a warpgroup to finish a tile combines them
//    through shared memory, and one red.global.add per column and query head
//    goes to score_inc (zeroed by the host call), or, with three or more row
//    tiles per head, a store into the tile's row of column partials that a
//    second kernel adds in row-tile order.  Pass 1 keeps one row per thread
//    (32x32b layout) for the row statistics.
//  * Key tiles are classified up front from slot_pos: tiles no row of the CTA
//    can see are skipped, tiles every row sees need no mask, the rest are
//    masked per element.
//  * Every wait is bounded; on expiry the CTA drains and reports
//    H2O_DEVERR_TIMEOUT instead of hanging.
#include <cmath>

#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kNumWG = 4;                       // softmax warpgroups
// warp 0 TMA producer, warps 1 and 3 Q K^T issuers (even / odd tiles), warp 2
// P V issuer
constexpr int kFirstSoftmaxWarp = 4;
constexpr int kSoftmaxWarps = 4 * kNumWG;
constexpr int kThreads = 32 * (kFirstSoftmaxWarp + kSoftmaxWarps);  // 640
constexpr uint16_t kTileChunk = 0x8000;
constexpr uint16_t kTilePartial = 0x4000;
constexpr uint16_t kTileIdxMask = 0x3FFF;
constexpr uint8_t kClsSkip = 0, kClsFull = 1, kClsPartial = 2;
// TMEM (512 columns).  Pass 1 needs no P or O: four S buffers (fp32, 128
// columns each), each free again as soon as the softmax has loaded it.
// Pass 2: three S buffers and the O accumulator (columns 384..).  Every
// warpgroup takes every pass-2 tile: warpgroup w loads the S of keys
// 32w .. 32w+31, then writes their bf16 P as pairs into columns 32w .. 32w+15
// of the same buffer (columns only that warpgroup loaded), where the P V MMA
// reads it; the buffer is free again when that P V has completed.  So writing
// P never waits for an earlier P V.
constexpr int kSBufs1 = 4;
constexpr int kSBufs2 = 3;
// Column-sum buffers, used round robin by the pass-2 tiles.  Buffer c of tile
// t is written again by tile t + 4, whose Q K^T was issued after the P V of
// tile t + 1 had completed, which needed every softmax warp's arrival for
// tile t + 1, which each warp makes after its reads of tile t's buffer.
constexpr int kColBufs = 4;

__device__ __forceinline__ int pass1_buffer_uses(int n_t, int b) {
  return n_t > b ? (n_t - 1 - b) / kSBufs1 + 1 : 0;
}

// S buffer of step n (pass-1 tile n < n_t, pass-2 tile n - n_t) and how many
// times that buffer was filled before.
__device__ __forceinline__ void s_buffer(int n, int n_t, int& buf, int& use) {
  if (n < n_t) {
    buf = n % kSBufs1;
    use = n / kSBufs1;
  } else {
    buf = (n - n_t) % kSBufs2;
    use = pass1_buffer_uses(n_t, buf) + (n - n_t) / kSBufs2;
  }
}

// Shared-memory ring geometry.  Pass 1 streams K tiles through all slots;
// pass 2 sends K tiles through ring A (consumed by the Q K^T issuer) and V
// tiles through ring B (consumed by the P V issuer).  Within each pass a slot
// has a single consumer that takes its loads in order, and pass 2 starts on a
// slot only after pass 1 has consumed it, which keeps every mbarrier wait at
// most one phase ahead.
//   1-SM (d = 64):  a slot holds a whole K or V tile, 16 KB.
//   pair (d = 128): a slot holds this CTA's half of a K tile (64 keys x 128
//                   columns, two 8 KB panels) or of a V tile (128 keys x 64
//                   columns, one 16 KB panel).
template <int D, bool kPair>
struct Geom {
  static constexpr int kPanels = D / 64;
  static constexpr int kSlotBytes = kPair ? 16384 : kPanels * kTileN * 128;
  static constexpr int kKPanelBytes = kPair ? (kTileN / 2) * 128 : kTileN * 128;
  static constexpr int kRA = kPair ? 6 : (D == 128 ? 3 : 6);
  static constexpr int kRB = kPair ? 4 : (D == 128 ? 2 : 4);
  static constexpr int kR = kRA + kRB;
  static constexpr int kCtas = kPair ? 2 : 1;
};

// Loads of pass 1 (tiles 0 .. n_t - 1, slot t % R) that land in slot s.
__device__ __forceinline__ int pass1_uses(int n_t, int R, int s) {
  return n_t > s ? (n_t - 1 - s) / R + 1 : 0;
}

template <int D, bool kPair>
struct __align__(1024) SdpaSmem {
  using G = Geom<D, kPair>;
  uint8_t q[G::kPanels][kTileM * 128];
  uint8_t kv[G::kR][G::kSlotBytes];
  float colsum[kColBufs][kNumWG][4][32];  // [buffer][warpgroup][warp][column]
  float rowstat[kNumWG][kTileM][2];
  uint64_t bar_q;
  uint64_t bar_full[G::kR], bar_empty[G::kR];
  uint64_t bar_sfull[kSBufs1], bar_sread[kSBufs1], bar_pfull[kSBufs2], bar_pvdone[kSBufs2];
  uint64_t bar_rowstat, bar_ofull, bar_drain[3];
  uint32_t cs_count[kColBufs][kNumWG];  // column-sum partials deposited (4 per tile)
  uint32_t taddr;
  int abort_flag;
  int n_tiles;
  uint8_t cls[kMaxKeyTiles];  // bits 0-1: this CTA's class, bits 2-3: the other CTA's
  uint16_t tiles[kMaxKeyTiles];
};

// One butterfly reduce-scatter step over lane bit O: of the L values a lane
// holds, it keeps the upper half if its bit O is set (the lower half
// otherwise) and adds the partner lane's copy of that half.
template <int L, int O>
__device__ __forceinline__ void rs_step(float (&v)[8], uint32_t lane) {
  const bool up = (lane & O) != 0;
#pragma unroll
  for (int k = 0; k < L / 2; ++k) {
    const float send = up ? v[k] : v[k + L / 2];
    const float keep = up ? v[k + L / 2] : v[k];
    v[k] = keep + __shfl_xor_sync(0xffffffffu, send, O);
  }
}

// Bounded barrier wait.  Every signal between the CTAs of a pair orders
// tcgen05 operations or TMA writes only (tcgen05 fences around the barrier,
// complete_tx accounting), so CTA-scope acquire suffices.
template <bool kPair>
__device__ __forceinline__ bool wait_b(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return wait_bar(bar, parity, abort, kWaitLimitNs);
}

// Arrival of a softmax warp on a barrier of the MMA-issuing CTA.
template <bool kPair>
__device__ __forceinline__ void arrive_issuer(uint64_t* bar) {
  if constexpr (kPair) bar_arrive_remote(cluster_addr(bar, 0));
  else bar_arrive(bar);
}

template <bool kPair>
__device__ __forceinline__ void commit_all(uint64_t* bar) {
  if constexpr (kPair) mma_commit_pair(bar, 3);
  else mma_commit(bar);
}

// Query rows of row tile r: head of the first row, first/last chunk row.
// False when r is past the last row tile (the odd CTA of the last pair).
__device__ __forceinline__ bool row_range(const SdpaArgs& a, int r, int& g_first, int& i_lo,
                                          int& i_hi) {
  if (r >= a.n_row_tiles) return false;
  if (a.tiles_per_head > 0) {
    g_first = r / a.tiles_per_head;
    i_lo = (r % a.tiles_per_head) * kTileM;
    i_hi = min(i_lo + kTileM, a.S) - 1;
  } else {
    g_first = r * a.heads_box;
    i_lo = 0;
    i_hi = a.S - 1;
  }
  return true;
}

template <int D, bool kPair>
__global__ void __launch_bounds__(kThreads, 1) sdpa_chunk_kernel(const __grid_constant__ SdpaArgs a) {
  using G = Geom<D, kPair>;
  constexpr int P = G::kPanels;
  extern __shared__ uint8_t smem_raw[];
  // 1024-byte aligned (128-byte swizzle atoms).  Offsetting the shared array
  // itself, rather than an integer copy of its address, keeps the pointer in
  // the shared state space, so accesses through `sm` compile to shared loads.
  auto& sm = *reinterpret_cast<SdpaSmem<D, kPair>*>(
      smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u));
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const uint32_t lane = tid & 31;
  const int grp = blockIdx.y;  // b * Hkv + kv head
  const int rt = blockIdx.x;   // row tile within the group
  const uint32_t rank = kPair ? cluster_rank() : 0u;
  const bool leader = rank == 0;
  const int b = grp / a.Hkv;
  const int hkv = grp % a.Hkv;
  const int NK = a.nk;         // key columns per query head (score_inc row length)

  int g_first = a.qg, i_lo = 0, i_hi = -1;
  const bool has_rows = row_range(a, rt, g_first, i_lo, i_hi);
  int pg = 0, p_lo = 0, p_hi = -1;
  const bool peer_rows = kPair && row_range(a, rt ^ 1, pg, p_lo, p_hi);
  // rows the Q box covers (the rest of the tile is zero-filled here)
  const int box_rows = a.tiles_per_head > 0 ? kTileM : a.rows_box * a.heads_box;
  // the kernels after it on the stream (column-sum reduction, update) may be
  // placed now; they wait for this grid before reading what it writes
  if (tid == 0) launch_dependents();
  // While the tiles are classified, bring Q and the first cache K tiles (this
  // CTA's halves) into L2, so the loads after the classification hit there.
  if (warp == 0 && lane == 0 && has_rows) {
    tma_prefetch_desc(&a.tm_q);
    for (int p = 0; p < P; ++p) tma_prefetch_4d(&a.tm_q, 64 * p, i_lo, g_first, grp);
    if (a.n_cache_tiles > 0) {
      tma_prefetch_desc(&a.tm_kc);
      const int n_pre = 0;
      for (int t = 0; t < n_pre; ++t)
        for (int p = 0; p < P; ++p)
          tma_prefetch_3d(&a.tm_kc, 64 * p, t * kTileN + (kPair ? (kTileN / 2) * static_cast<int>(rank) : 0),
                          grp);
    }
  }

  if (tid == 0) {
    bar_init(&sm.bar_q, 1);
    for (int s = 0; s < G::kR; ++s) {
      bar_init(&sm.bar_full[s], 1);
      bar_init(&sm.bar_empty[s], 1);
    }
    for (int x = 0; x < kSBufs1; ++x) {
      bar_init(&sm.bar_sfull[x], 1);
      // the 8 warps of the team owning the tile, in every CTA of the pair
      bar_init(&sm.bar_sread[x], G::kCtas * kSoftmaxWarps / 2);
    }
    for (int x = 0; x < kSBufs2; ++x) {
      // every softmax warp, in every CTA of the pair
      bar_init(&sm.bar_pfull[x], G::kCtas * kSoftmaxWarps);
      bar_init(&sm.bar_pvdone[x], 1);
    }
    for (int x = 0; x < kColBufs; ++x)
      for (int w = 0; w < kNumWG; ++w) sm.cs_count[x][w] = 0u;
    bar_init(&sm.bar_rowstat, kSoftmaxWarps);
    bar_init(&sm.bar_ofull, 1);
    for (int x = 0; x < 3; ++x) bar_init(&sm.bar_drain[x], 1);
    sm.abort_flag = 0;
    fence_bar_init();
  }
  if (warp == 1) {
    if constexpr (kPair) {
      tmem_alloc_pair(&sm.taddr, 512);
      tmem_relinquish_pair();
    } else {
      tmem_alloc(&sm.taddr, 512);
      tmem_relinquish();
    }
  }
  // Rows the Q box does not cover must still give finite logits.
  if (box_rows < kTileM) {
    const int words = (kTileM - box_rows) * 32;
    for (int p = 0; p < P; ++p)
      for (int x = tid; x < words; x += kThreads)
        reinterpret_cast<uint32_t*>(sm.q[p] + box_rows * 128)[x] = 0u;
    fence_proxy_async_smem();
  }
  // Classify key tiles against this CTA's rows (bits 0-1) and, on a pair, the
  // other CTA's rows (bits 2-3).
  if (warp >= kFirstSoftmaxWarp) {
    const int sw = warp - kFirstSoftmaxWarp;
    const int* sp = a.slot_pos + static_cast<size_t>(grp) * a.M;
    // four tiles per round, all their slot_pos loads in flight at once
    for (int ct0 = sw; ct0 < a.n_cache_tiles; ct0 += 4 * kSoftmaxWarps) {
      int pos4[4][4];
#pragma unroll
      for (int bt = 0; bt < 4; ++bt)
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int j = (ct0 + bt * kSoftmaxWarps) * kTileN + r * 32 + static_cast<int>(lane);
          pos4[bt][r] = j < a.M ? __ldg(sp + j) : -1;
        }
#pragma unroll
      for (int bt = 0; bt < 4; ++bt) {
        const int ct = ct0 + bt * kSoftmaxWarps;
        if (ct >= a.n_cache_tiles) break;
        bool any0 = false, all0 = true, any1 = false, all1 = true;
#pragma unroll
        for (int r = 0; r < 4; ++r) {
          const int pos = pos4[bt][r];
          any0 |= pos >= 0 && pos <= a.pos0 + i_hi;
          all0 &= pos >= 0 && pos <= a.pos0 + i_lo;
          any1 |= pos >= 0 && pos <= a.pos0 + p_hi;
          all1 &= pos >= 0 && pos <= a.pos0 + p_lo;
        }
        any0 = __any_sync(0xffffffffu, any0) && has_rows;
        all0 = __all_sync(0xffffffffu, all0);
        any1 = __any_sync(0xffffffffu, any1) && peer_rows;
        all1 = __all_sync(0xffffffffu, all1);
        const uint8_t c0 = any0 ? (all0 ? kClsFull : kClsPartial) : kClsSkip;
        const uint8_t c1 = any1 ? (all1 ? kClsFull : kClsPartial) : kClsSkip;
        if (lane == 0) sm.cls[ct] = static_cast<uint8_t>(c0 | (c1 << 2));
      }
    }
    for (int c = sw; c < a.n_chunk_tiles; c += kSoftmaxWarps) {
      const int c0 = c * kTileN;
      auto chunk_cls = [&](bool rows, int lo, int hi) -> uint8_t {
        if (!rows || c0 > hi) return kClsSkip;
        if (c0 + kTileN - 1 <= lo && c0 + kTileN <= a.S) return kClsFull;
        return kClsPartial;
      };
      const uint8_t cl = static_cast<uint8_t>(chunk_cls(has_rows, i_lo, i_hi) |
                                              (chunk_cls(peer_rows, p_lo, p_hi) << 2));
      if (lane == 0) sm.cls[a.n_cache_tiles + c] = cl;
    }
  }
  __syncthreads();
  if (warp == kFirstSoftmaxWarp) {
    // tile list: the union over the pair, in order; masked here unless this
    // CTA sees every key of the tile from every row
    const int total = a.n_cache_tiles + a.n_chunk_tiles;
    int n = 0;
    for (int base = 0; base < total; base += 32) {
      const int t = base + static_cast<int>(lane);
      const uint8_t cl = t < total ? sm.cls[t] : 0;
      const uint32_t m = __ballot_sync(0xffffffffu, cl != 0);
      if (cl != 0) {
        const int pos = n + __popc(m & ((1u << lane) - 1u));
        uint16_t e = t < a.n_cache_tiles ? static_cast<uint16_t>(t)
                                         : static_cast<uint16_t>(kTileChunk | (t - a.n_cache_tiles));
        if ((cl & 3) != kClsFull) e |= kTilePartial;
        sm.tiles[pos] = e;
      }
      n += __popc(m);
    }
    if (lane == 0) sm.n_tiles = n;
  }
  tc_fence_before_sync();
  __syncthreads();
  // On a pair, both CTAs' barriers are initialised (and the zero-filled Q rows
  // published) before any signal crosses between them.
  if constexpr (kPair) cluster_sync_all();
  tc_fence_after_sync();

  const uint32_t tmem = sm.taddr;
  const uint32_t tS = tmem;                          // S buffer b: columns 128 b ..
  const uint32_t tO = tmem + 128 * kSBufs2;          // O accumulator: columns 384 ..
  static_assert(128 * kSBufs2 + 128 == 128 * kSBufs1, "TMEM layout");
  const int n_t = sm.n_tiles;
  volatile int* abort_flag = &sm.abort_flag;

  if (warp == 0) {
    // ------------------------------------------------------- TMA producer --
    if (lane == 0 && n_t > 0) {
      tma_prefetch_desc(&a.tm_q);
      tma_prefetch_desc(&a.tm_kn);
      tma_prefetch_desc(&a.tm_vn);
      if (a.n_cache_tiles > 0) {
        tma_prefetch_desc(&a.tm_kc);
        tma_prefetch_desc(&a.tm_vc);
      }
      constexpr int RA = G::kRA, RB = G::kRB, R = G::kR;
      const uint32_t q_bytes = P * 128 * box_rows;
      if constexpr (kPair) {
        const uint32_t bq = cluster_addr(&sm.bar_q, 0);
        if (leader) bar_expect_tx(&sm.bar_q, 2 * q_bytes);
        for (int p = 0; p < P; ++p)
          tma_load_4d_pair(sm.q[p], &a.tm_q, bq, 64 * p, i_lo, g_first, grp);
      } else {
        bar_expect_tx(&sm.bar_q, q_bytes);
        for (int p = 0; p < P; ++p) tma_load_4d(sm.q[p], &a.tm_q, &sm.bar_q, 64 * p, i_lo, g_first, grp);
      }
      int uses[R];  // loads issued into each slot so far
#pragma unroll
      for (int x = 0; x < R; ++x) uses[x] = 0;
      auto load = [&](int s, bool is_v, int t) -> bool {
        const uint16_t e = sm.tiles[t];
        const bool chunk = (e & kTileChunk) != 0;
        const int row0 = (e & kTileIdxMask) * kTileN;
        const CUtensorMap* m =
            is_v ? (chunk ? &a.tm_vn : &a.tm_vc) : (chunk ? &a.tm_kn : &a.tm_kc);
        const int u = uses[s];
        if (u > 0 && !wait_b<kPair>(&sm.bar_empty[s], (u - 1) & 1, abort_flag)) return false;
        if constexpr (kPair) {
          // this CTA's half: keys 64 rank .. of a K tile (both column panels),
          // columns 64 rank .. of a V tile (all 128 keys)
          const uint32_t bf = cluster_addr(&sm.bar_full[s], 0);
          if (leader) bar_expect_tx(&sm.bar_full[s], 2 * G::kSlotBytes);
          if (is_v) {
            tma_load_3d_pair(sm.kv[s], m, bf, 64 * static_cast<int>(rank), row0, grp);
          } else {
            for (int p = 0; p < P; ++p)
              tma_load_3d_pair(sm.kv[s] + p * G::kKPanelBytes, m, bf, 64 * p,
                               row0 + (kTileN / 2) * static_cast<int>(rank), grp);
          }
        } else {
          bar_expect_tx(&sm.bar_full[s], G::kSlotBytes);
          for (int p = 0; p < P; ++p)
            tma_load_3d(sm.kv[s] + p * G::kKPanelBytes, m, &sm.bar_full[s], 64 * p, row0, grp);
        }
        uses[s] = u + 1;
        return true;
      };
      // pass 1: K_0..K_{n-1} over all slots; pass 2: K_t (ring A) interleaved
      // with V_{t-2} (ring B), then the last V's
      bool ok = true;
      for (int t = 0; ok && t < n_t; ++t) ok = load(t % R, false, t);
      const int n_t2 = a.lse != nullptr ? 0 : n_t;  // pass 2's tiles
      for (int t = 0; ok && t < n_t2; ++t) {
        ok = load(t % RA, false, t);
        if (ok && t >= 2) ok = load(RA + (t - 2) % RB, true, t - 2);
      }
      for (int t = max(0, n_t2 - 2); ok && t < n_t2; ++t) ok = load(RA + t % RB, true, t);
      if (*abort_flag) {
        // Let copies still in flight land before the CTA's shared memory goes
        // away: at most the latest load of each slot can be outstanding.  On a
        // pair the copies are counted on the even CTA's barriers, so this CTA
        // also gives them a fixed grace period.
        volatile int never = 0;
        if (leader)
          for (int x = 0; x < R; ++x)
            if (uses[x] > 0) wait_bar(&sm.bar_full[x], (uses[x] - 1) & 1, &never, 100000000ull);
        const uint64_t t0 = global_timer_ns();
        while (kPair && global_timer_ns() - t0 < 200000ull) {
        }
      }
    }
  } else if (warp < kFirstSoftmaxWarp) {
    // ------------------------------------------------------- MMA issuers --
    // Warps 1 and 3 issue the Q K^T of the even and the odd tiles of each
    // pass, warp 2 every P V (it owns the O accumulator).  An issuing thread
    // runs only about one MMA ahead of the tensor pipe and then spends several
    // hundred cycles on commits, barrier waits and the next tile's indices, so
    // the pipe is kept busy by having these threads overlap.  A ring slot's
    // loads are all consumed by the Q K^T issuer of the slot's parity (slot n
    // mod 10 in pass 1, t mod 6 in pass 2) or by the P V issuer, in order, so
    // no full-barrier wait can run two phases ahead.  On a pair only the even
    // CTA issues.
    if (lane == 0 && n_t > 0 && leader) {
      constexpr int kM = kPair ? 2 * kTileM : kTileM;
      constexpr uint32_t kIdescQK = idesc_bf16_f32(kM, kTileN, false);
      constexpr uint32_t kIdescPV = idesc_bf16_f32(kM, D, true);
      // Descriptors: per MMA only the 14-bit start-address field advances
      // (bytes >> 4): a K-step of 16 bf16 is 32 B inside a 128-B swizzle row, a
      // 64-column panel is 16 KB for Q (8 KB for a pair's half K tile), a ring
      // slot is kSlotBytes, 16 rows of V are 2 KB.  All eight are formed
      // before the first MMA of a tile is issued.
      constexpr uint32_t kQPanel = (kTileM * 128) >> 4;
      constexpr uint32_t kKPanel = G::kKPanelBytes >> 4;
      constexpr uint32_t kSlot = G::kSlotBytes >> 4;
      constexpr int RA = G::kRA, RB = G::kRB;
      static_assert(RA % 2 == 0 && (RA + RB) % 2 == 0, "ring slots split by issuer parity");
      const bool is_pv = warp == 2;
      const int par = warp == 1 ? 0 : 1;  // the Q K^T issuer's tile parity
      const uint64_t q_desc = sdesc_sw128(smem_addr(sm.q[0]), 16, 1024);
      const uint64_t k_desc0 = sdesc_sw128(smem_addr(sm.kv[0]), 16, 1024);
      uint64_t qd[8];
#pragma unroll
      for (int kk = 0; kk < 8; ++kk) qd[kk] = q_desc + kQPanel * (kk / 4) + 2 * (kk % 4);
      // S_n = Q K_t^T (tile t = n, or n - n_t in pass 2) into its S buffer
      auto issue_qk = [&](int n) -> bool {
        int buf, suse;
        s_buffer(n, n_t, buf, suse);
        // buffer reuse: a pass-1 S is released when the softmax has loaded
        // it, a pass-2 one when the P V that read its P has completed
        if (suse > 0) {
          const int c1 = pass1_buffer_uses(n_t, buf);
          const bool ok_wait =
              suse <= c1 ? wait_b<kPair>(&sm.bar_sread[buf], (suse - 1) & 1, abort_flag)
                         : wait_b<kPair>(&sm.bar_pvdone[buf], (suse - 1 - c1) & 1, abort_flag);
          if (!ok_wait) return false;
        }
        int s, use;
        if (n < n_t) {
          s = n % (RA + RB);
          use = n / (RA + RB);
        } else {
          s = (n - n_t) % RA;
          use = pass1_uses(n_t, RA + RB, s) + (n - n_t) / RA;
        }
        if (!wait_b<kPair>(&sm.bar_full[s], use & 1, abort_flag)) return false;
        tc_fence_after_sync();
        const uint64_t kd = k_desc0 + static_cast<uint64_t>(s) * kSlot;
        const uint32_t d_tmem = tS + buf * 128;
        if constexpr (D == 128) {
          uint64_t bd[8];
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) bd[kk] = kd + kKPanel * (kk / 4) + 2 * (kk % 4);
          mma_ss_x8<kPair>(d_tmem, qd, bd, kIdescQK, 0u);
        } else {
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk)
            mma_ss(d_tmem, qd[kk], kd + kKPanel * (kk / 4) + 2 * (kk % 4), kIdescQK, kk > 0 ? 1u : 0u);
        }
        commit_all<kPair>(&sm.bar_sfull[buf]);
        commit_all<kPair>(&sm.bar_empty[s]);
        return true;
      };
      bool ok = wait_b<kPair>(&sm.bar_q, 0, abort_flag);
      if (!is_pv) {
        for (int n = par; ok && n < n_t; n += 2) ok = issue_qk(n);
        for (int t = par; ok && a.lse == nullptr && t < n_t; t += 2) ok = issue_qk(n_t + t);
      } else {
        const uint64_t v_desc0 = sdesc_sw128(smem_addr(sm.kv[RA]), kTileN * 128, 1024);
        for (int t = 0; ok && a.lse == nullptr && t < n_t; ++t) {
          const int pb = t % kSBufs2;  // the S buffer of pass-2 tile t holds its P
          if (!wait_b<kPair>(&sm.bar_pfull[pb], (t / kSBufs2) & 1, abort_flag)) {
            ok = false;
            break;
          }
          const int vs = RA + t % RB;
          const int use = pass1_uses(n_t, RA + RB, vs) + t / RB;
          if (!wait_b<kPair>(&sm.bar_full[vs], use & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint64_t vd = v_desc0 + static_cast<uint64_t>(t % RB) * kSlot;
          uint64_t bd[8];
#pragma unroll
          for (int kk = 0; kk < 8; ++kk) bd[kk] = vd + 128 * kk;
          // keys 32w .. 32w+31 (two K-steps) as bf16 pairs in columns
          // 32w .. 32w+15 of the buffer
          mma_ts_x8<kPair>(tO, tS + 128 * pb, bd, kIdescPV, t > 0 ? 1u : 0u);
          commit_all<kPair>(&sm.bar_empty[vs]);
          commit_all<kPair>(&sm.bar_pvdone[pb]);
        }
        if (ok && a.lse == nullptr) commit_all<kPair>(&sm.bar_ofull);
      }
      // No MMA of this thread may still be running when TMEM is freed.
      uint64_t* drain = &sm.bar_drain[warp - 1];
      if constexpr (kPair) mma_commit_pair(drain, 1);
      else mma_commit(drain);
      volatile int never = 0;
      wait_b<kPair>(drain, 0, &never);
    }
  } else {
    // ------------------------------------------- softmax / column sums --
    // Pass 1: two teams of two warpgroups take alternate tiles (team 0 even,
    // team 1 odd), so one team's exp-bound phase overlaps the other team's TMEM
    // loads and barrier waits; within a team, warpgroup u owns key columns
    // 64u .. 64u+63.  Pass 2 is a chain (Q K^T, softmax, P V, and the next
    // Q K^T into the freed buffer), so there all four warpgroups take every
    // tile, warpgroup w its key columns 32w .. 32w+31, which halves the
    // softmax's share of that chain.
    const int sw = warp - kFirstSoftmaxWarp;
    const int wg = sw >> 2;          // 0..3
    const int team = wg >> 1;
    const int u = wg & 1;
    const int q4 = warp & 3;         // TMEM lane quarter (hardware: warp id % 4)
    const int row = q4 * 32 + static_cast<int>(lane);
    // tile row -> (head within the group, chunk row i); false for padding rows
    auto row_info = [&](int r, int& gg, int& ii) -> bool {
      gg = g_first;
      ii = i_lo;
      if (!has_rows) return false;
      if (a.tiles_per_head > 0) {
        ii = i_lo + r;
        return ii < a.S;
      }
      gg = g_first + r / a.rows_box;
      ii = r % a.rows_box;
      return r < box_rows && ii < a.S && gg < a.qg;
    };
    int g, i;
    const bool valid = row_info(row, g, i);
    const int qpos = a.pos0 + i;
    const int hq = hkv * a.qg + g;
    // Pass 2 reads S in the 16x256b layout: this thread then holds rows
    // 32 q4 + lane/4 + 8x (x = 0..3) and columns 8k + 2(lane%4) + {0,1}.
    int i4[4];
    bool v4[4];
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      int gg;
      v4[x] = row_info(q4 * 32 + static_cast<int>(lane >> 2) + 8 * x, gg, i4[x]);
    }
    // After the column reduce-scatter this lane holds column cl of a 32-block.
    const int cl = 8 * static_cast<int>((lane >> 3) & 3) + 2 * static_cast<int>(lane & 3) +
                   static_cast<int>((lane >> 2) & 1);
    const uint32_t lane_addr = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = a.scale_log2;
    const int* sp_base = a.slot_pos + static_cast<size_t>(grp) * a.M;
    float* inc_base = a.score_inc + static_cast<size_t>(b * a.Hq + hkv * a.qg) * NK;
    // head (within the group) of each lane quarter's rows; -1 = no valid rows
    int warp_head[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      int gw = -1;
      if (has_rows) {
        if (a.tiles_per_head > 0) gw = (i_lo + w * 32 < a.S) ? g_first : -1;
        else gw = (w * 32 < box_rows) ? g_first + (w * 32) / a.rows_box : -1;
      }
      warp_head[w] = (gw >= 0 && gw < a.qg) ? gw : -1;
    }
    // this CTA's row of column-sum partials (three or more row tiles per
    // head: all 128 rows belong to query head g_first, row tile rt % tph);
    // the columns of tiles neither CTA of the pair visits are zeroed here,
    // the others are stored by the combine after each pass-2 tile
    float* prow = nullptr;
    if (a.colpart != nullptr && has_rows) {
      prow = a.colpart + (static_cast<size_t>(b * a.Hq + hkv * a.qg + g_first) * a.tiles_per_head +
                          rt % a.tiles_per_head) * NK;
      const int total = a.n_cache_tiles + a.n_chunk_tiles;
      for (int tt = sw; tt < total; tt += kSoftmaxWarps) {
        if (sm.cls[tt] != 0) continue;
        const bool ch = tt >= a.n_cache_tiles;
        const int c0 = (ch ? tt - a.n_cache_tiles : tt) * kTileN;
        const int c1 = min(c0 + kTileN, ch ? a.S : a.M);
        for (int c = c0 + static_cast<int>(lane); c < c1; c += 32) prow[(ch ? a.M : 0) + c] = 0.f;
      }
    }
    float m_run = -INFINITY, l_run = 0.f;
    float lam4[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
    float2 nl4[4];  // (-lam, -lam) of the four rows, for the packed FMAs
#pragma unroll
    for (int x = 0; x < 4; ++x) nl4[x] = make_float2(-INFINITY, -INFINITY);
    bool ok = true;
    bool have_lambda = false;
    int k2 = 0;  // pass-2 tiles this warp has processed (column-sum buffer phase)
    const int n_end = a.lse != nullptr ? n_t : 2 * n_t;  // pass 1 only when lse is asked
    // this team's pass-1 tiles, then every pass-2 tile
    auto next_step = [n_t](int n) { return n >= n_t ? n + 1 : (n + 2 < n_t ? n + 2 : n_t); };
    for (int n = team < n_t ? team : n_t; ok && n < n_end; n = next_step(n)) {
      int buf, suse;
      s_buffer(n, n_t, buf, suse);
      const bool pass2 = n >= n_t;
      const int t = pass2 ? n - n_t : n;
      if (pass2 && !have_lambda) {
        // publish this thread's row statistics, then combine all four parts of
        // every row (§A.6.1 merge)
        sm.rowstat[wg][row][0] = m_run;
        sm.rowstat[wg][row][1] = l_run;
        __syncwarp();
        if (lane == 0) bar_arrive(&sm.bar_rowstat);
        if (!wait_bar(&sm.bar_rowstat, 0, abort_flag, kWaitLimitNs)) {
          ok = false;
          break;
        }
#pragma unroll
        for (int x = 0; x < 4; ++x) {
          const int r = q4 * 32 + static_cast<int>(lane >> 2) + 8 * x;
          float mm = -INFINITY;
#pragma unroll
          for (int w = 0; w < kNumWG; ++w) mm = fmaxf(mm, sm.rowstat[w][r][0]);
          float l = 0.f;
#pragma unroll
          for (int w = 0; w < kNumWG; ++w)
            l += sm.rowstat[w][r][1] * fast_exp2(sm.rowstat[w][r][0] - mm);
          lam4[x] = (v4[x] && mm > -INFINITY) ? mm + fast_log2(l) : INFINITY;
          nl4[x] = make_float2(-lam4[x], -lam4[x]);
          // the row's log-sum-exp in natural-log units, for a later backward
          // (the first warpgroup of a team, one lane of the four per row)
          if (a.lse_out != nullptr && u == 0 && (lane & 3u) == 0u && v4[x]) {
            int gg, ii;
            row_info(r, gg, ii);
            a.lse_out[static_cast<size_t>(b * a.Hq + hkv * a.qg + gg) * a.S + ii] =
                lam4[x] * 0.6931471805599453f;
          }
        }
        have_lambda = true;
      }
      if (!wait_b<kPair>(&sm.bar_sfull[buf], suse & 1, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const uint16_t e = sm.tiles[t];
      const bool chunk = (e & kTileChunk) != 0;
      const bool partial = (e & kTilePartial) != 0;
      if (!pass2) {
        const uint32_t s_base = tS + lane_addr + buf * 128 + u * 64;
        // pass 1 (one row per thread, 64 columns in two halves of 32): running
        // max and sum of exp2, updated after each half, so that only 32 values
        // are live; the S buffer is released once both halves are loaded
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          const int col0 = (e & kTileIdxMask) * kTileN + u * 64 + 32 * h;
          float v[32];
          {
            uint32_t r[32];
            tmem_ld32_async(s_base + 32 * h, r);
            tmem_wait_ld(r);
#pragma unroll
            for (int k = 0; k < 32; ++k) v[k] = __uint_as_float(r[k]);
          }
          if (h == 1) {
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) arrive_issuer<kPair>(&sm.bar_sread[buf]);  // S buffer may be overwritten
          }
          if (!partial) {
            // maximum: four chains of three-input max (16 instructions for 32
            // values); then exp2(s c - m) and the sum with packed fp32 pairs
            float c0 = max3f(v[0], v[1], v[2]), c1 = max3f(v[3], v[4], v[5]);
            float c2 = max3f(v[6], v[7], v[8]), c3 = max3f(v[9], v[10], v[11]);
#pragma unroll
            for (int k = 12; k < 28; k += 8) {
              c0 = max3f(c0, v[k], v[k + 1]);
              c1 = max3f(c1, v[k + 2], v[k + 3]);
              c2 = max3f(c2, v[k + 4], v[k + 5]);
              c3 = max3f(c3, v[k + 6], v[k + 7]);
            }
            c0 = max3f(c0, v[28], v[29]);
            c1 = max3f(c1, v[30], v[31]);
            const float m_new = fmaxf(m_run, max3f(c0, c1, fmaxf(c2, c3)) * sl2);
            const float2 sc = make_float2(sl2, sl2), nm = make_float2(-m_new, -m_new);
            float2 a0 = make_float2(0.f, 0.f), a1 = make_float2(0.f, 0.f);
#pragma unroll
            for (int k = 0; k < 32; k += 4) {
              const float2 x = ffma2(make_float2(v[k], v[k + 1]), sc, nm);
              const float2 y = ffma2(make_float2(v[k + 2], v[k + 3]), sc, nm);
              a0 = fadd2(a0, make_float2(fast_exp2(x.x), fast_exp2(x.y)));
              a1 = fadd2(a1, make_float2(fast_exp2(y.x), fast_exp2(y.y)));
            }
            const float2 s = fadd2(a0, a1);
            l_run = l_run * fast_exp2(m_run - m_new) + (s.x + s.y);
            m_run = m_new;
          } else {
            uint32_t vis = 0u;  // bit k: column col0 + k visible to this row
            if (valid) {
              if (chunk) {
#pragma unroll
                for (int k = 0; k < 32; ++k)
                  if (col0 + k <= i && col0 + k < a.S) vis |= 1u << k;
              } else {
                for (int k = 0; k < 32; ++k) {
                  const int j = col0 + k;
                  const int pos = j < a.M ? __ldg(sp_base + j) : -1;
                  if (pos >= 0 && pos <= qpos) vis |= 1u << k;
                }
              }
            }
            float mx = -INFINITY;
#pragma unroll
            for (int k = 0; k < 32; ++k)
              if ((vis >> k) & 1u) mx = fmaxf(mx, v[k] * sl2);
            const float m_new = fmaxf(m_run, mx);
            if (m_new > -INFINITY) {
              float s0 = 0.f, s1 = 0.f;
#pragma unroll
              for (int k = 0; k < 32; k += 2) {
                if ((vis >> k) & 1u) s0 += fast_exp2(fmaf(v[k], sl2, -m_new));
                if ((vis >> (k + 1)) & 1u) s1 += fast_exp2(fmaf(v[k + 1], sl2, -m_new));
              }
              l_run = l_run * fast_exp2(m_run - m_new) + (s0 + s1);
              m_run = m_new;
            }
          }
        }
      } else {
        // pass 2 (16x256b layout), this warpgroup's 32 columns: P in fp32,
        // its bf16 copy over the first 16 of those TMEM columns (loaded
        // before any P is stored) for P V, column sums of the fp32 P
        const int cb = k2 & (kColBufs - 1);
        const uint32_t s_base = tS + lane_addr + buf * 128 + wg * 32;
        const uint32_t p_base = s_base;
        {
          const int col0 = (e & kTileIdxMask) * kTileN + wg * 32;
          float pa[16], pb[16];  // rows lane/4 + {0, 8} and + {16, 24}
          {
            uint32_t r[32];
            tmem_ld_16x256b_x4x2_async(s_base, r);
            tmem_wait_ld(r);
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              pa[k] = __uint_as_float(r[k]);
              pb[k] = __uint_as_float(r[16 + k]);
            }
          }
          if (!partial) {
            // registers 4k, 4k+1 hold row A (pa) / C (pb), 4k+2, 4k+3 row B / D,
            // each a pair of adjacent columns: one packed FMA per pair
            const float2 sc = make_float2(sl2, sl2);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              const float2 xa = ffma2(make_float2(pa[4 * k], pa[4 * k + 1]), sc, nl4[0]);
              const float2 xb = ffma2(make_float2(pa[4 * k + 2], pa[4 * k + 3]), sc, nl4[1]);
              const float2 xc = ffma2(make_float2(pb[4 * k], pb[4 * k + 1]), sc, nl4[2]);
              const float2 xd = ffma2(make_float2(pb[4 * k + 2], pb[4 * k + 3]), sc, nl4[3]);
              pa[4 * k] = fast_exp2(xa.x);
              pa[4 * k + 1] = fast_exp2(xa.y);
              pa[4 * k + 2] = fast_exp2(xb.x);
              pa[4 * k + 3] = fast_exp2(xb.y);
              pb[4 * k] = fast_exp2(xc.x);
              pb[4 * k + 1] = fast_exp2(xc.y);
              pb[4 * k + 2] = fast_exp2(xd.x);
              pb[4 * k + 3] = fast_exp2(xd.y);
            }
          } else {
#pragma unroll
            for (int k = 0; k < 4; ++k) {
#pragma unroll
              for (int ee = 0; ee < 2; ++ee) {
                const int c = col0 + 8 * k + 2 * static_cast<int>(lane & 3) + ee;
                bool vis[4];
                if (chunk) {
#pragma unroll
                  for (int x = 0; x < 4; ++x) vis[x] = c <= i4[x] && c < a.S;
                } else {
                  const int pos = c < a.M ? __ldg(sp_base + c) : -1;
#pragma unroll
                  for (int x = 0; x < 4; ++x) vis[x] = pos >= 0 && pos <= a.pos0 + i4[x];
                }
                const int ia = 4 * k + ee, ib = 4 * k + 2 + ee;
                pa[ia] = vis[0] ? fast_exp2(fmaf(pa[ia], sl2, -lam4[0])) : 0.f;
                pa[ib] = vis[1] ? fast_exp2(fmaf(pa[ib], sl2, -lam4[1])) : 0.f;
                pb[ia] = vis[2] ? fast_exp2(fmaf(pb[ia], sl2, -lam4[2])) : 0.f;
                pb[ib] = vis[3] ? fast_exp2(fmaf(pb[ib], sl2, -lam4[3])) : 0.f;
              }
            }
          }
          {
            uint32_t pk[8];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              pk[2 * k] = pack_bf16x2(pa[4 * k], pa[4 * k + 1]);
              pk[2 * k + 1] = pack_bf16x2(pa[4 * k + 2], pa[4 * k + 3]);
            }
            tmem_st_16x128b_x4_async(p_base, pk);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              pk[2 * k] = pack_bf16x2(pb[4 * k], pb[4 * k + 1]);
              pk[2 * k + 1] = pack_bf16x2(pb[4 * k + 2], pb[4 * k + 3]);
            }
            tmem_st_16x128b_x4_async(p_base + (16u << 16), pk);
          }
          // column sums: 4 rows in-thread, then a reduce-scatter over lane bits
          // 4, 3, 2 leaves one column (summed over the warp's 32 rows) per lane
          float v[8];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            const float2 cs =
                fadd2(fadd2(make_float2(pa[4 * k], pa[4 * k + 1]), make_float2(pa[4 * k + 2], pa[4 * k + 3])),
                      fadd2(make_float2(pb[4 * k], pb[4 * k + 1]), make_float2(pb[4 * k + 2], pb[4 * k + 3])));
            v[2 * k] = cs.x;
            v[2 * k + 1] = cs.y;
          }
          rs_step<8, 16>(v, lane);
          rs_step<4, 8>(v, lane);
          rs_step<2, 4>(v, lane);
          sm.colsum[cb][wg][q4][cl] = v[0];
        }
        if (!ok) break;
        tmem_wait_st();
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) arrive_issuer<kPair>(&sm.bar_pfull[buf]);
        // The last of the warpgroup's four warps to get here adds the four
        // quarters' partial sums per query head and issues the reductions; the
        // others go straight on to their next tile.  The counter only grows
        // (four per tile), so "last" is old % 4 == 3.  Buffer cb is written
        // again four tiles later, after every warp's P arrival for the next
        // tile, which comes after the reads below in program order (see
        // kColBufs).
        int last = 0;
        if (lane == 0) last = (atomic_add_acq_rel_cta(&sm.cs_count[cb][wg], 1u) & 3u) == 3u;
        last = __shfl_sync(0xffffffffu, last, 0);
        if (last) {
          __syncwarp();
          const int colb = (e & kTileIdxMask) * kTileN + wg * 32;
          {
            const int c = static_cast<int>(lane);
            const int col = colb + c;
            if (prow != nullptr && (chunk ? col < a.S : col < a.M)) {
              // one head: the four quarters in order, stored (rows past S
              // have p = 0)
              float acc = 0.f;
#pragma unroll
              for (int w = 0; w < 4; ++w) acc += sm.colsum[cb][wg][w][c];
              prow[(chunk ? a.M : 0) + col] = acc;
            } else if (chunk ? col < a.S : col < a.M) {
              float* dst = inc_base + (chunk ? a.M + col : col);
              float acc = 0.f;
#pragma unroll
              for (int w = 0; w < 4; ++w) {
                acc += sm.colsum[cb][wg][w][c];
                const int gw = warp_head[w];
                const int gn = w < 3 ? warp_head[w + 1] : -2;
                if (gn != gw) {
                  if (gw >= 0 && acc != 0.f) red_add_f32(dst + static_cast<size_t>(gw) * NK, acc);
                  acc = 0.f;
                }
              }
            }
          }
        }
        ++k2;
      }
    }
    if (ok && !have_lambda && n_t > 0) {
      // this team had no pass-2 tile: it still takes part in the row merge
      sm.rowstat[wg][row][0] = m_run;
      sm.rowstat[wg][row][1] = l_run;
      __syncwarp();
      if (lane == 0) bar_arrive(&sm.bar_rowstat);
    }
    if (a.lse != nullptr && ok && n_t > 0 && wait_bar(&sm.bar_rowstat, 0, abort_flag, kWaitLimitNs)) {
      // pass 1 only: the merged log-sum-exp of each row (§A.6.1) and, for the
      // backward, D = dout . out.  Warpgroup wg takes rows q4 32 + lane/4 +
      // 8 wg; the four lanes holding a row (16x256b layout) each take a
      // quarter of d for D, and the first of them writes both values.
      const int r = q4 * 32 + static_cast<int>(lane >> 2) + 8 * wg;
      int gg = 0, ii = 0;
      const bool has = row_info(r, gg, ii);
      float dsum = 0.f;
      if (has && a.drow != nullptr) {
        const size_t orow = (static_cast<size_t>(b * a.Hq + hkv * a.qg + gg) * a.S + ii) * D +
                            (lane & 3u) * (D / 4);
        const uint4* o4 = reinterpret_cast<const uint4*>(a.bwd_out + orow);
        const uint4* g4 = reinterpret_cast<const uint4*>(a.bwd_dout + orow);
#pragma unroll
        for (int k = 0; k < D / 32; ++k) {
          const uint4 o = __ldg(o4 + k), g = __ldg(g4 + k);
          const uint32_t ow[4] = {o.x, o.y, o.z, o.w}, gw[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            dsum = fmaf(__uint_as_float(ow[e] << 16), __uint_as_float(gw[e] << 16), dsum);
            dsum = fmaf(__uint_as_float(ow[e] & 0xFFFF0000u), __uint_as_float(gw[e] & 0xFFFF0000u), dsum);
          }
        }
      }
      dsum += __shfl_xor_sync(0xffffffffu, dsum, 1);
      dsum += __shfl_xor_sync(0xffffffffu, dsum, 2);
      if (has && (lane & 3u) == 0u) {
        float mm = -INFINITY;
#pragma unroll
        for (int w = 0; w < kNumWG; ++w) mm = fmaxf(mm, sm.rowstat[w][r][0]);
        float l = 0.f;
#pragma unroll
        for (int w = 0; w < kNumWG; ++w)
          l += sm.rowstat[w][r][1] * fast_exp2(sm.rowstat[w][r][0] - mm);
        const size_t li = static_cast<size_t>(grp) * a.lse_stride + gg * a.S + ii;
        a.lse[li] = mm + fast_log2(l);
        if (a.drow != nullptr) a.drow[li] = dsum;
      }
    }
    // ------------------------------------------------------------ epilogue --
    if (ok && n_t > 0 && a.lse == nullptr && wait_b<kPair>(&sm.bar_ofull, 0, abort_flag)) {
      tc_fence_after_sync();
      constexpr int kPart = D / kNumWG;  // O columns per warpgroup: 32 or 16
      uint32_t pk[kPart / 2];
      if constexpr (kPart == 32) {
        uint32_t r[32];
        tmem_ld32(tO + lane_addr + wg * kPart, r);
#pragma unroll
        for (int x = 0; x < 16; ++x)
          pk[x] = pack_bf16x2(__uint_as_float(r[2 * x]), __uint_as_float(r[2 * x + 1]));
      } else {
        uint32_t r[16];
        tmem_ld16(tO + lane_addr + wg * kPart, r);
#pragma unroll
        for (int x = 0; x < 8; ++x)
          pk[x] = pack_bf16x2(__uint_as_float(r[2 * x]), __uint_as_float(r[2 * x + 1]));
      }
      if (valid) {
        uint16_t* dst = a.out + (static_cast<size_t>(b * a.Hq + hq) * a.S + i) * D + wg * kPart;
        uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
        for (int x = 0; x < kPart / 8; ++x)
          d4[x] = make_uint4(pk[4 * x], pk[4 * x + 1], pk[4 * x + 2], pk[4 * x + 3]);
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  // On a pair, neither CTA frees TMEM or leaves (its shared memory holds
  // barriers and operands the other one uses) before both are done.
  if constexpr (kPair) cluster_sync_all();
  if (warp == 1) {
    __syncwarp();
    if constexpr (kPair) tmem_dealloc_pair(tmem, 512);
    else tmem_dealloc(tmem, 512);
  }
  if (tid == 0 && sm.abort_flag) atomicOr(a.err, 1);
}

template <int D, bool kPair>
cudaError_t launch_d(const SdpaArgs& a, cudaStream_t stream) {
  const size_t smem = sizeof(SdpaSmem<D, kPair>) + 1024;
  static OncePerDevice configured;
  cudaError_t e = configured.run([smem](int) {
    return cudaFuncSetAttribute(sdpa_chunk_kernel<D, kPair>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
  });
  if (e != cudaSuccess) return e;
  const int ctas = kPair ? 2 * ((a.n_row_tiles + 1) / 2) : a.n_row_tiles;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(ctas), static_cast<unsigned>(a.B * a.Hkv));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = kPair ? 2 : 1;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, sdpa_chunk_kernel<D, kPair>, a);
}

}  // namespace

cudaError_t launch_sdpa(const SdpaArgs& a, cudaStream_t stream) {
  return a.d == 64 ? launch_d<64, false>(a, stream) : launch_d<128, true>(a, stream);
}

namespace {

constexpr int kReduceThreads = 256;

// One thread per score_inc element: the row tiles' partials in row-tile order
// (all loads issued before the adds).
__global__ void __launch_bounds__(kReduceThreads) colsum_reduce_kernel(
    const float* __restrict__ part, float* __restrict__ score_inc, int rows, int tph, int nk) {
  if (threadIdx.x == 0) launch_dependents();  // the update may be placed now
  grid_dependency_wait();                      // the attention kernel's partials
  const int col = blockIdx.x * kReduceThreads + static_cast<int>(threadIdx.x);
  if (col >= nk) return;
  for (int row = blockIdx.y; row < rows; row += gridDim.y) {
  const float* p = part + static_cast<size_t>(row) * tph * nk + col;
  float acc = __ldg(p);
  int r = 1;
  for (; r + 4 <= tph; r += 4) {
    const float x0 = __ldg(p + static_cast<size_t>(r) * nk);
    const float x1 = __ldg(p + static_cast<size_t>(r + 1) * nk);
    const float x2 = __ldg(p + static_cast<size_t>(r + 2) * nk);
    const float x3 = __ldg(p + static_cast<size_t>(r + 3) * nk);
    acc = (((acc + x0) + x1) + x2) + x3;
  }
  for (; r < tph; ++r) acc += __ldg(p + static_cast<size_t>(r) * nk);
  score_inc[static_cast<size_t>(row) * nk + col] = acc;
  }
}

}  // namespace

size_t sdpa_colpart_bytes(int B, int Hq, int S, int M) {
  const int tph = S > kTileM ? (S + kTileM - 1) / kTileM : 0;
  if (tph < kColpartMinTiles) return 0;
  return static_cast<size_t>(B) * Hq * tph * (static_cast<size_t>(M) + S) * sizeof(float);
}

cudaError_t launch_colsum_reduce(const float* colpart, float* score_inc, int rows, int tph, int nk,
                                 cudaStream_t stream) {
  const dim3 grid(static_cast<unsigned>((nk + kReduceThreads - 1) / kReduceThreads),
                  static_cast<unsigned>(rows < 65535 ? rows : 65535));
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kReduceThreads);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, colsum_reduce_kernel, colpart, score_inc, rows, tph, nk);
}

}  // namespace h2o
