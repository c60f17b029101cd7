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
//  * Warp roles: warp 0 issues TMA loads (Q once, then K tiles through ring A
//    and V tiles through ring B of shared-memory slots); warp 1 issues every
//    Q K^T and warp 2 every P V tcgen05 MMA, so one issuer keeps the tensor pipe
//    busy while the other waits on a barrier; warps 3-18 form four softmax
//    warpgroups in two teams that take alternate tiles; the two warpgroups of a
//    team own key columns 0-63 and 64-127 of their tiles.
//  * TMEM holds two fp32 S buffers, two bf16 P buffers and the O accumulator.
//    An S buffer is released as soon as the softmax has loaded it, so Q K^T of
//    later tiles never waits for P V; P is written as bf16 pairs into a P
//    buffer and consumed by the P V MMA directly from TMEM.
//  * Column sums use the fp32 P (not the bf16 copy fed to the MMA).  Pass 2
//    reads S in TMEM's 16x256b layout, where a thread holds 4 rows x 8
//    columns: it adds its 4 rows, a 3-step warp reduce-scatter leaves one
//    column sum (over the warp's 32 rows) per lane and 32-column block, the
//    four warps of a warpgroup combine through shared memory, and one red.global.add per
//    column and query head goes to score_inc (zeroed by the host call).
//    Pass 1 keeps one row per thread (32x32b layout) for the row statistics.
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
constexpr int kFirstSoftmaxWarp = 3;  // warp 0 TMA, warp 1 Q K^T issuer, warp 2 P V issuer
constexpr int kSoftmaxWarps = 4 * kNumWG;
constexpr int kThreads = 32 * (kFirstSoftmaxWarp + kSoftmaxWarps);  // 608
constexpr uint16_t kTileChunk = 0x8000;
constexpr uint16_t kTilePartial = 0x4000;
constexpr uint16_t kTileIdxMask = 0x3FFF;
constexpr uint8_t kClsSkip = 0, kClsFull = 1, kClsPartial = 2;
// TMEM: two S buffers (fp32, 128 columns each), two P buffers (bf16 pairs, 64
// columns each) and the O accumulator: 2*128 + 2*64 + 128 = 512 columns.  An S
// buffer is free again as soon as the softmax has loaded it; a P buffer when
// the P V that read it has completed.
constexpr int kSBufs = 2;
constexpr int kPBufs = 2;
constexpr int kPCols = kTileN / 2;

// K tiles go through ring A (consumed by the Q K^T issuer), V tiles through
// ring B (consumed by the P V issuer); each ring has a single consumer that
// takes its loads in order, which keeps every mbarrier wait at most one phase
// ahead.  Slots are 32 KB (d = 128) or 16 KB (d = 64).
template <int D>
__host__ __device__ constexpr int ring_a_slots() { return D == 128 ? 3 : 6; }
template <int D>
__host__ __device__ constexpr int ring_b_slots() { return D == 128 ? 2 : 4; }
template <int D>
__host__ __device__ constexpr int ring_slots() { return ring_a_slots<D>() + ring_b_slots<D>(); }

template <int D>
struct __align__(1024) SdpaSmem {
  static constexpr int kPanels = D / 64;
  uint8_t q[kPanels][kTileM * 128];
  uint8_t kv[ring_slots<D>()][kPanels][kTileN * 128];
  float colsum[2][kNumWG][4][64];  // [buffer][warpgroup][warp][column]
  float rowstat[kNumWG][kTileM][2];
  uint64_t bar_q;
  uint64_t bar_full[ring_slots<D>()], bar_empty[ring_slots<D>()];
  uint64_t bar_sfull[kSBufs], bar_sread[kSBufs], bar_pfull[kPBufs], bar_pvdone[kPBufs];
  uint64_t bar_cs[2][kNumWG];
  uint64_t bar_rowstat, bar_ofull, bar_drain[2];
  uint32_t taddr;
  int abort_flag;
  int n_tiles;
  uint8_t cls[kMaxKeyTiles];
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

template <int D>
__global__ void __launch_bounds__(kThreads, 1) sdpa_chunk_kernel(const __grid_constant__ SdpaArgs a) {
  constexpr int P = D / 64;
  extern __shared__ uint8_t smem_raw[];
  auto& sm = *reinterpret_cast<SdpaSmem<D>*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const uint32_t lane = tid & 31;
  const int grp = blockIdx.y;  // b * Hkv + kv head
  const int rt = blockIdx.x;   // row tile within the group
  const int b = grp / a.Hkv;
  const int hkv = grp % a.Hkv;
  const int NK = a.M + a.S;    // key columns per query head

  // Query rows of this tile: rows_box rows per head, heads_box heads.
  int g_first, i_lo, i_hi;
  if (a.tiles_per_head > 0) {
    g_first = rt / a.tiles_per_head;
    i_lo = (rt % a.tiles_per_head) * kTileM;
    i_hi = min(i_lo + kTileM, a.S) - 1;
  } else {
    g_first = rt * a.heads_box;
    i_lo = 0;
    i_hi = a.S - 1;
  }
  const int rows_used = a.tiles_per_head > 0 ? kTileM : a.rows_box * a.heads_box;

  if (tid == 0) {
    bar_init(&sm.bar_q, 1);
    for (int s = 0; s < ring_slots<D>(); ++s) {
      bar_init(&sm.bar_full[s], 1);
      bar_init(&sm.bar_empty[s], 1);
    }
    for (int x = 0; x < kSBufs; ++x) {
      bar_init(&sm.bar_sfull[x], 1);
      bar_init(&sm.bar_sread[x], kSoftmaxWarps / 2);  // the 8 warps of the team owning the tile
    }
    for (int x = 0; x < kPBufs; ++x) {
      bar_init(&sm.bar_pfull[x], kSoftmaxWarps / 2);
      bar_init(&sm.bar_pvdone[x], 1);
    }
    for (int x = 0; x < 2; ++x)
      for (int w = 0; w < kNumWG; ++w) bar_init(&sm.bar_cs[x][w], 4);
    bar_init(&sm.bar_rowstat, kSoftmaxWarps);
    bar_init(&sm.bar_ofull, 1);
    bar_init(&sm.bar_drain[0], 1);
    bar_init(&sm.bar_drain[1], 1);
    sm.abort_flag = 0;
    fence_bar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.taddr, 512);
    tmem_relinquish();
  }
  // Rows the Q box does not cover must still give finite logits.
  if (rows_used < kTileM) {
    const int words = (kTileM - rows_used) * 32;
    for (int p = 0; p < P; ++p)
      for (int x = tid; x < words; x += kThreads)
        reinterpret_cast<uint32_t*>(sm.q[p] + rows_used * 128)[x] = 0u;
    fence_proxy_async_smem();
  }
  // Classify key tiles against this CTA's rows.
  if (warp >= kFirstSoftmaxWarp) {
    const int sw = warp - kFirstSoftmaxWarp;
    const int* sp = a.slot_pos + static_cast<size_t>(grp) * a.M;
    const int lim_any = a.pos0 + i_hi;
    const int lim_all = a.pos0 + i_lo;
    for (int ct = sw; ct < a.n_cache_tiles; ct += kSoftmaxWarps) {
      bool any = false, all = true;
#pragma unroll
      for (int r = 0; r < 4; ++r) {
        const int j = ct * kTileN + r * 32 + static_cast<int>(lane);
        const int pos = j < a.M ? __ldg(sp + j) : -1;
        any |= pos >= 0 && pos <= lim_any;
        all &= pos >= 0 && pos <= lim_all;
      }
      any = __any_sync(0xffffffffu, any);
      all = __all_sync(0xffffffffu, all);
      if (lane == 0) sm.cls[ct] = any ? (all ? kClsFull : kClsPartial) : kClsSkip;
    }
    for (int c = sw; c < a.n_chunk_tiles; c += kSoftmaxWarps) {
      const int c0 = c * kTileN;
      uint8_t cl = kClsPartial;
      if (c0 > i_hi) cl = kClsSkip;
      else if (c0 + kTileN - 1 <= i_lo && c0 + kTileN <= a.S) cl = kClsFull;
      if (lane == 0) sm.cls[a.n_cache_tiles + c] = cl;
    }
  }
  __syncthreads();
  if (warp == kFirstSoftmaxWarp) {
    const int total = a.n_cache_tiles + a.n_chunk_tiles;
    int n = 0;
    for (int base = 0; base < total; base += 32) {
      const int t = base + static_cast<int>(lane);
      const uint8_t cl = t < total ? sm.cls[t] : kClsSkip;
      const uint32_t m = __ballot_sync(0xffffffffu, cl != kClsSkip);
      if (cl != kClsSkip) {
        const int pos = n + __popc(m & ((1u << lane) - 1u));
        uint16_t e = t < a.n_cache_tiles ? static_cast<uint16_t>(t)
                                         : static_cast<uint16_t>(kTileChunk | (t - a.n_cache_tiles));
        if (cl == kClsPartial) e |= kTilePartial;
        sm.tiles[pos] = e;
      }
      n += __popc(m);
    }
    if (lane == 0) sm.n_tiles = n;
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();

  const uint32_t tmem = sm.taddr;
  const uint32_t tS = tmem;                          // S buffer b: columns 128 b ..
  const uint32_t tP = tmem + 128 * kSBufs;           // P buffer p: columns 256 + 64 p ..
  const uint32_t tO = tP + kPCols * kPBufs;          // O accumulator: columns 384 ..
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
      bar_expect_tx(&sm.bar_q, P * 128 * a.rows_box * a.heads_box);
      for (int p = 0; p < P; ++p) tma_load_4d(sm.q[p], &a.tm_q, &sm.bar_q, 64 * p, i_lo, g_first, grp);
      constexpr int RA = ring_a_slots<D>(), RB = ring_b_slots<D>();
      int L[2] = {0, 0};  // loads issued per ring; ring r uses slots base_r + L % R_r
      auto load = [&](bool is_v, int t) -> bool {
        const uint16_t e = sm.tiles[t];
        const bool chunk = (e & kTileChunk) != 0;
        const int row0 = (e & kTileIdxMask) * kTileN;
        const CUtensorMap* m =
            is_v ? (chunk ? &a.tm_vn : &a.tm_vc) : (chunk ? &a.tm_kn : &a.tm_kc);
        const int r = is_v ? 1 : 0;
        const int R = is_v ? RB : RA;
        const int s = (is_v ? RA : 0) + L[r] % R;
        if (L[r] >= R &&
            !wait_bar(&sm.bar_empty[s], ((L[r] / R) - 1) & 1, abort_flag, kWaitLimitNs))
          return false;
        bar_expect_tx(&sm.bar_full[s], P * kTileN * 128);
        for (int p = 0; p < P; ++p) tma_load_3d(sm.kv[s][p], m, &sm.bar_full[s], 64 * p, row0, grp);
        ++L[r];
        return true;
      };
      // pass 1: K_0..K_{n-1}; pass 2: K_t interleaved with V_{t-2}, then the last V's
      bool ok = true;
      for (int t = 0; ok && t < n_t; ++t) ok = load(false, t);
      for (int t = 0; ok && t < n_t; ++t) {
        ok = load(false, t);
        if (ok && t >= 2) ok = load(true, t - 2);
      }
      for (int t = max(0, n_t - 2); ok && t < n_t; ++t) ok = load(true, t);
      if (*abort_flag) {
        // Let copies still in flight land before the CTA's shared memory goes away.
        volatile int never = 0;
        for (int x = max(0, L[0] - RA); x < L[0]; ++x)
          wait_bar(&sm.bar_full[x % RA], (x / RA) & 1, &never, 100000000ull);
        for (int x = max(0, L[1] - RB); x < L[1]; ++x)
          wait_bar(&sm.bar_full[RA + x % RB], (x / RB) & 1, &never, 100000000ull);
      }
    }
  } else if (warp == 1 || warp == 2) {
    // ------------------------------------------------------- MMA issuers --
    // Warp 1 issues every Q K^T (in tile order, so S buffers complete in
    // order); warp 2 issues every P V and owns the O accumulator.  With two
    // issuing threads the tensor pipe keeps working while one of them waits on
    // a barrier after its commits.
    if (lane == 0 && n_t > 0) {
      constexpr uint32_t kIdescQK = idesc_bf16_f32(kTileM, kTileN, false);
      constexpr uint32_t kIdescPV = idesc_bf16_f32(kTileM, D, true);
      // Descriptors are built once; per MMA only the 14-bit start-address
      // field advances, by compile-time immediates (bytes >> 4): a K-step of
      // 16 bf16 is 32 B inside a 128-B swizzle row, a 64-column panel is
      // 16 KB, a ring slot is P panels, 16 rows of V are 2 KB.
      constexpr uint32_t kPanel = (kTileN * 128) >> 4;
      constexpr uint32_t kSlot = P * kPanel;
      constexpr int RA = ring_a_slots<D>(), RB = ring_b_slots<D>();
      const bool is_qk = warp == 1;
      bool ok = true;
      if (is_qk) {
        const uint64_t q_desc = sdesc_sw128(smem_addr(sm.q[0]), 16, 1024);
        const uint64_t k_desc0 = sdesc_sw128(smem_addr(sm.kv[0][0]), 16, 1024);
        ok = wait_bar(&sm.bar_q, 0, abort_flag, kWaitLimitNs);
        for (int n = 0; ok && n < 2 * n_t; ++n) {
          const int buf = n % kSBufs;
          // buffer reuse: the softmax has loaded the S of tile n - 2
          if (n >= kSBufs &&
              !wait_bar(&sm.bar_sread[buf], ((n - kSBufs) / kSBufs) & 1, abort_flag, kWaitLimitNs)) {
            ok = false;
            break;
          }
          const int s = n % RA;  // ring A holds exactly the K tiles, in this order
          if (!wait_bar(&sm.bar_full[s], (n / RA) & 1, abort_flag, kWaitLimitNs)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint64_t kd = k_desc0 + static_cast<uint64_t>(s) * kSlot;
          const uint32_t d_tmem = tS + buf * 128;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = kPanel * (kk / 4) + 2 * (kk % 4);
            mma_ss(d_tmem, q_desc + off, kd + off, kIdescQK, kk > 0 ? 1u : 0u);
          }
          mma_commit(&sm.bar_sfull[buf]);
          mma_commit(&sm.bar_empty[s]);
        }
      } else {
        const uint64_t v_desc0 = sdesc_sw128(smem_addr(sm.kv[RA][0]), kTileN * 128, 1024);
        for (int t = 0; ok && t < n_t; ++t) {
          const int pb = t % kPBufs;
          if (!wait_bar(&sm.bar_pfull[pb], (t / kPBufs) & 1, abort_flag, kWaitLimitNs)) {
            ok = false;
            break;
          }
          const int vs = RA + t % RB;
          if (!wait_bar(&sm.bar_full[vs], (t / RB) & 1, abort_flag, kWaitLimitNs)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          const uint64_t vd = v_desc0 + static_cast<uint64_t>(t % RB) * kSlot;
          const uint32_t a_base = tP + kPCols * pb;
          const uint32_t acc0 = t > 0 ? 1u : 0u;
          // keys 16kk..16kk+15 sit as bf16 pairs in columns 8kk..8kk+7 of the P buffer
#pragma unroll
          for (int kk = 0; kk < kTileN / 16; ++kk)
            mma_ts(tO, a_base + 8 * kk, vd + 128 * kk, kIdescPV, kk > 0 ? 1u : acc0);
          mma_commit(&sm.bar_empty[vs]);
          mma_commit(&sm.bar_pvdone[pb]);
        }
        if (ok) mma_commit(&sm.bar_ofull);
      }
      // No MMA of this thread may still be running when TMEM is freed.
      mma_commit(&sm.bar_drain[is_qk ? 0 : 1]);
      volatile int never = 0;
      wait_bar(&sm.bar_drain[is_qk ? 0 : 1], 0, &never, kWaitLimitNs);
    }
  } else {
    // ------------------------------------------- softmax / column sums --
    // Two teams of two warpgroups take alternate tiles (team 0 even, team 1
    // odd), so one team's exp-bound phase overlaps the other team's TMEM loads,
    // column sums and barrier waits.  Within a team, warpgroup u owns key
    // columns 64u .. 64u+63 of its tiles.
    const int sw = warp - kFirstSoftmaxWarp;
    const int wg = sw >> 2;          // 0..3
    const int team = wg >> 1;
    const int u = wg & 1;
    const int q4 = warp & 3;         // TMEM lane quarter (hardware: warp id % 4)
    const int row = q4 * 32 + static_cast<int>(lane);
    // tile row -> (head within the group, chunk row i); false for padding rows
    auto row_info = [&](int r, int& gg, int& ii) -> bool {
      if (a.tiles_per_head > 0) {
        gg = g_first;
        ii = i_lo + r;
        return ii < a.S;
      }
      gg = g_first + r / a.rows_box;
      ii = r % a.rows_box;
      return r < rows_used && ii < a.S && gg < a.qg;
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
      int gw;
      if (a.tiles_per_head > 0) gw = (i_lo + w * 32 < a.S) ? g_first : -1;
      else gw = (w * 32 < rows_used) ? g_first + (w * 32) / a.rows_box : -1;
      warp_head[w] = (gw >= 0 && gw < a.qg) ? gw : -1;
    }
    float m_run = -INFINITY, l_run = 0.f;
    float lam4[4] = {INFINITY, INFINITY, INFINITY, INFINITY};
    bool ok = true;
    bool have_lambda = false;
    int k2 = 0;  // pass-2 tiles this warp has processed (column-sum buffer phase)
    for (int n = team; ok && n < 2 * n_t; n += 2) {
      const int buf = n % kSBufs;
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
        }
        have_lambda = true;
      }
      if (!wait_bar(&sm.bar_sfull[buf], (n / kSBufs) & 1, abort_flag, kWaitLimitNs)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const uint16_t e = sm.tiles[t];
      const bool chunk = (e & kTileChunk) != 0;
      const bool partial = (e & kTilePartial) != 0;
      const uint32_t s_base = tS + lane_addr + buf * 128 + u * 64;
      if (!pass2) {
        // pass 1 (one row per thread, 64 columns): running max and sum of exp2
        const int col0 = (e & kTileIdxMask) * kTileN + u * 64;
        float v[64];
        {
          uint32_t r[32];
          tmem_ld32_async(s_base, r);
          tmem_wait_ld(r);
#pragma unroll
          for (int k = 0; k < 32; ++k) v[k] = __uint_as_float(r[k]);
          tmem_ld32_async(s_base + 32, r);
          tmem_wait_ld(r);
#pragma unroll
          for (int k = 0; k < 32; ++k) v[32 + k] = __uint_as_float(r[k]);
        }
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) bar_arrive(&sm.bar_sread[buf]);  // S buffer may be overwritten
        if (!partial) {
          float mx0 = v[0], mx1 = v[1], mx2 = v[2], mx3 = v[3];
#pragma unroll
          for (int k = 4; k < 64; k += 4) {
            mx0 = fmaxf(mx0, v[k]);
            mx1 = fmaxf(mx1, v[k + 1]);
            mx2 = fmaxf(mx2, v[k + 2]);
            mx3 = fmaxf(mx3, v[k + 3]);
          }
          const float m_new = fmaxf(m_run, fmaxf(fmaxf(mx0, mx1), fmaxf(mx2, mx3)) * sl2);
          float s0 = 0.f, s1 = 0.f, s2 = 0.f, s3 = 0.f;
#pragma unroll
          for (int k = 0; k < 64; k += 4) {
            s0 += fast_exp2(fmaf(v[k], sl2, -m_new));
            s1 += fast_exp2(fmaf(v[k + 1], sl2, -m_new));
            s2 += fast_exp2(fmaf(v[k + 2], sl2, -m_new));
            s3 += fast_exp2(fmaf(v[k + 3], sl2, -m_new));
          }
          l_run = l_run * fast_exp2(m_run - m_new) + ((s0 + s1) + (s2 + s3));
          m_run = m_new;
        } else {
          uint64_t vis = 0ull;  // bit k: column col0 + k visible to this row
          if (chunk) {
#pragma unroll
            for (int k = 0; k < 64; ++k)
              if (col0 + k <= i && col0 + k < a.S) vis |= 1ull << k;
          } else {
            for (int k = 0; k < 64; ++k) {
              const int j = col0 + k;
              const int pos = j < a.M ? __ldg(sp_base + j) : -1;
              if (pos >= 0 && pos <= qpos) vis |= 1ull << k;
            }
          }
          float mx = -INFINITY;
#pragma unroll
          for (int k = 0; k < 64; ++k)
            if ((vis >> k) & 1ull) mx = fmaxf(mx, v[k] * sl2);
          const float m_new = fmaxf(m_run, mx);
          if (m_new > -INFINITY) {
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int k = 0; k < 64; k += 2) {
              if ((vis >> k) & 1ull) s0 += fast_exp2(fmaf(v[k], sl2, -m_new));
              if ((vis >> (k + 1)) & 1ull) s1 += fast_exp2(fmaf(v[k + 1], sl2, -m_new));
            }
            l_run = l_run * fast_exp2(m_run - m_new) + (s0 + s1);
            m_run = m_new;
          }
        }
      } else {
        // pass 2 (16x256b layout), in two halves of 32 columns: P in fp32,
        // bf16 copy to a TMEM P buffer for P V, column sums of the fp32 P
        const int cb = k2 & 1;
        const int pbuf = t % kPBufs;
        const uint32_t p_base = tP + lane_addr + kPCols * pbuf + u * 32;
#pragma unroll 1
        for (int h = 0; h < 2; ++h) {
          const uint32_t s_addr = s_base + 32 * h;
          const int col0 = (e & kTileIdxMask) * kTileN + u * 64 + 32 * h;
          float pa[16], pb[16];  // rows lane/4 + {0, 8} and + {16, 24}
          {
            uint32_t r[32];
            tmem_ld_16x256b_x4x2_async(s_addr, r);
            tmem_wait_ld(r);
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              pa[k] = __uint_as_float(r[k]);
              pb[k] = __uint_as_float(r[16 + k]);
            }
          }
          if (h == 1) {
            // both halves of S are in registers: the S buffer may be overwritten
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) bar_arrive(&sm.bar_sread[buf]);
          }
          if (!partial) {
#pragma unroll
            for (int k = 0; k < 16; ++k) {
              pa[k] = fast_exp2(fmaf(pa[k], sl2, -lam4[(k >> 1) & 1]));
              pb[k] = fast_exp2(fmaf(pb[k], sl2, -lam4[2 + ((k >> 1) & 1)]));
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
          if (h == 0 && t >= kPBufs) {
            // the P V of tile t - 2 must be done with this P buffer
            if (!wait_bar(&sm.bar_pvdone[pbuf], ((t - kPBufs) / kPBufs) & 1, abort_flag,
                          kWaitLimitNs)) {
              ok = false;
              break;
            }
            tc_fence_after_sync();
          }
          {
            uint32_t pk[8];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              pk[2 * k] = pack_bf16x2(pa[4 * k], pa[4 * k + 1]);
              pk[2 * k + 1] = pack_bf16x2(pa[4 * k + 2], pa[4 * k + 3]);
            }
            tmem_st_16x128b_x4(p_base + 16 * h, pk);
#pragma unroll
            for (int k = 0; k < 4; ++k) {
              pk[2 * k] = pack_bf16x2(pb[4 * k], pb[4 * k + 1]);
              pk[2 * k + 1] = pack_bf16x2(pb[4 * k + 2], pb[4 * k + 3]);
            }
            tmem_st_16x128b_x4(p_base + 16 * h + (16u << 16), pk);
          }
          // column sums: 4 rows in-thread, then a reduce-scatter over lane bits
          // 4, 3, 2 leaves one column (summed over the warp's 32 rows) per lane
          float v[8];
#pragma unroll
          for (int k = 0; k < 4; ++k) {
            v[2 * k] = (pa[4 * k] + pa[4 * k + 2]) + (pb[4 * k] + pb[4 * k + 2]);
            v[2 * k + 1] = (pa[4 * k + 1] + pa[4 * k + 3]) + (pb[4 * k + 1] + pb[4 * k + 3]);
          }
          rs_step<8, 16>(v, lane);
          rs_step<4, 8>(v, lane);
          rs_step<2, 4>(v, lane);
          sm.colsum[cb][wg][q4][32 * h + cl] = v[0];
        }
        if (!ok) break;
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) {
          bar_arrive(&sm.bar_pfull[pbuf]);
          bar_arrive(&sm.bar_cs[cb][wg]);
        }
        if (!wait_bar(&sm.bar_cs[cb][wg], (k2 >> 1) & 1, abort_flag, kWaitLimitNs)) {
          ok = false;
          break;
        }
        // one warp of the warpgroup (a different one every tile) adds the four
        // quarters' partial sums per query head and issues the reductions
        if (q4 == (k2 & 3)) {
          const int colb = (e & kTileIdxMask) * kTileN + u * 64;
#pragma unroll
          for (int hh = 0; hh < 2; ++hh) {
            const int c = 32 * hh + static_cast<int>(lane);
            const int col = colb + c;
            if (chunk ? col < a.S : col < a.M) {
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
    // ------------------------------------------------------------ epilogue --
    if (ok && n_t > 0 && wait_bar(&sm.bar_ofull, 0, abort_flag, kWaitLimitNs)) {
      tc_fence_after_sync();
      constexpr int kPart = D / kNumWG;  // O columns per warpgroup: 32 or 16
      uint16_t* dst = a.out + (static_cast<size_t>(b * a.Hq + hq) * a.S + i) * D + wg * kPart;
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
        uint4* d4 = reinterpret_cast<uint4*>(dst);
#pragma unroll
        for (int x = 0; x < kPart / 8; ++x)
          d4[x] = make_uint4(pk[4 * x], pk[4 * x + 1], pk[4 * x + 2], pk[4 * x + 3]);
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, 512);
  }
  if (tid == 0 && sm.abort_flag) atomicOr(a.err, 1);
}

template <int D>
cudaError_t launch_d(const SdpaArgs& a, cudaStream_t stream) {
  const size_t smem = sizeof(SdpaSmem<D>) + 1024;
  static bool configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 64 && !configured[dev]) {
    e = cudaFuncSetAttribute(sdpa_chunk_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  dim3 grid(a.n_row_tiles, a.B * a.Hkv);
  sdpa_chunk_kernel<D><<<grid, kThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_sdpa(const SdpaArgs& a, cudaStream_t stream) {
  return a.d == 64 ? launch_d<64>(a, stream) : launch_d<128>(a, stream);
}

}  // namespace h2o
