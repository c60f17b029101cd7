// Gradient of the chunk SDPA (§3.1 Eq. 2 under the position mask of §3.3.1):
// the backward pass the paper's fine-tuning runs through every chunk (§3.2,
// §A.4).  For L = sum(out * dout), with m_ij the attention weights of the
// forward, per (b, kv head) group with the q_g heads' rows stacked:
//
//   D_i    = sum_d dout_id out_id
//   dP_ij  = dout_i . v_j,   dS_ij = m_ij (dP_ij - D_i)
//   dq_i   = scale sum_j dS_ij k_j
//   dk_j   = scale sum_i dS_ij q_i,   dv_j = sum_i m_ij dout_i
//
// with m_ij = exp2(scale log2e q_i . k_j - lambda_i) rebuilt from each row's
// log-sum-exp lambda (log2 units), which the forward kernel's pass 1 writes.
// Hidden (i, j) pairs have m_ij = 0, so cache slots no row sees get zero
// gradients.
//
// Two kinds of tcgen05 CTA in one launch, neither materialising a score
// matrix and neither using atomics (so the result does not depend on
// scheduling):
//  * bwd_dq_kernel: one CTA per 128 stacked rows; per key tile, S = Q K^T and
//    dP = dO V^T into TMEM, the softmax warps (one row per thread) form dS in
//    bf16 over S's columns, and dQ += dS K accumulates in TMEM.
//  * bwd_dkv_kernel: one CTA per 128-key tile; per tile of stacked rows,
//    S^T = K Q^T and dP^T = V dO^T into TMEM (one key per lane), the softmax
//    warps form P^T and dS^T in bf16 over those columns, and dV += P^T dO,
//    dK += dS^T Q accumulate in TMEM (A from TMEM, B = the row tile in
//    shared memory).
// Row and key tiles that no (row, key) pair of which is visible are skipped;
// tiles every pair of which is visible take no mask.  Products whose B
// operand is a row or key tile read along d (N = d) read it MN-major, the
// two 64-column panels of d = 128 one LBO apart.  Every wait is bounded;
// on expiry a CTA drains its MMAs, frees TMEM and reports H2O_DEVERR_TIMEOUT.
#include <climits>
#include <cmath>

#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kBT = 128;               // rows or keys per tile
constexpr int kBwdSoftmaxWarps = 8;    // two teams of four warps (one per TMEM lane quarter)
constexpr int kBwdFirstSoftmax = 3;    // warp 0 TMA, warps 1 and 2 MMA issue
constexpr int kBwdThreads = 32 * (kBwdFirstSoftmax + kBwdSoftmaxWarps);  // 352
constexpr int kBwdStages = 2;          // shared-memory ring of streamed tile pairs
constexpr int kBwdBufs = 3;            // at most three S / dP buffer pairs in TMEM
constexpr uint8_t kBClsSkip = 0, kBClsFull = 1, kBClsPartial = 2;
constexpr uint16_t kBPartial = 0x8000;  // tile-list entry: masked tile
constexpr uint16_t kBIdxMask = 0x7FFF;
constexpr int kDqStep = 64;            // keys per dq step (two steps per key tile)

template <int D>
struct BwdGeom {
  static constexpr int kPanels = D / 64;
  static constexpr int kTileBytes = kPanels * kBT * 128;  // 128 rows of D bf16
  // dkv: stacked rows per step (the N of S^T and dP^T: an MMA costs at
  // least ~45 cycles, so N = 32 would run the tensor pipe at a third of its
  // rate) and S^T / dP^T buffers; TMEM holds dV and dK (D columns each)
  // and the buffers (2 W columns each): 2D + 2W bufs <= 512.
  static constexpr int kW = 64;
  static constexpr int kStepsPerTile = kBT / kW;
  static constexpr int kDkvBufs = D == 128 ? 2 : 3;
};

// Shared memory of both kernels: two resident tiles (dq: Q and dO; dkv: K and
// V), a ring of kBwdStages pairs of streamed tiles (dq: K_j, V_j; dkv: Q_i,
// dO_i), per stage the streamed rows' lambda and D (dkv), the tile list.
template <int D>
struct __align__(1024) BwdSmem {
  uint8_t res[2][BwdGeom<D>::kTileBytes];
  uint8_t ring[kBwdStages][2][BwdGeom<D>::kTileBytes];
  float rowv[kBwdStages][2][kBT];  // dkv: lambda and D of the stage's rows
  uint64_t bar_res, bar_full[kBwdStages], bar_empty[kBwdStages];
  uint64_t bar_sfull[kBwdBufs], bar_pfull[kBwdBufs], bar_done[kBwdBufs];
  uint64_t bar_acc, bar_drain[2];
  uint32_t taddr;
  int abort_flag;
  int n_tiles;
  uint16_t tiles[kMaxKeyTiles];  // kBPartial | tile index
  uint8_t cls[kMaxKeyTiles];
};

__device__ __forceinline__ bool bwait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return wait_bar(bar, parity, abort, kWaitLimitNs);
}

// Stacked row r of a group -> (head within the group, chunk row i).
__device__ __forceinline__ void split_row(int r, int S, int& g, int& i) {
  g = r / S;
  i = r - g * S;
}

// From a saved forward lse (natural log) and the output: lambda (log2 units)
// and D = dout . out (fp32) of every stacked row, one warp per row; row r of
// group grp (memory row grp R + r) goes to index grp R_pad + r.
template <int D>
__global__ void __launch_bounds__(256) bwd_rows_kernel(const uint16_t* __restrict__ out,
                                                      const uint16_t* __restrict__ dout,
                                                      const float* __restrict__ lse_saved,
                                                      float* __restrict__ lam, float* __restrict__ drow,
                                                      int rows, int R, int R_pad) {
  const int r = blockIdx.x * 8 + static_cast<int>(threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (r >= rows) return;
  constexpr int kPer = D / 32;  // elements per lane: 4 or 2
  float s = 0.f;
  if constexpr (kPer == 4) {
    const uint2 o = reinterpret_cast<const uint2*>(out + static_cast<size_t>(r) * D)[lane];
    const uint2 g = reinterpret_cast<const uint2*>(dout + static_cast<size_t>(r) * D)[lane];
    const uint32_t ow[2] = {o.x, o.y}, gw[2] = {g.x, g.y};
#pragma unroll
    for (int x = 0; x < 2; ++x) {
      s = fmaf(__uint_as_float(ow[x] << 16), __uint_as_float(gw[x] << 16), s);
      s = fmaf(__uint_as_float(ow[x] & 0xFFFF0000u), __uint_as_float(gw[x] & 0xFFFF0000u), s);
    }
  } else {
    const uint32_t o = reinterpret_cast<const uint32_t*>(out + static_cast<size_t>(r) * D)[lane];
    const uint32_t g = reinterpret_cast<const uint32_t*>(dout + static_cast<size_t>(r) * D)[lane];
    s = fmaf(__uint_as_float(o << 16), __uint_as_float(g << 16), s);
    s = fmaf(__uint_as_float(o & 0xFFFF0000u), __uint_as_float(g & 0xFFFF0000u), s);
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
  if (lane == 0) {
    const size_t i = static_cast<size_t>(r / R) * R_pad + r % R;
    drow[i] = s;
    lam[i] = lse_saved[r] * 1.4426950408889634f;
  }
}

// K-major 128-byte-swizzled operand descriptors of a 128-row tile (kPanels
// panels of 64 columns): the eight K-steps of 16 elements along D.
template <int D>
__device__ __forceinline__ void kmajor_steps(uint32_t base, uint64_t (&d)[D / 16]) {
  const uint64_t d0 = sdesc_sw128(base, 16, 1024);
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk)
    d[kk] = d0 + static_cast<uint64_t>((kBT * 128 >> 4) * (kk / 4) + 2 * (kk % 4));
}

// Warp-uniform bounded wait: every lane waits, and the warp goes on only if
// all of them saw the phase complete (so that the .sync.aligned TMEM
// instructions after it are reached by the whole warp or by none of it).
__device__ __forceinline__ bool wwait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  const bool r = bwait(bar, parity, abort);
  return __all_sync(0xffffffffu, r) != 0;
}

// Smallest and largest chunk row i among the valid stacked rows r0 .. r0+127
// of a group (R = q_g S rows, row r = head r / S, chunk row r % S); a tile that
// crosses a head boundary holds both i = S - 1 and i = 0.
__device__ __forceinline__ void row_tile_range(int r0, int R, int S, int& i_min, int& i_max) {
  const int r1 = min(r0 + kBT, R) - 1;
  const int g0 = r0 / S, g1 = r1 / S;
  if (g0 == g1) {
    i_min = r0 - g0 * S;
    i_max = r1 - g0 * S;
  } else {
    i_min = 0;
    i_max = S - 1;
  }
}

// Compacts the classes in sm.cls[0 .. total) into the ordered list of tiles
// to visit (one warp).
template <int D>
__device__ __forceinline__ void build_tile_list(BwdSmem<D>& sm, int total, uint32_t lane) {
  int n = 0;
  for (int base = 0; base < total; base += 32) {
    const int t = base + static_cast<int>(lane);
    const uint8_t cl = t < total ? sm.cls[t] : kBClsSkip;
    const uint32_t m = __ballot_sync(0xffffffffu, cl != kBClsSkip);
    if (cl != kBClsSkip)
      sm.tiles[n + __popc(m & ((1u << lane) - 1u))] =
          static_cast<uint16_t>(t | (cl == kBClsPartial ? kBPartial : 0));
    n += __popc(m);
  }
  if (lane == 0) sm.n_tiles = n;
}

// pfull_count: softmax warps that arrive per step.
template <int D>
__device__ __forceinline__ void init_barriers(BwdSmem<D>& sm, int pfull_count) {
  bar_init(&sm.bar_res, 1);
  for (int s = 0; s < kBwdStages; ++s) {
    bar_init(&sm.bar_full[s], 1);
    bar_init(&sm.bar_empty[s], 1);
  }
  for (int b = 0; b < kBwdBufs; ++b) {
    bar_init(&sm.bar_sfull[b], 1);
    bar_init(&sm.bar_pfull[b], pfull_count);
    bar_init(&sm.bar_done[b], 1);
  }
  bar_init(&sm.bar_acc, 1);
  bar_init(&sm.bar_drain[0], 1);
  bar_init(&sm.bar_drain[1], 1);
  sm.abort_flag = 0;
  fence_bar_init();
}

// After an abort: lets the copies still in flight land before the CTA's
// shared memory goes away (at most the latest load of each stage).
template <int D>
__device__ void drain_loads(BwdSmem<D>& sm, const int (&uses)[kBwdStages], bool res_issued) {
  volatile int never = 0;
  if (res_issued) wait_bar(&sm.bar_res, 0, &never, 100000000ull);
  for (int s = 0; s < kBwdStages; ++s)
    if (uses[s] > 0) wait_bar(&sm.bar_full[s], (uses[s] - 1) & 1, &never, 100000000ull);
}

// Issuer epilogue: no MMA of this issuing thread may still be running when
// TMEM is freed.
template <int D>
__device__ __forceinline__ void drain_mmas(BwdSmem<D>& sm, int issuer) {
  mma_commit(&sm.bar_drain[issuer]);
  volatile int never = 0;
  wait_bar(&sm.bar_drain[issuer], 0, &never, kWaitLimitNs);
}

// ------------------------------------------------------------------ dq ------
// One CTA per 128 stacked rows r0 .. r0+127 of a group.  The key
// tiles (cache tiles, then chunk tiles) run as steps of 64 keys, step n in
// TMEM buffer n % 3: S at columns 128 + 128 b, dP 64 columns after it; the
// softmax writes bf16 dS over S's first 32 columns, dQ (D columns from 0)
// accumulates dS K.  One thread issues S and dP up to three steps ahead,
// another the dQ of each step once its dS is in, so the tensor pipe has
// work while the softmax runs; a buffer is refilled only after the dQ that
// read it has completed (MMAs into different accumulators are not ordered
// by issue).
template <int D>
__device__ __forceinline__ void bwd_dq(const BackwardArgs& a, BwdSmem<D>& sm, int rt, int grp) {
  using G = BwdGeom<D>;
  constexpr int P = G::kPanels;
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const uint32_t lane = tid & 31;
  const int R = a.qg * a.S;
  const int r0 = rt * kBT;
  const int n_ct = (a.M + kBT - 1) / kBT;
  const int n_nt = (a.S + kBT - 1) / kBT;
  int i_min, i_max;
  row_tile_range(r0, R, a.S, i_min, i_max);

  if (tid == 0) init_barriers(sm, kBwdSoftmaxWarps / 2);  // one team per step
  if (warp == 1) {
    tmem_alloc(&sm.taddr, 512);
    tmem_relinquish();
  }
  // key tiles against this CTA's rows: skipped when no row sees a key of
  // it, unmasked when every row sees every key (rows past R have lambda =
  // +inf, so their weights are 0 either way)
  if (warp >= kBwdFirstSoftmax) {
    const int sw = warp - kBwdFirstSoftmax;
    const int* sp = a.slot_pos + static_cast<size_t>(grp) * a.M;
    for (int ct = sw; ct < n_ct; ct += kBwdSoftmaxWarps) {
      bool any = false, all = true;
#pragma unroll
      for (int x = 0; x < 4; ++x) {
        const int j = ct * kBT + 32 * x + static_cast<int>(lane);
        const int pos = j < a.M ? __ldg(sp + j) : -1;
        any |= pos >= 0 && pos <= a.pos0 + i_max;
        all &= pos >= 0 && pos <= a.pos0 + i_min;
      }
      any = __any_sync(0xffffffffu, any);
      all = __all_sync(0xffffffffu, all);
      if (lane == 0) sm.cls[ct] = any ? (all ? kBClsFull : kBClsPartial) : kBClsSkip;
    }
    for (int c = sw; c < n_nt; c += kBwdSoftmaxWarps) {
      const int c0 = c * kBT;
      const uint8_t cl = c0 > i_max ? kBClsSkip
                         : (c0 + kBT - 1 <= i_min && c0 + kBT <= a.S) ? kBClsFull
                                                                       : kBClsPartial;
      if (lane == 0) sm.cls[n_ct + c] = cl;
    }
  }
  __syncthreads();
  if (warp == kBwdFirstSoftmax) build_tile_list(sm, n_ct + n_nt, lane);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();

  const uint32_t tmem = sm.taddr;
  const uint32_t tdQ = tmem;
  const int n_t = sm.n_tiles;
  const int n_steps = 2 * n_t;
  volatile int* abort_flag = &sm.abort_flag;

  if (warp == 0) {
    // --------------------------------------------------------- TMA producer --
    if (lane == 0 && n_t > 0) {
      tma_prefetch_desc(&a.tm_q);
      tma_prefetch_desc(&a.tm_do);
      tma_prefetch_desc(&a.tm_kn);
      tma_prefetch_desc(&a.tm_vn);
      if (n_ct > 0) {
        tma_prefetch_desc(&a.tm_kc);
        tma_prefetch_desc(&a.tm_vc);
      }
      bar_expect_tx(&sm.bar_res, 2 * G::kTileBytes);
      for (int p = 0; p < P; ++p) {
        tma_load_3d(sm.res[0] + p * kBT * 128, &a.tm_q, &sm.bar_res, 64 * p, r0, grp);
        tma_load_3d(sm.res[1] + p * kBT * 128, &a.tm_do, &sm.bar_res, 64 * p, r0, grp);
      }
      int uses[kBwdStages] = {};
      for (int t = 0; t < n_t; ++t) {
        const int s = t % kBwdStages;
        if (uses[s] > 0 && !bwait(&sm.bar_empty[s], (uses[s] - 1) & 1, abort_flag)) break;
        const int idx = sm.tiles[t] & kBIdxMask;
        const bool chunk = idx >= n_ct;
        const int key0 = (chunk ? idx - n_ct : idx) * kBT;
        const CUtensorMap* mk = chunk ? &a.tm_kn : &a.tm_kc;
        const CUtensorMap* mv = chunk ? &a.tm_vn : &a.tm_vc;
        bar_expect_tx(&sm.bar_full[s], 2 * G::kTileBytes);
        for (int p = 0; p < P; ++p) {
          tma_load_3d(sm.ring[s][0] + p * kBT * 128, mk, &sm.bar_full[s], 64 * p, key0, grp);
          tma_load_3d(sm.ring[s][1] + p * kBT * 128, mv, &sm.bar_full[s], 64 * p, key0, grp);
        }
        ++uses[s];
      }
      if (*abort_flag) drain_loads(sm, uses, true);
    }
  } else if (warp == 1 || warp == 2) {
    // ----------------------------------------------------------- MMA issue --
    // Warp 1 issues S and dP of every step, warp 2 every dQ: while one
    // issuing thread waits on a barrier the other keeps the tensor pipe fed
    // (an issuing thread runs only about one MMA ahead of the pipe).
    if (lane == 0 && n_t > 0) {
      constexpr uint32_t kIdS = idesc_bf16_f32(kBT, kDqStep, false);  // S, dP: N = 64 keys
      constexpr uint32_t kIdQ = idesc_bf16_f32(kBT, D, true);         // dQ: N = D
      // Descriptors: only the 14-bit start address (bytes >> 4) moves: a
      // ring stage is 2 kTileBytes, half h of a key tile starts 64 rows
      // (8 KB) in, a K-step of 16 bf16 is 32 B of a 128-B swizzle row, a
      // 64-column panel is 16 KB; for the MN-major K in dQ a K-step is 16
      // key rows (2 KB) and the panels are LBO apart.  Everything but the
      // stage / half offset is formed once, before the first MMA.
      constexpr uint64_t kStage = (2 * G::kTileBytes) >> 4;
      constexpr uint64_t kHalf = (kDqStep * 128) >> 4;
      uint64_t qd[D / 16], od[D / 16], kd0[D / 16], vd0[D / 16];
      kmajor_steps<D>(smem_addr(sm.res[0]), qd);
      kmajor_steps<D>(smem_addr(sm.res[1]), od);
      kmajor_steps<D>(smem_addr(sm.ring[0][0]), kd0);
      kmajor_steps<D>(smem_addr(sm.ring[0][1]), vd0);
      const uint64_t kmn0 = sdesc_sw128(smem_addr(sm.ring[0][0]), kBT * 128, 1024);
      // S = Q K^T and dP = dO V^T of step m (keys 64 h .. of tile m / 2)
      auto issue_sdp = [&](int m) -> bool {
        const int b = m % kBwdBufs, t = m >> 1, h = m & 1, s = t % kBwdStages;
        if (m >= kBwdBufs && !bwait(&sm.bar_done[b], (m / kBwdBufs - 1) & 1, abort_flag))
          return false;
        if (h == 0 && !bwait(&sm.bar_full[s], (t / kBwdStages) & 1, abort_flag)) return false;
        tc_fence_after_sync();
        const uint64_t off = kStage * s + kHalf * h;
        uint64_t kd[D / 16], vd[D / 16];
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          kd[kk] = kd0[kk] + off;
          vd[kk] = vd0[kk] + off;
        }
        const uint32_t tSb = tmem + 128 + 128 * b;
        if constexpr (D == 128) {
          mma_ss_x8<false>(tSb, qd, kd, kIdS, 0u);
          mma_ss_x8<false>(tSb + kDqStep, od, vd, kIdS, 0u);
        } else {
          mma_ss_x4(tSb, qd, kd, kIdS, 0u);
          mma_ss_x4(tSb + kDqStep, od, vd, kIdS, 0u);
        }
        mma_commit(&sm.bar_sfull[b]);
        return true;
      };
      // dQ += dS K_step (A = dS from TMEM, 4 K-steps of 16 keys; B = the
      // step's 64 key rows, MN-major, N = D)
      auto issue_dq = [&](int n) -> bool {
        const int b = n % kBwdBufs, t = n >> 1, h = n & 1, s = t % kBwdStages;
        if (!bwait(&sm.bar_pfull[b], (n / kBwdBufs) & 1, abort_flag)) return false;
        tc_fence_after_sync();
        const uint64_t kb = kmn0 + kStage * s + 128 * 4 * h;
        const uint64_t bd[4] = {kb, kb + 128, kb + 256, kb + 384};
        const uint32_t tSb = tmem + 128 + 128 * b;
        mma_ts_x4(tdQ, tSb, tSb + 16, bd, kIdQ, n > 0 ? 1u : 0u);
        mma_commit(&sm.bar_done[b]);
        if (h == 1) mma_commit(&sm.bar_empty[s]);  // both halves of K_t, V_t read
        return true;
      };
      bool ok = true;
      if (warp == 1) {
        ok = bwait(&sm.bar_res, 0, abort_flag);
        for (int m = 0; ok && m < n_steps; ++m) ok = issue_sdp(m);
      } else {
        for (int n = 0; ok && n < n_steps; ++n) ok = issue_dq(n);
        if (ok) mma_commit(&sm.bar_acc);
      }
      drain_mmas(sm, warp - 1);
    }
  } else {
    // ---------------------------------------------------- dS = P (dP - D) --
    // Team t (warps 3-6 or 7-10) takes steps n = t, t + 2, ...; each thread
    // owns one stacked row (the 32x32b layout: lane quarter warp % 4).
    const int sw = warp - kBwdFirstSoftmax;
    const int team = sw >> 2;
    const int q4 = warp & 3;
    const int row = q4 * 32 + static_cast<int>(lane);
    const int r = r0 + row;
    const bool valid = r < R;
    int g = 0, i = 0;
    if (valid) split_row(r, a.S, g, i);
    const size_t ri = static_cast<size_t>(grp) * backward_row_stride(a.qg, a.S) + r;
    const float nlam = valid ? -__ldg(a.lse + ri) : -INFINITY;
    const float drow = valid ? __ldg(a.drow + ri) : 0.f;
    const float sl2 = a.scale_log2;
    const int qpos = a.pos0 + i;
    const int* sp = a.slot_pos + static_cast<size_t>(grp) * a.M;
    const uint32_t lane_addr = static_cast<uint32_t>(q4 * 32) << 16;
    bool ok = true;
    for (int n = team; n < n_steps; n += 2) {
      const int b = n % kBwdBufs, t = n >> 1, h = n & 1;
      if (!wwait(&sm.bar_sfull[b], (n / kBwdBufs) & 1, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const uint16_t e = sm.tiles[t];
      const int idx = e & kBIdxMask;
      const bool partial = (e & kBPartial) != 0;
      const bool chunk = idx >= n_ct;
      const int key0 = (chunk ? idx - n_ct : idx) * kBT + h * kDqStep;
      const uint32_t tSb = tmem + 128 + 128 * b + lane_addr;
#pragma unroll 1
      for (int hh = 0; hh < 2; ++hh) {
        uint32_t sr[32], pr[32];
        tmem_ld32_async(tSb + 32 * hh, sr);
        tmem_ld32_async(tSb + kDqStep + 32 * hh, pr);
        uint32_t vis = 0xffffffffu;  // bit k: key key0 + 32 hh + k visible to this row
        if (partial) {
          vis = 0u;
          const int j0 = key0 + 32 * hh;
          if (valid) {
            if (chunk) {
#pragma unroll
              for (int k = 0; k < 32; ++k)
                if (j0 + k <= i && j0 + k < a.S) vis |= 1u << k;
            } else {
              for (int k = 0; k < 32; ++k) {
                const int j = j0 + k;
                const int pos = j < a.M ? __ldg(sp + j) : -1;
                if (pos >= 0 && pos <= qpos) vis |= 1u << k;
              }
            }
          }
        }
        tmem_wait_ld(sr);
        tmem_wait_ld(pr);
        uint32_t ds[16];
        const float2 sc = make_float2(sl2, sl2), nl = make_float2(nlam, nlam);
        const float2 nd = make_float2(-drow, -drow);
#pragma unroll
        for (int k = 0; k < 32; k += 2) {
          const float2 x = ffma2(make_float2(__uint_as_float(sr[k]), __uint_as_float(sr[k + 1])), sc, nl);
          const float2 p = make_float2(fast_exp2(x.x), fast_exp2(x.y));
          const float2 dp = fadd2(make_float2(__uint_as_float(pr[k]), __uint_as_float(pr[k + 1])), nd);
          float d0 = p.x * dp.x, d1 = p.y * dp.y;
          if (partial) {
            d0 = (vis >> k) & 1u ? d0 : 0.f;
            d1 = (vis >> (k + 1)) & 1u ? d1 : 0.f;
          }
          ds[k / 2] = pack_bf16x2(d0, d1);
        }
        // keys 32 hh .. 32 hh + 31 as bf16 pairs over columns 16 hh .. of S
        // (columns this thread has already loaded)
        tmem_st16_async(tSb + 16 * hh, ds);
      }
      tmem_wait_st();
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) bar_arrive(&sm.bar_pfull[b]);
    }
    // ------------------------------------------------------------ epilogue --
    // dq = scale dQ: team t stores columns t D / 2 .. of its rows
    if (ok && n_steps > 0) ok = wwait(&sm.bar_acc, 0, abort_flag);
    if (ok) {
      tc_fence_after_sync();
      float* dst = a.dq + (static_cast<size_t>(grp) * R + r) * D + team * (D / 2);
#pragma unroll 1
      for (int c = 0; c < D / 2; c += 32) {
        uint32_t v[32];
        if (n_steps > 0) {
          tmem_ld32(tdQ + lane_addr + team * (D / 2) + c, v);
        } else {
#pragma unroll
          for (int k = 0; k < 32; ++k) v[k] = 0u;
        }
        if (valid) {
          float4* d4 = reinterpret_cast<float4*>(dst + c);
#pragma unroll
          for (int k = 0; k < 8; ++k)
            d4[k] = make_float4(a.scale * __uint_as_float(v[4 * k]), a.scale * __uint_as_float(v[4 * k + 1]),
                                a.scale * __uint_as_float(v[4 * k + 2]), a.scale * __uint_as_float(v[4 * k + 3]));
        }
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, 512);
  }
}

// ----------------------------------------------------------------- dkv ------
// One CTA per key tile kt of a group (cache tiles, then chunk tiles), K and V
// resident.  The row tiles of the group's stacked rows stream through the
// ring with their lambda and D and run as steps of W = 64 rows, step n in
// TMEM buffer n % NB (two buffers for d = 128, three for d = 64): S^T at
// columns 2D + 2W b, dP^T W columns after it; the softmax writes bf16 P^T
// over S^T's first W/2 columns and dS^T over dP^T's, dV (columns 0 ..)
// accumulates P^T dO and dK (columns D ..) dS^T Q.  The two issuing
// threads work as in the dq kernel.
template <int D>
__device__ __forceinline__ void bwd_dkv(const BackwardArgs& a, BwdSmem<D>& sm, int kt, int grp) {
  using G = BwdGeom<D>;
  constexpr int P = G::kPanels;
  constexpr int W = G::kW;
  constexpr int SPT = G::kStepsPerTile;
  constexpr int NB = G::kDkvBufs;
  static_assert(W == 64, "each softmax team takes 32 rows of a step");
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const uint32_t lane = tid & 31;
  const int R = a.qg * a.S;
  const int Rp = backward_row_stride(a.qg, a.S);
  const int n_ct = (a.M + kBT - 1) / kBT;
  const bool chunk = kt >= n_ct;
  const int key0 = (chunk ? kt - n_ct : kt) * kBT;
  const int n_keys = min(kBT, (chunk ? a.S : a.M) - key0);
  const int n_rt = (R + kBT - 1) / kBT;
  const int* sp = a.slot_pos + static_cast<size_t>(grp) * a.M;
  // key j of the tile is seen by chunk row i iff thr(j) <= i (cache slot:
  // occupied and pos - pos0 <= i; chunk token c: c <= i); keys that do not
  // exist or are empty never are
  auto key_thr = [&](int kl) -> int {
    const int j = key0 + kl;
    if (chunk) return kl < n_keys ? j : INT_MAX;
    const int pos = kl < n_keys ? __ldg(sp + j) : -1;
    return pos >= 0 ? pos - a.pos0 : INT_MAX;
  };

  if (tid == 0) init_barriers(sm, kBwdSoftmaxWarps);  // both teams on every step
  if (warp == 1) {
    tmem_alloc(&sm.taddr, 512);
    tmem_relinquish();
  }
  if (warp == kBwdFirstSoftmax) {
    // row tiles against this key tile: skipped when no row sees a key,
    // unmasked when every row exists and sees every key
    int tmin = INT_MAX, tmax = INT_MIN;
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      const int th = key_thr(32 * x + static_cast<int>(lane));
      tmin = min(tmin, th);
      tmax = max(tmax, th);
    }
    tmin = __reduce_min_sync(0xffffffffu, tmin);
    tmax = __reduce_max_sync(0xffffffffu, tmax);  // INT_MAX when a key is never seen
    for (int rt = static_cast<int>(lane); rt < n_rt; rt += 32) {
      int i_min, i_max;
      row_tile_range(rt * kBT, R, a.S, i_min, i_max);
      const bool all_rows = rt * kBT + kBT <= R;
      sm.cls[rt] = tmin > i_max                              ? kBClsSkip
                   : (all_rows && tmax != INT_MAX && tmax <= i_min) ? kBClsFull
                                                              : kBClsPartial;
    }
    __syncwarp();
    build_tile_list(sm, n_rt, lane);
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();

  const uint32_t tmem = sm.taddr;
  const uint32_t tdV = tmem, tdK = tmem + D;
  const int n_t = sm.n_tiles;
  const int n_steps = n_t * SPT;
  volatile int* abort_flag = &sm.abort_flag;

  if (warp == 0) {
    // --------------------------------------------------------- TMA producer --
    if (lane == 0 && n_t > 0) {
      const CUtensorMap* mk = chunk ? &a.tm_kn : &a.tm_kc;
      const CUtensorMap* mv = chunk ? &a.tm_vn : &a.tm_vc;
      tma_prefetch_desc(mk);
      tma_prefetch_desc(mv);
      tma_prefetch_desc(&a.tm_q);
      tma_prefetch_desc(&a.tm_do);
      bar_expect_tx(&sm.bar_res, 2 * G::kTileBytes);
      for (int p = 0; p < P; ++p) {
        tma_load_3d(sm.res[0] + p * kBT * 128, mk, &sm.bar_res, 64 * p, key0, grp);
        tma_load_3d(sm.res[1] + p * kBT * 128, mv, &sm.bar_res, 64 * p, key0, grp);
      }
      int uses[kBwdStages] = {};
      for (int t = 0; t < n_t; ++t) {
        const int s = t % kBwdStages;
        if (uses[s] > 0 && !bwait(&sm.bar_empty[s], (uses[s] - 1) & 1, abort_flag)) break;
        const int row0 = (sm.tiles[t] & kBIdxMask) * kBT;
        const size_t ro = static_cast<size_t>(grp) * Rp + row0;
        bar_expect_tx(&sm.bar_full[s], 2 * G::kTileBytes + 2 * kBT * 4);
        for (int p = 0; p < P; ++p) {
          tma_load_3d(sm.ring[s][0] + p * kBT * 128, &a.tm_q, &sm.bar_full[s], 64 * p, row0, grp);
          tma_load_3d(sm.ring[s][1] + p * kBT * 128, &a.tm_do, &sm.bar_full[s], 64 * p, row0, grp);
        }
        bulk_load_once(sm.rowv[s][0], a.lse + ro, kBT * 4, &sm.bar_full[s]);
        bulk_load_once(sm.rowv[s][1], a.drow + ro, kBT * 4, &sm.bar_full[s]);
        ++uses[s];
      }
      if (*abort_flag) drain_loads(sm, uses, true);
    }
  } else if (warp == 1 || warp == 2) {
    // ----------------------------------------------------------- MMA issue --
    // warp 1: S^T and dP^T of every step; warp 2: dV and dK
    if (lane == 0 && n_t > 0) {
      constexpr uint32_t kIdS = idesc_bf16_f32(kBT, W, false);  // S^T, dP^T: N = W rows
      constexpr uint32_t kIdG = idesc_bf16_f32(kBT, D, true);   // dV, dK: N = D
      // descriptors as in the dq kernel; step w of a row tile starts W rows
      // (W * 128 B) into it
      constexpr uint64_t kStage = (2 * G::kTileBytes) >> 4;
      constexpr uint64_t kRows = (W * 128) >> 4;
      uint64_t kd[D / 16], vd[D / 16], qd0[D / 16], od0[D / 16];
      kmajor_steps<D>(smem_addr(sm.res[0]), kd);
      kmajor_steps<D>(smem_addr(sm.res[1]), vd);
      kmajor_steps<D>(smem_addr(sm.ring[0][0]), qd0);
      kmajor_steps<D>(smem_addr(sm.ring[0][1]), od0);
      const uint64_t qmn0 = sdesc_sw128(smem_addr(sm.ring[0][0]), kBT * 128, 1024);
      const uint64_t omn0 = sdesc_sw128(smem_addr(sm.ring[0][1]), kBT * 128, 1024);
      // S^T = K Q_w^T and dP^T = V dO_w^T of step m (rows W w .. of row tile m / SPT)
      auto issue_sdp = [&](int m) -> bool {
        const int b = m % NB, t = m / SPT, w = m % SPT, s = t % kBwdStages;
        if (m >= NB && !bwait(&sm.bar_done[b], (m / NB - 1) & 1, abort_flag))
          return false;
        if (w == 0 && !bwait(&sm.bar_full[s], (t / kBwdStages) & 1, abort_flag)) return false;
        tc_fence_after_sync();
        const uint64_t off = kStage * s + kRows * w;
        uint64_t qd[D / 16], od[D / 16];
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          qd[kk] = qd0[kk] + off;
          od[kk] = od0[kk] + off;
        }
        const uint32_t tSb = tmem + 2 * D + 2 * W * b;
        if constexpr (D == 128) {
          mma_ss_x8<false>(tSb, kd, qd, kIdS, 0u);
          mma_ss_x8<false>(tSb + W, vd, od, kIdS, 0u);
        } else {
          mma_ss_x4(tSb, kd, qd, kIdS, 0u);
          mma_ss_x4(tSb + W, vd, od, kIdS, 0u);
        }
        mma_commit(&sm.bar_sfull[b]);
        return true;
      };
      // dV += P^T dO_w, dK += dS^T Q_w (A from TMEM, W / 16 K-steps of 16
      // rows; B = the step's rows, MN-major, N = D)
      auto issue_kv = [&](int n) -> bool {
        const int b = n % NB, t = n / SPT, w = n % SPT, s = t % kBwdStages;
        if (!bwait(&sm.bar_pfull[b], (n / NB) & 1, abort_flag)) return false;
        tc_fence_after_sync();
        const uint32_t tSb = tmem + 2 * D + 2 * W * b;
        const uint64_t off = kStage * s + 128 * (W / 16) * w;
        const uint32_t acc = n > 0 ? 1u : 0u;
        // rows 0-31 of the step (K-steps 0, 1) as bf16 pairs at columns 0-15
        // of the buffer half, rows 32-63 (K-steps 2, 3) at columns 32-47
        const uint64_t bo[4] = {omn0 + off, omn0 + off + 128, omn0 + off + 256, omn0 + off + 384};
        const uint64_t bq[4] = {qmn0 + off, qmn0 + off + 128, qmn0 + off + 256, qmn0 + off + 384};
        mma_ts_x4(tdV, tSb, tSb + 32, bo, kIdG, acc);
        mma_ts_x4(tdK, tSb + W, tSb + W + 32, bq, kIdG, acc);
        mma_commit(&sm.bar_done[b]);
        if (w == SPT - 1) mma_commit(&sm.bar_empty[s]);  // the row tile's last step
        return true;
      };
      bool ok = true;
      if (warp == 1) {
        ok = bwait(&sm.bar_res, 0, abort_flag);
        for (int m = 0; ok && m < n_steps; ++m) ok = issue_sdp(m);
      } else {
        for (int n = 0; ok && n < n_steps; ++n) ok = issue_kv(n);
        if (ok) mma_commit(&sm.bar_acc);
      }
      drain_mmas(sm, warp - 1);
    }
  } else {
    // ------------------------------------ P^T and dS^T = P^T (dP^T - D) --
    // Both teams work on every step, team t on its rows 32 t .. 32 t + 31
    // (with two buffers at d = 128 the steps cannot overlap, so the step's
    // softmax latency is what matters); each thread owns one key (the 32x32b
    // layout: lane quarter warp % 4), the columns are stacked rows.
    const int sw = warp - kBwdFirstSoftmax;
    const int team = sw >> 2;
    const int q4 = warp & 3;
    const int kl = q4 * 32 + static_cast<int>(lane);
    const int thr = key_thr(kl);
    const float sl2 = a.scale_log2;
    const float2 sc = make_float2(sl2, sl2);
    const uint32_t lane_addr = static_cast<uint32_t>(q4 * 32) << 16;
    bool ok = true;
    for (int n = 0; n < n_steps; ++n) {
      const int b = n % NB, t = n / SPT, w = n % SPT, s = t % kBwdStages;
      // the S^T buffer, and the stage's lambda and D (complete with its tiles)
      if (!wwait(&sm.bar_sfull[b], (n / NB) & 1, abort_flag) ||
          !wwait(&sm.bar_full[s], (t / kBwdStages) & 1, abort_flag)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      const uint16_t e = sm.tiles[t];
      const bool partial = (e & kBPartial) != 0;
      const int rs0 = (e & kBIdxMask) * kBT + w * W;  // first stacked row of the step
      const uint32_t tSb = tmem + 2 * D + 2 * W * b + lane_addr;
      {
        const int hh = team;
        uint32_t sr[32], pr[32];
        tmem_ld32_async(tSb + 32 * hh, sr);
        tmem_ld32_async(tSb + W + 32 * hh, pr);
        uint32_t vis = 0xffffffffu;  // bit k: row rs0 + 32 hh + k sees this key
        if (partial) {
          vis = 0u;
          const int rr = rs0 + 32 * hh;
          int i = rr % a.S;
#pragma unroll
          for (int k = 0; k < 32; ++k) {
            if (rr + k < R && thr <= i) vis |= 1u << k;
            i = i + 1 == a.S ? 0 : i + 1;
          }
        }
        tmem_wait_ld(sr);
        tmem_wait_ld(pr);
        const float* lam = sm.rowv[s][0] + w * W + 32 * hh;
        const float* dr = sm.rowv[s][1] + w * W + 32 * hh;
        uint32_t pk[16], dk[16];
#pragma unroll
        for (int k = 0; k < 32; k += 4) {
          const float4 l4 = *reinterpret_cast<const float4*>(lam + k);
          const float4 d4 = *reinterpret_cast<const float4*>(dr + k);
#pragma unroll
          for (int x = 0; x < 4; x += 2) {
            const float l0 = x == 0 ? l4.x : l4.z, l1 = x == 0 ? l4.y : l4.w;
            const float e0 = x == 0 ? d4.x : d4.z, e1 = x == 0 ? d4.y : d4.w;
            const float2 z = ffma2(make_float2(__uint_as_float(sr[k + x]), __uint_as_float(sr[k + x + 1])),
                                   sc, make_float2(-l0, -l1));
            float p0 = fast_exp2(z.x), p1 = fast_exp2(z.y);
            const float2 dd = fadd2(make_float2(__uint_as_float(pr[k + x]), __uint_as_float(pr[k + x + 1])),
                                    make_float2(-e0, -e1));
            float g0 = p0 * dd.x, g1 = p1 * dd.y;
            if (partial) {
              const bool v0 = (vis >> (k + x)) & 1u, v1 = (vis >> (k + x + 1)) & 1u;
              p0 = v0 ? p0 : 0.f;
              p1 = v1 ? p1 : 0.f;
              g0 = v0 ? g0 : 0.f;
              g1 = v1 ? g1 : 0.f;
            }
            pk[(k + x) / 2] = pack_bf16x2(p0, p1);
            dk[(k + x) / 2] = pack_bf16x2(g0, g1);
          }
        }
        // rows 32 hh .. 32 hh + 31 of the step as bf16 pairs over the first
        // 16 of the columns this thread has just loaded, in S^T and in dP^T
        tmem_st16_async(tSb + 32 * hh, pk);
        tmem_st16_async(tSb + W + 32 * hh, dk);
      }
      tmem_wait_st();
      tc_fence_before_sync();
      __syncwarp();
      if (lane == 0) bar_arrive(&sm.bar_pfull[b]);
    }
    // ------------------------------------------------------------ epilogue --
    // team 0 stores dv = dV, team 1 dk = scale dK, one key row per thread
    if (ok && n_steps > 0) ok = wwait(&sm.bar_acc, 0, abort_flag);
    if (ok) {
      tc_fence_after_sync();
      float* base = team == 0 ? (chunk ? a.dv_new : a.dv_cache) : (chunk ? a.dk_new : a.dk_cache);
      const float f = team == 0 ? 1.f : a.scale;
      const int rows = chunk ? a.S : a.M;
      float* dst = base + (static_cast<size_t>(grp) * rows + key0 + kl) * D;
#pragma unroll 1
      for (int c = 0; c < D; c += 32) {
        uint32_t v[32];
        if (n_steps > 0) {
          tmem_ld32((team == 0 ? tdV : tdK) + lane_addr + c, v);
        } else {
#pragma unroll
          for (int k = 0; k < 32; ++k) v[k] = 0u;
        }
        if (kl < n_keys) {
          float4* d4 = reinterpret_cast<float4*>(dst + c);
#pragma unroll
          for (int k = 0; k < 8; ++k)
            d4[k] = make_float4(f * __uint_as_float(v[4 * k]), f * __uint_as_float(v[4 * k + 1]),
                                f * __uint_as_float(v[4 * k + 2]), f * __uint_as_float(v[4 * k + 3]));
        }
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, 512);
  }
}

// One launch for both halves of the gradient, a 1-D grid: the first
// n_row_tiles x groups CTAs form dq (row tile, group), the rest dk / dv (key
// tile, group), key-tile major.  The dq CTAs, the longest, are dispatched
// first; the dk / dv CTAs fill the SMs around them and after them, the
// cache tiles (every row sees them) before the chunk tiles (causal, fewer
// rows the later the tile).
template <int D>
__global__ void __launch_bounds__(kBwdThreads, 1) bwd_kernel(const __grid_constant__ BackwardArgs a,
                                                            int n_row_tiles, int n_key_tiles) {
  extern __shared__ uint8_t smem_raw[];
  auto& sm = *reinterpret_cast<BwdSmem<D>*>(smem_raw +
                                            ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u));
  const int x = static_cast<int>(blockIdx.x);
  const int n_dq = n_row_tiles * a.B * a.Hkv;
  if (x < n_dq) {
    bwd_dq<D>(a, sm, x % n_row_tiles, x / n_row_tiles);
  } else {
    const int y = x - n_dq;
    const int groups = a.B * a.Hkv;
    bwd_dkv<D>(a, sm, y / groups, y % groups);
  }
  if (threadIdx.x == 0 && sm.abort_flag) atomicOr(a.err, H2O_DEVERR_TIMEOUT);
}

template <int D>
cudaError_t launch_backward_d(const BackwardArgs& a, cudaStream_t stream) {
  const int R = a.qg * a.S;
  const size_t smem = sizeof(BwdSmem<D>) + 1024;
  static OncePerDevice configured;
  const cudaError_t e = configured.run([smem](int) {
    return cudaFuncSetAttribute(bwd_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(smem));
  });
  if (e != cudaSuccess) return e;
  const int n_row_tiles = (R + kBT - 1) / kBT;
  const int n_key_tiles = (a.M + kBT - 1) / kBT + (a.S + kBT - 1) / kBT;
  const int64_t ctas = static_cast<int64_t>(n_row_tiles + n_key_tiles) * a.B * a.Hkv;
  bwd_kernel<D><<<static_cast<unsigned>(ctas), kBwdThreads, smem, stream>>>(a, n_row_tiles,
                                                                            n_key_tiles);
  return cudaGetLastError();
}

}  // namespace

size_t backward_workspace_bytes(int B, int Hq, int Hkv, int S, int M) {
  (void)M;
  const int qg = Hkv > 0 ? Hq / Hkv : 0;
  // lambda and D per stacked row, each group's rows padded to 128
  return 2 * static_cast<size_t>(B) * Hkv * backward_row_stride(qg, S) * sizeof(float);
}

cudaError_t launch_backward_rows(const BackwardArgs& a, const uint16_t* out, const uint16_t* dout,
                                 const float* lse_saved, cudaStream_t stream) {
  const int rows = a.B * a.Hq * a.S;
  const int R = a.qg * a.S;
  const unsigned grid = static_cast<unsigned>((rows + 7) / 8);
  const int Rp = backward_row_stride(a.qg, a.S);
  if (a.d == 64)
    bwd_rows_kernel<64><<<grid, 256, 0, stream>>>(out, dout, lse_saved, a.lse, a.drow, rows, R, Rp);
  else
    bwd_rows_kernel<128><<<grid, 256, 0, stream>>>(out, dout, lse_saved, a.lse, a.drow, rows, R, Rp);
  return cudaGetLastError();
}

cudaError_t launch_backward(const BackwardArgs& a, cudaStream_t stream) {
  return a.d == 64 ? launch_backward_d<64>(a, stream) : launch_backward_d<128>(a, stream);
}

}  // namespace h2o
