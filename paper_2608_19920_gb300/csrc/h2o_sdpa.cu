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
//  * Warp roles: warp 0 issues TMA loads (Q once, then K and V tiles through a
//    2-stage ring), warp 1 issues tcgen05 MMAs (accumulators in TMEM: two S
//    buffers and the O accumulator), warps 4-11 are two softmax warpgroups;
//    warpgroup w owns key columns 64w..64w+63 of every S tile and TMEM lanes =
//    query rows.  P is written back to TMEM as bf16 over its own S columns and
//    consumed by the P V MMA directly from TMEM.
//  * Column sums use the fp32 P (not the bf16 copy fed to the MMA): a warp
//    reduce-scatter leaves two column sums per lane, the four warps of a
//    warpgroup combine through shared memory, and one red.global.add per
//    column and query head goes to score_inc (zeroed by the host call).
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

constexpr int kStages = 2;
constexpr int kThreads = 384;
constexpr uint16_t kTileChunk = 0x8000;
constexpr uint16_t kTilePartial = 0x4000;
constexpr uint16_t kTileIdxMask = 0x3FFF;
constexpr uint8_t kClsSkip = 0, kClsFull = 1, kClsPartial = 2;

template <int D>
struct __align__(1024) SdpaSmem {
  static constexpr int kPanels = D / 64;
  uint8_t q[kPanels][kTileM * 128];
  uint8_t k[kStages][kPanels][kTileN * 128];
  uint8_t v[kStages][kPanels][kTileN * 128];
  float colsum[2][2][4][64];  // [buffer][warpgroup][warp][column]
  float rowstat[2][kTileM][2];
  uint64_t bar_q;
  uint64_t bar_kfull[kStages], bar_kempty[kStages];
  uint64_t bar_vfull[kStages], bar_vempty[kStages];
  uint64_t bar_sfull[2], bar_pfull[2], bar_pvdone[2];
  uint64_t bar_cs[2][2];
  uint64_t bar_rowstat, bar_ofull, bar_drain;
  uint32_t taddr;
  int abort_flag;
  int n_tiles;
  uint8_t cls[kMaxKeyTiles];
  uint16_t tiles[kMaxKeyTiles];
};

// Butterfly reduce-scatter of 64 values over the 32 lanes of a warp: on
// return v[0], v[1] hold the warp-wide sums of columns 2*lane, 2*lane+1.
template <int L, int O>
__device__ __forceinline__ void rs_step(float (&v)[64], uint32_t lane) {
  const bool up = (lane & O) != 0;
#pragma unroll
  for (int k = 0; k < L / 2; ++k) {
    const float send = up ? v[k] : v[k + L / 2];
    const float keep = up ? v[k + L / 2] : v[k];
    v[k] = keep + __shfl_xor_sync(0xffffffffu, send, O);
  }
}

__device__ __forceinline__ void reduce_scatter64(float (&v)[64], uint32_t lane) {
  rs_step<64, 16>(v, lane);
  rs_step<32, 8>(v, lane);
  rs_step<16, 4>(v, lane);
  rs_step<8, 2>(v, lane);
  rs_step<4, 1>(v, lane);
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
    for (int s = 0; s < kStages; ++s) {
      bar_init(&sm.bar_kfull[s], 1);
      bar_init(&sm.bar_kempty[s], 1);
      bar_init(&sm.bar_vfull[s], 1);
      bar_init(&sm.bar_vempty[s], 1);
    }
    for (int x = 0; x < 2; ++x) {
      bar_init(&sm.bar_sfull[x], 1);
      bar_init(&sm.bar_pfull[x], 8);
      bar_init(&sm.bar_pvdone[x], 1);
      bar_init(&sm.bar_cs[x][0], 4);
      bar_init(&sm.bar_cs[x][1], 4);
    }
    bar_init(&sm.bar_rowstat, 8);
    bar_init(&sm.bar_ofull, 1);
    bar_init(&sm.bar_drain, 1);
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
  if (warp >= 4) {
    const int sw = warp - 4;
    const int* sp = a.slot_pos + static_cast<size_t>(grp) * a.M;
    const int lim_any = a.pos0 + i_hi;
    const int lim_all = a.pos0 + i_lo;
    for (int ct = sw; ct < a.n_cache_tiles; ct += 8) {
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
    for (int c = sw; c < a.n_chunk_tiles; c += 8) {
      const int c0 = c * kTileN;
      uint8_t cl = kClsPartial;
      if (c0 > i_hi) cl = kClsSkip;
      else if (c0 + kTileN - 1 <= i_lo && c0 + kTileN <= a.S) cl = kClsFull;
      if (lane == 0) sm.cls[a.n_cache_tiles + c] = cl;
    }
  }
  __syncthreads();
  if (warp == 4) {
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
  const uint32_t tS = tmem;        // S / P buffers: columns [0,128), [128,256)
  const uint32_t tO = tmem + 256;  // O accumulator: columns [256, 256 + D)
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
      int nk = 0, nv = 0;
      for (int n = 0; n < 2 * n_t; ++n) {
        const bool pass2 = n >= n_t;
        const int t = pass2 ? n - n_t : n;
        const uint16_t e = sm.tiles[t];
        const bool chunk = (e & kTileChunk) != 0;
        const int row0 = (e & kTileIdxMask) * kTileN;
        const CUtensorMap* mk = chunk ? &a.tm_kn : &a.tm_kc;
        const CUtensorMap* mv = chunk ? &a.tm_vn : &a.tm_vc;
        const int s = n % kStages;
        if (n >= kStages &&
            !wait_bar(&sm.bar_kempty[s], ((n / kStages) - 1) & 1, abort_flag, kWaitLimitNs))
          break;
        bar_expect_tx(&sm.bar_kfull[s], P * kTileN * 128);
        for (int p = 0; p < P; ++p) tma_load_3d(sm.k[s][p], mk, &sm.bar_kfull[s], 64 * p, row0, grp);
        ++nk;
        if (pass2) {
          const int vs = t % kStages;
          if (t >= kStages &&
              !wait_bar(&sm.bar_vempty[vs], ((t / kStages) - 1) & 1, abort_flag, kWaitLimitNs))
            break;
          bar_expect_tx(&sm.bar_vfull[vs], P * kTileN * 128);
          for (int p = 0; p < P; ++p) tma_load_3d(sm.v[vs][p], mv, &sm.bar_vfull[vs], 64 * p, row0, grp);
          ++nv;
        }
      }
      if (*abort_flag) {
        // Let copies still in flight land before the CTA's shared memory goes away.
        volatile int never = 0;
        for (int x = max(0, nk - kStages); x < nk; ++x)
          wait_bar(&sm.bar_kfull[x % kStages], (x / kStages) & 1, &never, 100000000ull);
        for (int x = max(0, nv - kStages); x < nv; ++x)
          wait_bar(&sm.bar_vfull[x % kStages], (x / kStages) & 1, &never, 100000000ull);
      }
    }
  } else if (warp == 1) {
    // -------------------------------------------------------- MMA issuer --
    if (lane == 0 && n_t > 0) {
      constexpr uint32_t kIdescQK = idesc_bf16_f32(kTileM, kTileN, false);
      constexpr uint32_t kIdescPV = idesc_bf16_f32(kTileM, D, true);
      bool ok = wait_bar(&sm.bar_q, 0, abort_flag, kWaitLimitNs);
      uint32_t pv_phase[2] = {0u, 0u};
      auto issue_pv = [&](int t) -> bool {
        const int n = n_t + t;
        const int buf = n & 1;
        if (!wait_bar(&sm.bar_pfull[buf], (n >> 1) & 1, abort_flag, kWaitLimitNs)) return false;
        const int vs = t % kStages;
        if (!wait_bar(&sm.bar_vfull[vs], (t / kStages) & 1, abort_flag, kWaitLimitNs)) return false;
        tc_fence_after_sync();
#pragma unroll
        for (int kk = 0; kk < kTileN / 16; ++kk) {
          const uint32_t a_tmem = tS + buf * 128 + 64 * (kk / 4) + 8 * (kk % 4);
          const uint64_t bd = sdesc_sw128(smem_addr(sm.v[vs][0]) + 2048 * kk, kTileN * 128, 1024);
          mma_ts(tO, a_tmem, bd, kIdescPV, (t > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(&sm.bar_vempty[vs]);
        mma_commit(&sm.bar_pvdone[buf]);
        return true;
      };
      int pending_pv = -1;
      for (int n = 0; ok && n < 2 * n_t; ++n) {
        const int buf = n & 1;
        if (n >= 2) {
          const int prev = n - 2;
          if (prev < n_t) {
            ok = wait_bar(&sm.bar_pfull[buf], (prev >> 1) & 1, abort_flag, kWaitLimitNs);
          } else {
            ok = wait_bar(&sm.bar_pvdone[buf], pv_phase[buf], abort_flag, kWaitLimitNs);
            pv_phase[buf] ^= 1u;
          }
          if (!ok) break;
        }
        const int s = n % kStages;
        if (!wait_bar(&sm.bar_kfull[s], (n / kStages) & 1, abort_flag, kWaitLimitNs)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t ad = sdesc_sw128(smem_addr(sm.q[kk / 4]) + 32 * (kk % 4), 16, 1024);
          const uint64_t bd = sdesc_sw128(smem_addr(sm.k[s][kk / 4]) + 32 * (kk % 4), 16, 1024);
          mma_ss(tS + buf * 128, ad, bd, kIdescQK, kk > 0 ? 1u : 0u);
        }
        mma_commit(&sm.bar_sfull[buf]);
        mma_commit(&sm.bar_kempty[s]);
        if (n >= n_t) {
          if (pending_pv >= 0 && !issue_pv(pending_pv)) {
            ok = false;
            break;
          }
          pending_pv = n - n_t;
        }
      }
      if (ok && pending_pv >= 0) ok = issue_pv(pending_pv);
      if (ok) mma_commit(&sm.bar_ofull);
      // No MMA may still be running when TMEM is freed.
      mma_commit(&sm.bar_drain);
      volatile int never = 0;
      wait_bar(&sm.bar_drain, 0, &never, kWaitLimitNs);
    }
  } else if (warp >= 4) {
    // ------------------------------------------- softmax / column sums --
    const int wg = (warp - 4) >> 2;  // key columns 64*wg .. 64*wg + 63 of each tile
    const int q4 = warp & 3;         // TMEM lane quarter
    const int row = q4 * 32 + static_cast<int>(lane);
    int g, i;
    bool valid;
    if (a.tiles_per_head > 0) {
      g = g_first;
      i = i_lo + row;
      valid = i < a.S;
    } else {
      g = g_first + row / a.rows_box;
      i = row % a.rows_box;
      valid = row < rows_used && i < a.S && g < a.qg;
    }
    const int qpos = a.pos0 + i;
    const int hq = hkv * a.qg + g;
    const uint32_t lane_addr = static_cast<uint32_t>(q4 * 32) << 16;
    const float sl2 = a.scale_log2;
    const int* sp_base = a.slot_pos + static_cast<size_t>(grp) * a.M;
    float* inc_base = a.score_inc + static_cast<size_t>(b * a.Hq + hkv * a.qg) * NK;
    // head (within the group) of each warp of this warpgroup; -1 = no valid rows
    int warp_head[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      int gw;
      if (a.tiles_per_head > 0) gw = (i_lo + w * 32 < a.S) ? g_first : -1;
      else gw = (w * 32 < rows_used) ? g_first + (w * 32) / a.rows_box : -1;
      warp_head[w] = (gw >= 0 && gw < a.qg) ? gw : -1;
    }
    float m_run = -INFINITY, l_run = 0.f, lam2 = INFINITY;
    bool ok = true;
    for (int n = 0; n < 2 * n_t; ++n) {
      const int buf = n & 1;
      const bool pass2 = n >= n_t;
      const int t = pass2 ? n - n_t : n;
      if (n == n_t) {
        // combine the two warpgroups' halves of every row (§A.6.1 merge)
        sm.rowstat[wg][row][0] = m_run;
        sm.rowstat[wg][row][1] = l_run;
        __syncwarp();
        if (lane == 0) bar_arrive(&sm.bar_rowstat);
        if (!wait_bar(&sm.bar_rowstat, 0, abort_flag, kWaitLimitNs)) {
          ok = false;
          break;
        }
        const float m0 = sm.rowstat[0][row][0], l0 = sm.rowstat[0][row][1];
        const float m1 = sm.rowstat[1][row][0], l1 = sm.rowstat[1][row][1];
        const float mm = fmaxf(m0, m1);
        const float l = l0 * fast_exp2(m0 - mm) + l1 * fast_exp2(m1 - mm);
        lam2 = (valid && mm > -INFINITY) ? mm + fast_log2(l) : INFINITY;
      }
      if (!wait_bar(&sm.bar_sfull[buf], (n >> 1) & 1, abort_flag, kWaitLimitNs)) {
        ok = false;
        break;
      }
      tc_fence_after_sync();
      float v[64];
      {
        uint32_t r[32];
        tmem_ld32(tS + lane_addr + buf * 128 + wg * 64, r);
#pragma unroll
        for (int k = 0; k < 32; ++k) v[k] = __uint_as_float(r[k]);
        tmem_ld32(tS + lane_addr + buf * 128 + wg * 64 + 32, r);
#pragma unroll
        for (int k = 0; k < 32; ++k) v[32 + k] = __uint_as_float(r[k]);
      }
      const uint16_t e = sm.tiles[t];
      const bool chunk = (e & kTileChunk) != 0;
      const bool partial = (e & kTilePartial) != 0;
      const int col0 = (e & kTileIdxMask) * kTileN + wg * 64;
      uint64_t vis_lo = ~0ull;  // bit k: column col0 + k visible to this row
      if (partial) {
        vis_lo = 0ull;
        if (chunk) {
#pragma unroll
          for (int k = 0; k < 64; ++k) {
            const int c = col0 + k;
            if (c <= i && c < a.S) vis_lo |= 1ull << k;
          }
        } else {
          for (int k = 0; k < 64; ++k) {
            const int j = col0 + k;
            const int pos = j < a.M ? __ldg(sp_base + j) : -1;
            if (pos >= 0 && pos <= qpos) vis_lo |= 1ull << k;
          }
        }
      }
      if (!pass2) {
        // pass 1: running max and sum of exp2 (log2 domain)
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
          float mx = -INFINITY;
#pragma unroll
          for (int k = 0; k < 64; ++k)
            if ((vis_lo >> k) & 1ull) mx = fmaxf(mx, v[k] * sl2);
          const float m_new = fmaxf(m_run, mx);
          if (m_new > -INFINITY) {
            float s0 = 0.f, s1 = 0.f;
#pragma unroll
            for (int k = 0; k < 64; k += 2) {
              if ((vis_lo >> k) & 1ull) s0 += fast_exp2(fmaf(v[k], sl2, -m_new));
              if ((vis_lo >> (k + 1)) & 1ull) s1 += fast_exp2(fmaf(v[k + 1], sl2, -m_new));
            }
            l_run = l_run * fast_exp2(m_run - m_new) + (s0 + s1);
            m_run = m_new;
          }
        }
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) bar_arrive(&sm.bar_pfull[buf]);
      } else {
        // pass 2: P in fp32, bf16 copy to TMEM for the P V MMA
#pragma unroll
        for (int k = 0; k < 64; ++k) {
          const float p = fast_exp2(fmaf(v[k], sl2, -lam2));
          v[k] = ((vis_lo >> k) & 1ull) ? p : 0.f;
        }
        {
          uint32_t pk[32];
#pragma unroll
          for (int x = 0; x < 32; ++x) pk[x] = pack_bf16x2(v[2 * x], v[2 * x + 1]);
          tmem_st32(tS + lane_addr + buf * 128 + wg * 64, pk);
        }
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) bar_arrive(&sm.bar_pfull[buf]);
        // column sums of P over this warp's 32 rows, then over the warpgroup
        reduce_scatter64(v, lane);
        const int cb = t & 1;
        *reinterpret_cast<float2*>(&sm.colsum[cb][wg][q4][2 * lane]) = make_float2(v[0], v[1]);
        __syncwarp();
        if (lane == 0) bar_arrive(&sm.bar_cs[cb][wg]);
        if (!wait_bar(&sm.bar_cs[cb][wg], (t >> 1) & 1, abort_flag, kWaitLimitNs)) {
          ok = false;
          break;
        }
        if (q4 < 2) {
          const int c = q4 * 32 + static_cast<int>(lane);
          const int col = col0 + c;
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
    }
    // ------------------------------------------------------------ epilogue --
    if (ok && n_t > 0 && wait_bar(&sm.bar_ofull, 0, abort_flag, kWaitLimitNs)) {
      tc_fence_after_sync();
      constexpr int kHalf = D / 2;
      uint16_t* dst = a.out + (static_cast<size_t>(b * a.Hq + hq) * a.S + i) * D + wg * kHalf;
#pragma unroll
      for (int c = 0; c < kHalf; c += 32) {
        uint32_t r[32];
        tmem_ld32(tO + lane_addr + wg * kHalf + c, r);
        uint32_t pk[16];
#pragma unroll
        for (int x = 0; x < 16; ++x)
          pk[x] = pack_bf16x2(__uint_as_float(r[2 * x]), __uint_as_float(r[2 * x + 1]));
        if (valid) {
          uint4* d4 = reinterpret_cast<uint4*>(dst + c);
#pragma unroll
          for (int x = 0; x < 4; ++x)
            d4[x] = make_uint4(pk[4 * x], pk[4 * x + 1], pk[4 * x + 2], pk[4 * x + 3]);
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
