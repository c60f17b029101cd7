// Decode (S = 1) split kernel on the tensor cores, for d = 128 and bf16 cache
// buffers: the same work items and the same per-split partials as
// decode_split_kernel (h2o_decode.cu), which decode_combine_kernel merges.
//
// What one work item (b, kv head, split of the cache slots) computes (§3.1
// Eq. 2 with the mask of §3.3.1, one query token at position pos0, split-K
// partials merged with §A.6.1's operator): for each of the q_g query heads g
// of the group, the logits a_j = scale log2(e) q_g . k_j of the split's slots
// (-inf when the slot is empty or its position is past pos0), written to
// score_inc; the split's maximum m, sum l = sum_j exp2(a_j - m) and
// unnormalised output o = sum_j exp2(a_j - m) v_j.  The last split of a
// group also takes the new token (key column M).
//
// Reading each K and V row once is the whole cost (HBM bound); the CUDA-core
// kernel spent ~80 instructions per key on its dot products and fell short
// of the copy bandwidth.  Here the products run as tcgen05 MMAs with the
// keys on the M side, so the arithmetic is a few MMAs per 32 KB tile:
//  * S^T = K Q^T: M = 128 keys of a tile, N = 16 (the q_g heads, padded with
//    whatever q rows follow them; those columns are never read), K = d.
//  * O^T += V^T P^T: M = d (the V tile read MN-major, its two 64-column
//    panels one LBO apart), N = 16, K = 128 keys; P^T is written to shared
//    memory in bf16 by the key warps, as the MMA's B operand.
// Warp 0 streams q (per item) and the K and V tiles through a four-stage
// ring of 32 KB TMA tiles, the K tiles of each item interleaved with the V
// tiles of the one before (below); warp 1 issues the MMAs, warps 2-5 hold
// one key each (TMEM lane = key) for the mask, the logits and P, and one d
// row each for the output.  The new
// token's dot products and its share of the output run on the CUDA cores.
// Every wait is bounded; on expiry the CTA drains and reports
// H2O_DEVERR_TIMEOUT.
#include <climits>
#include <cmath>
#include <cstddef>

#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kTcKeyWarps = 4;
// 8-bit buffers: warps turning code tiles into bf16 tiles (~17 instructions
// per four codes: eight warps keep up with the code stream, four did not)
constexpr int kTcConvWarps = 8;
// warp 0 TMA, warp 1 MMA, warps 2-5 keys, with 8-bit buffers warps 6-13 convert
template <bool Q8>
constexpr int tc_threads() { return 32 * (2 + kTcKeyWarps + (Q8 ? kTcConvWarps : 0)); }
// bf16 tile ring (with 8-bit buffers the code ring in front of it streams)
template <bool Q8, int QG>
constexpr int tc_stages() { return Q8 ? 2 : 4; }
// code ring: the bytes it keeps in flight set the stream's rate (a code tile
// arrived 5-6 k cycles after its TMA was issued under the full stream, so
// four 16 KB stages held it to ~22 GB/s per SM); six fit beside q_g <= 4's
// smaller logit buffers
template <int QG>
constexpr int tc_code_stages() { return QG <= 4 ? 6 : 4; }
constexpr int kTcCodeBytes = 128 * 128;      // a tile of 128 code rows
constexpr int kTcKeys = kDecodeTcTileKeys;   // 128 keys per tile
constexpr int kTcD = 128;
constexpr int kTcPanel = kTcKeys * 128;      // one 64-column panel of a tile: 16 KB
constexpr int kTcTileBytes = 2 * kTcPanel;   // a K or V tile: 32 KB
constexpr int kTcN = 16;                     // MMA N: the group's heads, padded
constexpr int kTcSmallPanel = kTcN * 128;    // a 64-column panel of 16 rows (q, P^T): 2 KB
constexpr int kTcMaxItemKeys = kDecodeTcMaxSplitLen;  // cache keys of an item
constexpr int kTcMaxItemTiles = kTcMaxItemKeys / kDecodeTcTileKeys;
// TMEM: two S^T buffers (columns 0 and 16) and the O^T accumulator (32)
constexpr uint32_t kTcTmemCols = 64;
constexpr uint32_t kTcO = 32;

// 8-bit buffers: the code tiles and their row scales, as loaded
template <bool Q8, int CS>
struct TcCodeRing {};
template <int CS>
struct TcCodeRing<true, CS> {
  alignas(1024) uint8_t codes[CS][kTcCodeBytes];
  float scl[CS][kTcKeys];
  uint64_t cfull[CS], cempty[CS];
};

template <int QG, bool Q8>
struct __align__(1024) TcSmem {
  uint8_t ring[tc_stages<Q8, QG>()][kTcTileBytes];  // bf16 K or V tiles, 2 panels of 128 rows
  TcCodeRing<Q8, tc_code_stages<QG>()> cr;
  // (128-byte-swizzled operands: 1024-byte aligned swizzle atoms)
  alignas(1024) uint8_t q[2][2][kTcSmallPanel];  // per item parity: q rows, 2 panels of 16 rows
  alignas(1024) uint8_t p[2][2][kTcSmallPanel];  // P^T of a tile (double buffer), 2 panels of 64 keys
  float lg[2][kTcMaxItemKeys * QG];       // per item parity: its logits (log2 units), key-major
  int32_t pos[2][kTcMaxItemKeys];         // per item parity: its slots' positions
  float red[2][kTcKeyWarps][QG];          // per phase parity: per-warp maxima
  float red2[2][kTcKeyWarps][QG];         // per phase parity: per-warp sums
  float newlg[2][QG];                     // per item parity: the new token's logits
  uint64_t full[tc_stages<Q8, QG>()], empty[tc_stages<Q8, QG>()];
  uint64_t qfull[2], qempty[2], sfull[2], sfree[2], pfull[2], pempty[2];
  uint64_t ofull, oempty, ksync, drain;
  uint32_t taddr;
  int abort_flag;
};

// swizzled operands start on 1024-byte boundaries, TMA tiles at least 128
template <int QG, bool Q8>
constexpr bool tc_layout_ok() {
  using T = TcSmem<QG, Q8>;
  return offsetof(T, ring) % 1024 == 0 && offsetof(T, q) % 1024 == 0 &&
         offsetof(T, p) % 1024 == 0 && offsetof(T, cr) % 1024 == 0;
}
static_assert(tc_layout_ok<4, false>() && tc_layout_ok<8, false>() && tc_layout_ok<4, true>() &&
                  tc_layout_ok<8, true>(),
              "decode_tc_kernel shared-memory layout");

__device__ __forceinline__ bool twait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  return wait_bar(bar, parity, abort, kWaitLimitNs);
}

// Warp-uniform bounded wait (the TMEM loads after it are .sync.aligned).
__device__ __forceinline__ bool twwait(uint64_t* bar, uint32_t parity, volatile int* abort) {
  const bool r = twait(bar, parity, abort);
  return __all_sync(0xffffffffu, r) != 0;
}

// One work item: (b, kv head) group, split s of the cache slots.
struct TcItem {
  int grp, s, j0, n_cache, n_kt;
  bool last;
};

__device__ __forceinline__ TcItem tc_item(const DecodeArgs& a, int it) {
  TcItem x;
  x.grp = it / a.n_split;
  x.s = it % a.n_split;
  x.j0 = x.s * a.split_len;
  x.n_cache = min(a.split_len, a.M - x.j0);  // >= 1
  x.last = x.s == a.n_split - 1 && a.with_new;
  x.n_kt = (x.n_cache + kTcKeys - 1) / kTcKeys;
  return x;
}

// Two 8-bit codes of a cache row read back as the 8-bit format defines,
// bf16(code * scale), packed (element i in the low half).  `wb` holds four
// codes with their sign bits flipped (code + 128 as unsigned bytes); byte i
// placed under the exponent of 2^23 gives the float 2^23 + 128 + code
// exactly, and subtracting 2^23 + 128 leaves the code; then an fp32
// multiply and round-to-nearest-even to bf16, as in the read-back kernel.
__device__ __forceinline__ uint32_t q8_bf16x2(uint32_t wb, int i, float s) {
  const float lo = __uint_as_float(__byte_perm(wb, 0x4B000000u, 0x7650u | i));
  const float hi = __uint_as_float(__byte_perm(wb, 0x4B000000u, 0x7650u | (i + 1)));
  const float2 c = __fadd2_rn(make_float2(lo, hi), make_float2(-8388736.f, -8388736.f));
  const float2 x = __fmul2_rn(c, make_float2(s, s));
  return pack_bf16x2(x.x, x.y);
}

// K-major SW128 descriptors of the eight K-steps (16 of d each) of an
// operand of 64-column panels `panel` bytes apart.
__device__ __forceinline__ void kmajor8(uint32_t base, uint32_t panel, uint64_t (&d)[8]) {
  const uint64_t d0 = sdesc_sw128(base, 16, 1024);
#pragma unroll
  for (int kk = 0; kk < 8; ++kk)
    d[kk] = d0 + static_cast<uint64_t>((panel >> 4) * (kk / 4) + 2 * (kk % 4));
}

// The CTA's items k = 0 .. n-1 (items blockIdx.x + k gridDim.x) run as
// phases ph = 0 .. n: phase ph takes the K tiles of item ph interleaved with
// the V tiles of item ph - 1 (tile t of each in turn), in the ring, in the
// MMA issue and in the key warps, which form item ph's logits and item
// ph - 1's P^T side by side.  At the end of a phase one barrier of the key
// warps completes item ph's maximum and item ph - 1's sum, then item ph - 1's
// output is read out.  So the K and V streams of consecutive items overlap
// and no item waits for its own maximum with an idle ring.
template <int QG, bool Q8>
__global__ void __launch_bounds__(tc_threads<Q8>(), 1) decode_tc_kernel(const __grid_constant__ DecodeArgs a) {
  constexpr int NS = tc_stages<Q8, QG>();
  constexpr int CSt = tc_code_stages<QG>();
  extern __shared__ uint8_t smem_raw[];
  auto& sm = *reinterpret_cast<TcSmem<QG, Q8>*>(smem_raw +
                                                ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u));
  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const uint32_t lane = tid & 31;
  const int n_items = a.n_split * a.B * a.Hkv;
  // this CTA's items (grid <= n_items, so at least one)
  const int n_mine = (n_items - static_cast<int>(blockIdx.x) + static_cast<int>(gridDim.x) - 1) /
                     static_cast<int>(gridDim.x);
  auto item_of = [&](int k) { return tc_item(a, static_cast<int>(blockIdx.x) + k * static_cast<int>(gridDim.x)); };

  if (tid == 0) launch_dependents();  // the combine may be placed (it waits for this grid)
  if (tid == 0) {
    for (int s = 0; s < NS; ++s) {
      bar_init(&sm.full[s], Q8 ? kTcConvWarps : 1);  // (8-bit: the converter warps)
      bar_init(&sm.empty[s], 1);
    }
    if constexpr (Q8) {
      for (int s = 0; s < CSt; ++s) {
        bar_init(&sm.cr.cfull[s], 1);
        bar_init(&sm.cr.cempty[s], kTcConvWarps);
      }
    }
    for (int x = 0; x < 2; ++x) {
      bar_init(&sm.qfull[x], 1);
      bar_init(&sm.qempty[x], 1);
      bar_init(&sm.sfull[x], 1);
      bar_init(&sm.sfree[x], kTcKeyWarps);
      bar_init(&sm.pfull[x], kTcKeyWarps);
      bar_init(&sm.pempty[x], 1);
    }
    bar_init(&sm.ofull, 1);
    bar_init(&sm.oempty, kTcKeyWarps);
    bar_init(&sm.ksync, kTcKeyWarps);
    bar_init(&sm.drain, 1);
    sm.abort_flag = 0;
    fence_bar_init();
  }
  if (warp == 1) {
    tmem_alloc(&sm.taddr, kTcTmemCols);
    tmem_relinquish();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = sm.taddr;
  volatile int* abort_flag = &sm.abort_flag;

  if (warp == 0) {
    // ---------------------------------------------------------- TMA producer --
    if (lane == 0) {
      tma_prefetch_desc(&a.tm_q);
      tma_prefetch_desc(&a.tm_kc);
      tma_prefetch_desc(&a.tm_vc);
      uint32_t slot = 0;  // tiles issued so far
      int qloads = 0;     // q loads issued so far
      bool ok = true;
      // one tile into the next ring slot; K and V are read once: evict-first,
      // so that the logits written to score_inc stay in L2 for the combine
      // (8-bit buffers: the code tile and its scales into the code ring)
      constexpr int RS = Q8 ? CSt : NS;
      auto load = [&](const CUtensorMap* m, const TcItem& x, int t) -> bool {
        const int s = slot % RS;
        if constexpr (Q8) {
          if (slot >= RS && !twait(&sm.cr.cempty[s], ((slot / RS) - 1) & 1, abort_flag))
            return false;
          const bool is_v = m == &a.tm_vc;
          bar_expect_tx(&sm.cr.cfull[s], kTcCodeBytes + kTcKeys * 4);
          tma_load_3d_once(sm.cr.codes[s], m, &sm.cr.cfull[s], 0, x.j0 + kTcKeys * t, x.grp);
          tma_load_1d(sm.cr.scl[s], is_v ? &a.tm_vs : &a.tm_ks, &sm.cr.cfull[s],
                      x.grp * a.M + x.j0 + kTcKeys * t);
        } else {
          if (slot >= RS && !twait(&sm.empty[s], ((slot / RS) - 1) & 1, abort_flag)) return false;
          bar_expect_tx(&sm.full[s], kTcTileBytes);
          for (int p = 0; p < 2; ++p)
            tma_load_3d_once(sm.ring[s] + p * kTcPanel, m, &sm.full[s], 64 * p,
                             x.j0 + kTcKeys * t, x.grp);
        }
        ++slot;
        return true;
      };
      for (int ph = 0; ok && ph <= n_mine; ++ph) {
        const bool hk = ph < n_mine, hv = ph > 0;
        TcItem xk{}, xv{};
        if (hk) xk = item_of(ph);
        if (hv) xv = item_of(ph - 1);
        if (hk) {
          const int qb = ph & 1;
          if (ph >= 2 && !twait(&sm.qempty[qb], ((ph >> 1) - 1) & 1, abort_flag)) break;
          const int b = xk.grp / a.Hkv, h = xk.grp % a.Hkv;
          bar_expect_tx(&sm.qfull[qb], 2 * kTcSmallPanel);
          for (int p = 0; p < 2; ++p)
            tma_load_3d(sm.q[qb][p], &a.tm_q, &sm.qfull[qb], 64 * p, h * a.qg, b);
          ++qloads;
        }
        const int tk = hk ? xk.n_kt : 0, tv = hv ? xv.n_kt : 0;
        for (int t = 0; ok && t < max(tk, tv); ++t) {
          if (t < tk) ok = load(&a.tm_kc, xk, t);
          if (ok && t < tv) ok = load(&a.tm_vc, xv, t);
        }
      }
      if (*abort_flag) {
        // let the copies still in flight land: the latest load of each stage
        // and of each q buffer
        volatile int never = 0;
        for (uint32_t u = slot > RS ? slot - RS : 0; u < slot; ++u) {
          if constexpr (Q8)
            wait_bar(&sm.cr.cfull[u % RS], (u / RS) & 1, &never, 100000000ull);
          else
            wait_bar(&sm.full[u % RS], (u / RS) & 1, &never, 100000000ull);
        }
        for (int u = qloads > 2 ? qloads - 2 : 0; u < qloads; ++u)
          wait_bar(&sm.qfull[u & 1], (u >> 1) & 1, &never, 100000000ull);
      }
    }
  } else if (warp == 1) {
    // ------------------------------------------------------------- MMA issue --
    if (lane == 0) {
      constexpr uint32_t kIdS = idesc_bf16_f32(128, kTcN, false);      // S^T: A = K, B = q
      constexpr uint32_t kIdO = idesc_bf16_f32_amn(128, kTcN, false);  // O^T: A = V^T, B = P^T
      constexpr uint64_t kStage = kTcTileBytes >> 4;
      // buffer 1 of q / P^T lies two small panels after buffer 0
      constexpr uint64_t kSmallBuf = (2 * kTcSmallPanel) >> 4;
      uint64_t kd0[8], qd0[8], pd0[8];
      kmajor8(smem_addr(sm.ring[0]), kTcPanel, kd0);
      kmajor8(smem_addr(sm.q[0][0]), kTcSmallPanel, qd0);
      kmajor8(smem_addr(sm.p[0][0]), kTcSmallPanel, pd0);
      // V tile as A = V^T (M = d): MN-major, panels LBO apart, a K-step of 16
      // keys is 2 KB
      const uint64_t vd0 = sdesc_sw128(smem_addr(sm.ring[0]), kTcPanel, 1024);
      uint32_t slot = 0, kt_g = 0, vt_g = 0;
      bool ok = true;
      // a tile in the ring: with 8-bit buffers it is signalled by the
      // converter warps, whose arrivals a suspended wait noticed only
      // ~650 cycles later (measured), so it is polled
      auto tile_wait = [&](uint64_t* bar, uint32_t parity, volatile int* abort) -> bool {
        if constexpr (Q8) return wait_bar_poll(bar, parity, abort, kWaitLimitNs);
        else return twait(bar, parity, abort);
      };
      // S^T of item k's tile t
      auto issue_s = [&](int qb) -> bool {
        const int sb = kt_g & 1, s = slot % NS;
        if ((kt_g >= 2 && !twait(&sm.sfree[sb], ((kt_g >> 1) - 1) & 1, abort_flag)) ||
            !tile_wait(&sm.full[s], (slot / NS) & 1, abort_flag))
          return false;
        tc_fence_after_sync();
        uint64_t kd[8], qd[8];
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          kd[kk] = kd0[kk] + kStage * s;
          qd[kk] = qd0[kk] + kSmallBuf * qb;
        }
        mma_ss_x8<false>(tmem + 16 * sb, kd, qd, kIdS, 0u);
        mma_commit(&sm.sfull[sb]);
        mma_commit(&sm.empty[s]);
        ++kt_g;
        ++slot;
        return true;
      };
      // O^T (+)= V^T P^T of the previous item's tile t
      auto issue_pv = [&](int t) -> bool {
        const int pb = vt_g & 1, s = slot % NS;
        if (!twait(&sm.pfull[pb], (vt_g >> 1) & 1, abort_flag) ||
            !tile_wait(&sm.full[s], (slot / NS) & 1, abort_flag))
          return false;
        tc_fence_after_sync();
        uint64_t vd[8], pd[8];
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          vd[kk] = vd0 + kStage * s + 128 * kk;
          pd[kk] = pd0[kk] + kSmallBuf * pb;
        }
        mma_ss_x8<false>(tmem + kTcO, vd, pd, kIdO, t > 0 ? 1u : 0u);
        mma_commit(&sm.pempty[pb]);
        mma_commit(&sm.empty[s]);
        ++vt_g;
        ++slot;
        return true;
      };
      for (int ph = 0; ok && ph <= n_mine; ++ph) {
        const bool hk = ph < n_mine, hv = ph > 0;
        const int tk = hk ? item_of(ph).n_kt : 0, tv = hv ? item_of(ph - 1).n_kt : 0;
        const int qb = ph & 1;
        if (hk && !twait(&sm.qfull[qb], (ph >> 1) & 1, abort_flag)) break;
        for (int t = 0; ok && t < max(tk, tv); ++t) {
          if (t < tk) ok = issue_s(qb);
          // item ph - 1's first P V overwrites O^T: item ph - 2's must have
          // been read out (at the end of the previous phase)
          if (ok && t == 0 && hv && ph >= 2) ok = twait(&sm.oempty, (ph - 2) & 1, abort_flag);
          if (ok && t < tv) ok = issue_pv(t);
        }
        if (!ok) break;
        if (hk) mma_commit(&sm.qempty[qb]);
        if (hv) mma_commit(&sm.ofull);
      }
      // no MMA may still be running when TMEM is freed
      mma_commit(&sm.drain);
      volatile int never = 0;
      wait_bar(&sm.drain, 0, &never, kWaitLimitNs);
    }
  } else if (warp < 2 + kTcKeyWarps) {
    // -------------------------------------------------------------- key warps --
    // Thread kl holds key kl of each tile (TMEM lane kl of S^T) and row d = kl
    // of O^T; lane quarter warp % 4.
    const int q4 = warp & 3;
    const int kl = q4 * 32 + static_cast<int>(lane);
    const uint32_t lane_addr = static_cast<uint32_t>(q4 * 32) << 16;
    const size_t nk = static_cast<size_t>(a.nk);
    uint32_t kt_g = 0, vt_g = 0;
    float m_prev[QG], pn_prev[QG];  // the previous item's maximum and new-token weight
#pragma unroll
    for (int g = 0; g < QG; ++g) {
      m_prev[g] = -INFINITY;
      pn_prev[g] = 0.f;
    }
    // The slots' positions of an item are loaded one phase ahead (the loads
    // are in flight while the phase streams; a load issued just before its
    // tile waited out the HBM latency under the K / V stream) and staged in
    // shared memory.  This thread's keys of item k: kl + 128 u.
    int pnext[kTcMaxItemTiles];
    auto load_pos = [&](int k) {
      const TcItem x = item_of(k);
      const int32_t* sp = a.slot_pos + static_cast<size_t>(x.grp) * a.M + x.j0;
#pragma unroll
      for (int u = 0; u < kTcMaxItemTiles; ++u) {
        const int kli = u * kTcKeys + kl;
        pnext[u] = kli < x.n_cache ? __ldg(sp + kli) : -1;
      }
    };
    auto store_pos = [&](int k) {
#pragma unroll
      for (int u = 0; u < kTcMaxItemTiles; ++u) sm.pos[k & 1][u * kTcKeys + kl] = pnext[u];
    };
    load_pos(0);
    store_pos(0);
    bool ok = true;
    for (int ph = 0; ok && ph <= n_mine; ++ph) {
      const bool hk = ph < n_mine, hv = ph > 0;
      TcItem xk{}, xv{};
      if (hk) xk = item_of(ph);
      if (hv) xv = item_of(ph - 1);
      const int ib = ph & 1;  // item ph's parity (item ph - 1: ib ^ 1)
      if (ph + 1 < n_mine) load_pos(ph + 1);
      const size_t row0k = hk ? static_cast<size_t>(xk.grp / a.Hkv) * a.Hq +
                                    static_cast<size_t>(xk.grp % a.Hkv) * a.qg
                              : 0;
      if (hk && xk.last && warp == 2) {
        // the new token's logits: lanes over d, four elements each
        const uint2 kw = __ldg(reinterpret_cast<const uint2*>(a.k_new + static_cast<size_t>(xk.grp) * kTcD) + lane);
        const float k4[4] = {__uint_as_float(kw.x << 16), __uint_as_float(kw.x & 0xFFFF0000u),
                             __uint_as_float(kw.y << 16), __uint_as_float(kw.y & 0xFFFF0000u)};
#pragma unroll
        for (int g = 0; g < QG; ++g) {
          float dsum = 0.f;
          if (g < a.qg) {
            const uint2 qw = __ldg(reinterpret_cast<const uint2*>(a.q + (row0k + g) * kTcD) + lane);
            dsum = fmaf(__uint_as_float(qw.x << 16), k4[0], dsum);
            dsum = fmaf(__uint_as_float(qw.x & 0xFFFF0000u), k4[1], dsum);
            dsum = fmaf(__uint_as_float(qw.y << 16), k4[2], dsum);
            dsum = fmaf(__uint_as_float(qw.y & 0xFFFF0000u), k4[3], dsum);
          }
#pragma unroll
          for (int o = 16; o > 0; o >>= 1) dsum += __shfl_xor_sync(0xffffffffu, dsum, o);
          if (lane == 0) sm.newlg[ib][g] = dsum * a.scale_log2;
        }
      }
      float mx[QG], ls[QG];
#pragma unroll
      for (int g = 0; g < QG; ++g) {
        mx[g] = -INFINITY;
        ls[g] = 0.f;
      }
      const int tk = hk ? xk.n_kt : 0, tv = hv ? xv.n_kt : 0;
      for (int t = 0; t < max(tk, tv); ++t) {
        if (t < tk) {
          // ---- item ph's logits of tile t: mask, log2 scale, to score_inc
          const int sb = kt_g & 1;
          const int kli = t * kTcKeys + kl;  // key within the item
          const bool valid = kli < xk.n_cache;
          const int pos = sm.pos[ib][kli];  // (this thread's own entry)
          if (!twwait(&sm.sfull[sb], (kt_g >> 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          uint32_t r[8];
          tmem_ld8(tmem + lane_addr + 16 * sb, r);
          tc_fence_before_sync();
          __syncwarp();
          if (lane == 0) bar_arrive(&sm.sfree[sb]);
          ++kt_g;
          const bool vis = pos >= 0 && pos <= a.pos0;
          if (valid) {
#pragma unroll
            for (int g = 0; g < QG; ++g) {
              if (g < a.qg) {
                const float av = vis ? __uint_as_float(r[g]) * a.scale_log2 : -INFINITY;
                a.score_inc[(row0k + g) * nk + xk.j0 + kli] = av;
                sm.lg[ib][kli * QG + g] = av;
                mx[g] = fmaxf(mx[g], av);
              }
            }
          }
        }
        if (t < tv) {
          // ---- item ph - 1's P^T of tile t: exp2(a - m) in bf16 for the MMA,
          // its sum in fp32
          const int pb = vt_g & 1;
          if (vt_g >= 2 && !twwait(&sm.pempty[pb], ((vt_g >> 1) - 1) & 1, abort_flag)) {
            ok = false;
            break;
          }
          const int kli = t * kTcKeys + kl;
          const bool valid = kli < xv.n_cache;
          uint8_t* prow = sm.p[pb][kl >> 6];
#pragma unroll
          for (int g = 0; g < QG; ++g) {
            float pv = 0.f;
            if (valid && g < a.qg && m_prev[g] > -INFINITY)
              pv = fast_exp2(sm.lg[ib ^ 1][kli * QG + g] - m_prev[g]);
            ls[g] += pv;
            // row g, key kl of the 128-byte-swizzled K-major panel
            const uint32_t c = static_cast<uint32_t>(((kl & 63) >> 3) ^ (g & 7));
            *reinterpret_cast<uint16_t*>(prow + g * 128 + c * 16 + (kl & 7) * 2) =
                static_cast<uint16_t>(pack_bf16x2(pv, 0.f) & 0xFFFFu);
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) bar_arrive(&sm.pfull[pb]);
          ++vt_g;
        }
      }
      if (!ok) break;
      // the next item's positions (each thread's own entries; read after the
      // next phase began, and item ph's parity buffer is not touched)
      if (ph + 1 < n_mine) store_pos(ph + 1);
      // ---- end of the phase: item ph's maximum and item ph - 1's sum over
      // the four key warps.  The barrier is polled: the warps arrive within a
      // few hundred cycles of each other, and a suspended wait took ~1 us to
      // wake.  red / red2 alternate by phase: a warp can be at most one
      // phase ahead of the slowest.
#pragma unroll
      for (int g = 0; g < QG; ++g) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
          mx[g] = fmaxf(mx[g], __shfl_xor_sync(0xffffffffu, mx[g], o));
          ls[g] += __shfl_xor_sync(0xffffffffu, ls[g], o);
        }
        if (lane == 0) {
          sm.red[ib][q4][g] = mx[g];
          sm.red2[ib][q4][g] = ls[g];
        }
      }
      __syncwarp();
      if (lane == 0) bar_arrive(&sm.ksync);
      {
        const bool r = wait_bar_poll(&sm.ksync, ph & 1, abort_flag, kWaitLimitNs);
        if (!__all_sync(0xffffffffu, r)) break;
      }
      if (hv) {
        // ---- item ph - 1's partials: (max, sum, unnormalised output) per head
        const size_t row0v = static_cast<size_t>(xv.grp / a.Hkv) * a.Hq +
                             static_cast<size_t>(xv.grp % a.Hkv) * a.qg;
        float l[QG];
#pragma unroll
        for (int g = 0; g < QG; ++g)
          l[g] = ((sm.red2[ib][0][g] + sm.red2[ib][1][g]) + (sm.red2[ib][2][g] + sm.red2[ib][3][g])) +
                 pn_prev[g];
        if (!twwait(&sm.ofull, (ph - 1) & 1, abort_flag)) break;
        tc_fence_after_sync();
        uint32_t o[8];
        tmem_ld8(tmem + lane_addr + kTcO, o);
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) bar_arrive(&sm.oempty);
        float vn = 0.f;  // the new token's value, element d = kl
        if (xv.last) {
          const uint16_t vb = __ldg(a.v_new + static_cast<size_t>(xv.grp) * kTcD + kl);
          vn = __uint_as_float(static_cast<uint32_t>(vb) << 16);
        }
#pragma unroll
        for (int g = 0; g < QG; ++g) {
          if (g < a.qg) {
            float* pm = a.part + ((row0v + g) * a.n_split + xv.s) * (2 + kTcD);
            pm[2 + kl] = fmaf(pn_prev[g], vn, __uint_as_float(o[g]));
            if (kl == g) {
              pm[0] = m_prev[g];
              pm[1] = l[g];
            }
          }
        }
      }
      if (hk) {
        // item ph's maximum (with its new token) and the new token's weight
#pragma unroll
        for (int g = 0; g < QG; ++g) {
          float mg = fmaxf(fmaxf(sm.red[ib][0][g], sm.red[ib][1][g]),
                           fmaxf(sm.red[ib][2][g], sm.red[ib][3][g]));
          float pn = 0.f;
          if (xk.last) {
            const float an = sm.newlg[ib][g];
            mg = fmaxf(mg, an);
            pn = mg > -INFINITY ? fast_exp2(an - mg) : 0.f;
            if (kl == g && g < a.qg) a.score_inc[(row0k + g) * nk + a.M] = an;
          }
          m_prev[g] = mg;
          pn_prev[g] = pn;
        }
      }
    }
  } else if constexpr (Q8) {
    // ------------------------------------------------------------ converters --
    // 8-bit buffers: the converter warps turn each code tile into the bf16
    // tile the MMA reads, in the ring order of the producer: warp cw takes
    // rows 4 (8 i + cw) .. + 3, sixteen codes of a row per lane, read back as
    // the 8-bit format defines, bf16(code * scale) (q8_bf16x2), and written
    // where a 128-byte-swizzled TMA load of the bf16 row would have put them.
    const int cw = warp - 2 - kTcKeyWarps;
    // lane: codes 16 g .. 16 g + 15 (g = lane % 8) of row 4 i + lane / 8 of
    // the warp's rows; bf16 columns 16 g .. are chunks 2 g' and 2 g' + 1 of
    // panel g / 4 (g' = g % 4)
    const int g8 = static_cast<int>(lane & 7u), rsub = static_cast<int>(lane >> 3);
    const uint32_t c_lo = static_cast<uint32_t>(2 * (g8 & 3));
    uint32_t n = 0;  // tiles converted so far
    bool ok = true;
    for (int ph = 0; ok && ph <= n_mine; ++ph) {
      const int tk = ph < n_mine ? item_of(ph).n_kt : 0, tv = ph > 0 ? item_of(ph - 1).n_kt : 0;
      for (int t = 0; ok && t < max(tk, tv); ++t) {
        for (int v = 0; v < 2; ++v) {
          if (t >= (v == 0 ? tk : tv)) continue;
          const int cs = n % CSt, s = n % NS;
          if (!twait(&sm.cr.cfull[cs], (n / CSt) & 1, abort_flag) ||
              (n >= static_cast<uint32_t>(NS) && !twait(&sm.empty[s], ((n / NS) - 1) & 1, abort_flag))) {
            ok = false;
            break;
          }
          const uint8_t* src = sm.cr.codes[cs] + 16 * g8;
          uint8_t* dst = sm.ring[s] + (g8 >> 2) * kTcPanel;
#pragma unroll
          for (int i = 0; i < kTcKeys / (4 * kTcConvWarps); ++i) {
            const int r = (i * kTcConvWarps + cw) * 4 + rsub;  // row of the tile
            const uint4 w = *reinterpret_cast<const uint4*>(src + r * 128);
            const float sc = sm.cr.scl[cs][r];
            const uint32_t w4[4] = {w.x ^ 0x80808080u, w.y ^ 0x80808080u, w.z ^ 0x80808080u,
                                    w.w ^ 0x80808080u};
            uint4 o0, o1;
            o0.x = q8_bf16x2(w4[0], 0, sc);
            o0.y = q8_bf16x2(w4[0], 2, sc);
            o0.z = q8_bf16x2(w4[1], 0, sc);
            o0.w = q8_bf16x2(w4[1], 2, sc);
            o1.x = q8_bf16x2(w4[2], 0, sc);
            o1.y = q8_bf16x2(w4[2], 2, sc);
            o1.z = q8_bf16x2(w4[3], 0, sc);
            o1.w = q8_bf16x2(w4[3], 2, sc);
            uint8_t* row = dst + r * 128;
            const uint32_t sw = static_cast<uint32_t>(r & 7);
            *reinterpret_cast<uint4*>(row + ((c_lo ^ sw) << 4)) = o0;
            *reinterpret_cast<uint4*>(row + (((c_lo + 1) ^ sw) << 4)) = o1;
          }
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            bar_arrive(&sm.full[s]);
            bar_arrive(&sm.cr.cempty[cs]);
          }
          ++n;
        }
      }
    }
  }
  tc_fence_before_sync();
  __syncthreads();
  if (warp == 1) {
    __syncwarp();
    tmem_dealloc(tmem, kTcTmemCols);
  }
  if (tid == 0 && sm.abort_flag) atomicOr(a.err, H2O_DEVERR_TIMEOUT);
}

template <int QG, bool Q8>
cudaError_t launch_tc(const DecodeArgs& a, cudaStream_t stream) {
  const size_t smem = sizeof(TcSmem<QG, Q8>) + 1024;
  static OncePerDevice once;
  static int resident[kMaxDevices];
  cudaError_t e = once.run([smem](int d) {
    cudaError_t r = cudaFuncSetAttribute(decode_tc_kernel<QG, Q8>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (r != cudaSuccess) return r;
    int per_sm = 0, sms = 0;
    r = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_tc_kernel<QG, Q8>,
                                                      tc_threads<Q8>(), smem);
    if (r != cudaSuccess) return r;
    r = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, d);
    if (r != cudaSuccess) return r;
    resident[d] = (per_sm > 0 ? per_sm : 1) * sms;
    return cudaSuccess;
  });
  if (e != cudaSuccess) return e;
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const int n_items = a.n_split * a.B * a.Hkv;
  const int grid = n_items < resident[dev] ? n_items : resident[dev];
  decode_tc_kernel<QG, Q8><<<grid, tc_threads<Q8>(), smem, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t stream) {
  if (a.q8) return a.qg <= 4 ? launch_tc<4, true>(a, stream) : launch_tc<8, true>(a, stream);
  return a.qg <= 4 ? launch_tc<4, false>(a, stream) : launch_tc<8, false>(a, stream);
}

}  // namespace h2o
