// H2O cache update: score accumulation, eviction selection and K/V scatter.
//
// One CTA of 1024 threads per (batch, KV head); per §3.1.1 Eq. 3 the score of
// a slot is the running sum of the attention weights its column received, and
// the S slots with the smallest scores are overwritten by the chunk (§3.1.1);
// the write is the scatter along the slot axis of §3.2 / §A.1.1.
//
//  1. acc_j = scores_j + (inc_0j + inc_1j + ... ) in float32, query heads of the
//     GQA group added in ascending order with no fused multiply-add, so the
//     result is bit-identical to any implementation that follows that order.
//  2. Each candidate slot gets a 32-bit key that orders (empty first, then acc
//     ascending): 0 for an empty slot, bits(acc) + 1 otherwise (non-negative
//     floats order like their bit patterns); protected slots (inside the recent
//     window) get 0xFFFFFFFF.  Ties on the key are broken by the slot index.
//  3. S = 1 is an argmin over (key, slot).  Otherwise a 4-pass radix select
//     (8-bit digits, shared-memory histogram) finds the S-th smallest key T and
//     how many keys equal to T are taken (the lowest slots first).
//  4. One sweep in slot order computes with block scans the rank c of every
//     evicted slot (the c-th smallest evicted slot receives token pos0 + c) and
//     writes slot_pos, scores, evict_idx; whole warps copy the K and V rows of
//     the evicted slots with 16-byte vector loads and stores.
//
// Two variants.  When the keys and accumulated scores of one (b, kv head)
// fit in shared memory and S > 1, a cluster of C CTAs handles the (b, kv
// head): every CTA computes keys and scores into shared memory (each thread
// owns a contiguous run of slots and issues all loads of a batch before the
// first sum), runs the same deterministic selection (one packed scan of the
// counts below and equal to the threshold gives every slot's rank), a cluster
// barrier separates all reads of the old state from the writes, CTA 0 writes
// scores / slot_pos / evict_idx, and the C CTAs share the row copies with
// several 16-byte loads in flight per thread.  The whole update is latency
// bound (a few MB per chunk), so the design minimises dependent round trips.
// Otherwise one CTA per (b, kv head) recomputes keys from global memory on
// every pass.  S = 1 has a kernel of its own (update_decode_kernel).
#include <algorithm>

#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kUpdThreads = 1024;
constexpr int kUpdWarps = kUpdThreads / 32;
constexpr uint32_t kProtected = 0xFFFFFFFFu;

struct UpdSmem {
  uint32_t hist[256];
  uint32_t warp_tot[kUpdWarps];
  uint32_t warp_tot2[kUpdWarps];
  uint32_t bcast[4];
};

__device__ __forceinline__ float group_sum(const float* inc, int stride, int qg, int j) {
  float t = __ldg(inc + j);
  for (int g = 1; g < qg; ++g) t = __fadd_rn(t, __ldg(inc + static_cast<size_t>(g) * stride + j));
  return t;
}

// The group sum of score_inc, or 0 for h2o_evict_insert (a.insert: the
// paper's order ranks and keeps the scores as they were before the chunk).
__device__ __forceinline__ float inc_group(const UpdateArgs& a, const float* inc, int stride,
                                           int j) {
  return a.insert ? 0.f : group_sum(inc, stride, a.qg, j);
}

// Tokens processed when the choice is made: t of h2o_norm's age t - t(j).
__device__ __forceinline__ int t_choice(const UpdateArgs& a) {
  return a.insert ? a.pos0 : a.pos0 + a.S;
}

// Selection key of a slot (step 2 above).  The rank value is the score for
// h2o and h2o_orig (the caller passes the batch sum) and, for h2o_norm, the
// score over the slot's age t - t(j), t = pos0 + S (fp32, rounded to nearest).
__device__ __forceinline__ uint32_t make_key(float acc, int pos, int thr, int policy, int t_now) {
  if (pos >= thr) return kProtected;
  if (pos < 0) return 0u;
  const float r = policy == H2O_POLICY_NORM ? __fdiv_rn(acc, __int2float_rn(t_now - pos)) : acc;
  return min(__float_as_uint(r) + 1u, kProtected - 1u);
}

// Eq. 3 for slot j of (b, h): scores + the group's summed weights.
__device__ __forceinline__ float slot_acc(const UpdateArgs& a, int b, int h, int j) {
  const size_t grp = static_cast<size_t>(b) * a.Hkv + h;
  const float* inc = a.score_inc + static_cast<size_t>(b * a.Hq + h * a.qg) * (a.M + a.S);
  return __fadd_rn(a.scores[grp * a.M + j], inc_group(a, inc, a.M + a.S, j));
}

// Key of slot j for the selection of (b, h) (h2o_orig: of KV head h, b = 0);
// *acc_out receives the score of (b, h).
__device__ __forceinline__ uint32_t slot_key(const UpdateArgs& a, int b, int h, int j, int thr,
                                             float* acc_out) {
  const int pos = a.slot_pos[(static_cast<size_t>(b) * a.Hkv + h) * a.M + j];
  float acc = slot_acc(a, b, h, j);
  *acc_out = acc;
  if (a.policy == H2O_POLICY_ORIG)
    for (int bb = 1; bb < a.B; ++bb) acc = __fadd_rn(acc, slot_acc(a, bb, h, j));
  return make_key(acc, pos, thr, a.policy, t_choice(a));
}

// Exclusive block scan of one bit per thread; returns the prefix, total in *tot.
__device__ __forceinline__ uint32_t block_scan_bit(bool f, uint32_t* warp_tot, uint32_t* tot) {
  const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;
  const uint32_t m = __ballot_sync(0xffffffffu, f);
  if (l == 0) warp_tot[w] = __popc(m);
  __syncthreads();
  uint32_t before = 0, total = 0;
  for (int x = 0; x < kUpdWarps; ++x) {
    const uint32_t c = warp_tot[x];
    before += x < w ? c : 0u;
    total += c;
  }
  __syncthreads();
  *tot = total;
  return before + __popc(m & ((1u << l) - 1u));
}

__device__ __forceinline__ void copy_row(const UpdateArgs& a, int grp, int c, int e, int lane) {
  // 32 lanes: lanes 0-15 copy the K row, 16-31 the V row, in 16-byte pieces.
  // No cache pointers: the rows are written by another kernel (8-bit buffers).
  if (a.k_cache == nullptr) return;
  const int vec = a.d / 8;  // uint4 per row
  const bool is_v = lane >= 16;
  const int l = lane & 15;
  const uint16_t* src = (is_v ? a.v_new : a.k_new) + (static_cast<size_t>(grp) * a.S + c) * a.d;
  uint16_t* dst = (is_v ? a.v_cache : a.k_cache) + (static_cast<size_t>(grp) * a.M + e) * a.d;
  for (int x = l; x < vec; x += 16)
    reinterpret_cast<uint4*>(dst)[x] = __ldg(reinterpret_cast<const uint4*>(src) + x);
}

__global__ void __launch_bounds__(kUpdThreads, 1) update_kernel(const UpdateArgs a) {
  grid_dependency_wait();  // (a no-op unless launched as a programmatic dependent)
  __shared__ UpdSmem sm;
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  // one (b, h) per CTA; h2o_orig: one KV head per CTA, for every b
  const bool orig = a.policy == H2O_POLICY_ORIG;
  const int b = orig ? 0 : static_cast<int>(blockIdx.x) / a.Hkv;
  const int h = orig ? static_cast<int>(blockIdx.x) : static_cast<int>(blockIdx.x) % a.Hkv;
  const int nb = orig ? a.B : 1;  // batch entries whose state this CTA writes
  const int thr = a.pos0 + a.S - a.W;  // slots holding positions >= thr are protected
  const int M = a.M, S = a.S;

  uint32_t T = 0;         // threshold key
  uint32_t take_eq = 0;   // keys equal to T that are evicted (lowest slots first)
  {
    uint32_t prefix = 0, mask = 0, kth = static_cast<uint32_t>(S);
    for (int pass = 0; pass < 4; ++pass) {
      const int shift = 24 - 8 * pass;
      for (int x = tid; x < 256; x += kUpdThreads) sm.hist[x] = 0u;
      __syncthreads();
      for (int j = tid; j < M; j += kUpdThreads) {
        float acc;
        const uint32_t key = slot_key(a, b, h, j, thr, &acc);
        if ((key & mask) == prefix) atomicAdd(&sm.hist[(key >> shift) & 255u], 1u);
      }
      __syncthreads();
      if (warp == 0) {
        // lane l owns bins 8l .. 8l+7; find the bin holding the kth key
        uint32_t c[8], s = 0;
#pragma unroll
        for (int x = 0; x < 8; ++x) {
          c[x] = sm.hist[8 * lane + x];
          s += c[x];
        }
        uint32_t incl = s;
        for (int o = 1; o < 32; o <<= 1) {
          const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
          if (lane >= o) incl += y;
        }
        uint32_t run = incl - s;
#pragma unroll
        for (int x = 0; x < 8; ++x) {
          if (run < kth && kth <= run + c[x]) {
            sm.bcast[0] = static_cast<uint32_t>(8 * lane + x);
            sm.bcast[1] = kth - run;
          }
          run += c[x];
        }
      }
      __syncthreads();
      if (pass == 0) {
        // protected keys all fall into the top bin; count the candidates
        const uint32_t n_cand = static_cast<uint32_t>(M) - sm.hist[255];
        if (n_cand < static_cast<uint32_t>(S)) {
          if (tid == 0) atomicOr(a.err, 2);
          return;
        }
      }
      prefix |= sm.bcast[0] << shift;
      mask |= 255u << shift;
      kth = sm.bcast[1];
      __syncthreads();
    }
    T = prefix;
    take_eq = kth;
  }

  // Sweep in slot order: evicted slots get ranks 0..S-1.
  uint32_t eq_base = 0, sel_base = 0;
  for (int base = 0; base < M; base += kUpdThreads) {
    const int j = base + tid;
    float acc = 0.f;
    const uint32_t key = j < M ? slot_key(a, b, h, j, thr, &acc) : kProtected;
    const bool lt = key < T;
    const bool eq = j < M && key == T;
    uint32_t eq_tot;
    const uint32_t eq_rank = eq_base + block_scan_bit(eq, sm.warp_tot, &eq_tot);
    // (c < S always holds by construction; the guard keeps every access in bounds)
    const bool sel0 = lt || (eq && eq_rank < take_eq);
    uint32_t sel_tot;
    const uint32_t c = sel_base + block_scan_bit(sel0, sm.warp_tot2, &sel_tot);
    const bool sel = sel0 && c < static_cast<uint32_t>(S);
    if (j < M) {
      for (int bi = 0; bi < nb; ++bi) {
        const int bb = b + bi;
        const size_t g = static_cast<size_t>(bb) * a.Hkv + h;
        const float* inc = a.score_inc + static_cast<size_t>(bb * a.Hq + h * a.qg) * (M + S);
        if (sel) {
          // the new token's own column
          a.scores[g * M + j] = inc_group(a, inc + M, M + S, static_cast<int>(c));
          a.slot_pos[g * M + j] = a.pos0 + static_cast<int>(c);
          if (a.evict_idx) a.evict_idx[g * S + c] = j;
        } else {
          a.scores[g * M + j] = bi == 0 ? acc : slot_acc(a, bb, h, j);
        }
      }
    }
    // warp-cooperative K/V copies of this warp's evicted slots
    uint32_t m = __ballot_sync(0xffffffffu, sel);
    while (m) {
      const int src_lane = __ffs(m) - 1;
      m &= m - 1;
      const int cc = __shfl_sync(0xffffffffu, static_cast<int>(c), src_lane);
      const int jj = __shfl_sync(0xffffffffu, j, src_lane);
      for (int bi = 0; bi < nb; ++bi) copy_row(a, (b + bi) * a.Hkv + h, cc, jj, lane);
    }
    eq_base += eq_tot;
    sel_base += sel_tot;
  }
}

// ----------------------------------------------------- cluster variant --
constexpr int kCThreads = 512;
constexpr int kCWarps = kCThreads / 32;
// dynamic shared memory of the cluster variant: keys and scores of the M
// slots, scores and evicted slots of the S new tokens (M < 25600 < 65536,
// which the packed 16-bit counts of phase 3 need)
constexpr size_t kMaxClusterSmem = 200 * 1024;

// Keys a thread keeps in registers during the selection (M <= 16 * 512).
constexpr int kRegKeys = 16;

// Exclusive prefix sum over the block of one value per thread.
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t* warp_tot,
                                                    uint32_t* total) {
  const int tid = threadIdx.x, w = tid >> 5, l = tid & 31;
  uint32_t incl = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
    if (l >= o) incl += y;
  }
  if (l == 31) warp_tot[w] = incl;
  __syncthreads();
  if (w == 0) {
    uint32_t x = l < kCWarps ? warp_tot[l] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
      if (l >= o) x += y;
    }
    if (l < kCWarps) warp_tot[l] = x;
  }
  __syncthreads();
  const uint32_t base = w > 0 ? warp_tot[w - 1] : 0u;
  *total = warp_tot[kCWarps - 1];
  __syncthreads();
  return base + incl - v;
}


__global__ void __launch_bounds__(kCThreads, 1) update_cluster_kernel(const UpdateArgs a, int C,
                                                                      int prefetch) {
  extern __shared__ __align__(16) uint32_t dyn[];
  __shared__ __align__(16) uint32_t hist[3][256];
  __shared__ uint64_t rows_bar;
  __shared__ int abort_flag;
  __shared__ uint32_t warp_tot[kCWarps];
  __shared__ uint32_t bcast[4];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rank = static_cast<int>(cluster_rank());
  // one (b, h) per cluster; h2o_orig: one KV head per cluster, for every b
  const bool orig = a.policy == H2O_POLICY_ORIG;
  const int gidx = static_cast<int>(blockIdx.x) / C;
  const int b0 = orig ? 0 : gidx / a.Hkv, h = orig ? gidx : gidx % a.Hkv;
  const int nb = orig ? a.B : 1;  // batch entries whose state this cluster writes
  const int M = a.M, S = a.S, NK = M + S, qg = a.qg;
  const int thr = a.pos0 + S - a.W;
  uint32_t* keys = dyn;                                          // [M]
  float* accs = reinterpret_cast<float*>(dyn + M);               // [M] scores of (b0, h)
  float* nscore = reinterpret_cast<float*>(dyn + 2 * M);         // [S] score of new token c
  int* elist = reinterpret_cast<int*>(dyn + 2 * M + S);          // [S] evicted slot of rank c
  // prefetch: this CTA copies the ranks [c_lo, c_lo + n_rows); their K rows
  // then V rows are bulk-loaded here at the start and stored in phase 5
  const int c_per = (S + C - 1) / C;
  const int c_lo = min(S, rank * c_per), n_rows = min(S, c_lo + c_per) - c_lo;
  uint16_t* rowbuf = reinterpret_cast<uint16_t*>(
      reinterpret_cast<uint8_t*>(dyn) + ((2 * static_cast<size_t>(M) + 2 * S) * 4 + 15) / 16 * 16);
  if (tid == 0) {
    abort_flag = 0;
    if (prefetch && n_rows > 0) {
      bar_init(&rows_bar, 1);
      fence_bar_init();
      const uint32_t bytes = static_cast<uint32_t>(n_rows) * a.d * 2u;
      bar_expect_tx(&rows_bar, 2 * bytes);
      const size_t src = ((static_cast<size_t>(b0) * a.Hkv + h) * S + c_lo) * a.d;
      bulk_load_once(rowbuf, a.k_new + src, bytes, &rows_bar);
      bulk_load_once(rowbuf + static_cast<size_t>(c_per) * a.d, a.v_new + src, bytes, &rows_bar);
    }
  }
  // histograms of passes 0 and 1 (the cluster barrier below orders the clears
  // before any count)
  for (int x = tid; x < 2 * 256; x += kCThreads) hist[x >> 8][x & 255] = 0u;
  auto scores_of = [&](int b) { return a.scores + (static_cast<size_t>(b) * a.Hkv + h) * M; };
  auto pos_of = [&](int b) { return a.slot_pos + (static_cast<size_t>(b) * a.Hkv + h) * M; };
  auto inc_of = [&](int b) { return a.score_inc + static_cast<size_t>(b * a.Hq + h * qg) * NK; };

  // Thread t owns slots [t R, t R + R) in slot order.
  const int R = (M + kCThreads - 1) / kCThreads;
  const int j0 = min(M, tid * R), j1 = min(M, j0 + R);
  // 16-byte loads need every row start (b, h rows of M and NK) and j0 aligned
  const bool vec = R % 4 == 0 && M % 4 == 0 && NK % 4 == 0;

  // Phase 1: scores and selection keys of every slot (positions of b0).
  // CTA r of the cluster computes the slots of its share [r share, (r + 1)
  // share) and stores each key into every CTA's key array, so that every CTA
  // ends up with all M keys while each loads only its share of the old
  // state; the accumulated scores stay with the share's CTA, which also
  // writes the share's new state in phase 4.  acc_j = scores_j + (inc_0j +
  // inc_1j + ...) in fp32, heads in order (Eq. 3); h2o_orig adds the batch
  // entries' accumulated scores in ascending b.  (share is a multiple of R,
  // so each thread's run of slots lies in one share.)
  const int share = ((M + C - 1) / C + R - 1) / R * R;
  const int lo = min(M, rank * share), hi = min(M, lo + share);
  // Launched as a programmatic dependent of the attention kernels before it
  // on the stream, this kernel can start while they finish: what it reads
  // besides score_inc (scores, positions, the chunk's rows above) they do not
  // write, so it is pulled toward L2 first; then wait for them (score_inc,
  // and the cache rows they read, which phase 5 overwrites).
  for (int bi = 0; bi < nb; ++bi)
    for (int x = lo + tid * 32; x < hi; x += kCThreads * 32) {
      prefetch_l2(scores_of(b0 + bi) + x);
      prefetch_l2(pos_of(b0 + bi) + x);
    }
  grid_dependency_wait();
  {
    const int* sp = pos_of(b0);
    uint32_t key_dst[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) key_dst[r] = r < C ? cluster_addr(keys, r) : 0u;
    for (int j = lo + tid; j < hi; j += kCThreads) {
      const int pos = sp[j];
      float tot = 0.f;
      for (int bi = 0; bi < nb; ++bi) {
        const float acc = __fadd_rn(scores_of(b0 + bi)[j], inc_group(a, inc_of(b0 + bi), NK, j));
        tot = bi == 0 ? acc : __fadd_rn(tot, acc);
      }
      const uint32_t key = make_key(tot, pos, thr, a.policy, t_choice(a));
      const uint32_t off = static_cast<uint32_t>(j) * 4u;
#pragma unroll
      for (int r = 0; r < 8; ++r)
        if (r < C) st_cluster_u32(key_dst[r] + off, key);
      if (!orig) accs[j] = tot;
    }
    // scores of the new tokens (their own columns M + c, summed over the
    // group), 1/C of them here, into every CTA
    if (!orig) {
      const int cs = (S + C - 1) / C;
      uint32_t ns_dst[8];
#pragma unroll
      for (int r = 0; r < 8; ++r) ns_dst[r] = r < C ? cluster_addr(nscore, r) : 0u;
      for (int c = rank * cs + tid; c < min(S, rank * cs + cs); c += kCThreads) {
        const uint32_t v = __float_as_uint(inc_group(a, inc_of(b0) + M, NK, c));
#pragma unroll
        for (int r = 0; r < 8; ++r)
          if (r < C) st_cluster_u32(ns_dst[r] + static_cast<uint32_t>(c) * 4u, v);
      }
    }
  }
  // Every CTA of the cluster has read the old state before CTA 0 rewrites it,
  // and every CTA's keys (and CTA 0's scores) are in place.
  cluster_sync_all();

  // This thread's keys, slots j0 .. j1 - 1, are held in registers for the
  // selection passes (16-byte loads: a run of R slots read one key at a time
  // would hit the same shared-memory banks from every lane); long runs
  // (M > 8192) are read from shared memory.
  const int nR = j1 - j0;
  const bool in_regs = R <= kRegKeys;
  uint32_t kr[kRegKeys];
#pragma unroll
  for (int k = 0; k < kRegKeys; ++k) kr[k] = 0u;
  if (in_regs) {
    if (R % 4 == 0) {
#pragma unroll
      for (int q = 0; q < kRegKeys / 4; ++q)
        if (4 * q < nR) {
          const uint4 v = *reinterpret_cast<const uint4*>(keys + j0 + 4 * q);
          kr[4 * q] = v.x; kr[4 * q + 1] = v.y; kr[4 * q + 2] = v.z; kr[4 * q + 3] = v.w;
        }
    } else {
#pragma unroll
      for (int k = 0; k < kRegKeys; ++k)
        if (k < nR) kr[k] = keys[j0 + k];
    }
  }
  // body(key, j) for this thread's slots in slot order
  auto for_keys = [&](auto&& body) {
    if (in_regs) {
#pragma unroll
      for (int k = 0; k < kRegKeys; ++k)
        if (k < nR) body(kr[k], j0 + k);
    } else {
      for (int j = j0; j < j1; ++j) body(keys[j], j);
    }
  };

  // Phase 2: radix select of the S-th smallest key T, and how many keys equal
  // to T are taken (the lowest slots first).  One barrier per pass: every
  // warp scans the pass's histogram itself, and the histograms rotate over
  // three buffers: pass p counts into buffer p % 3 and clears buffer
  // (p + 1) % 3, which the warps last read in pass p - 2, before barrier
  // p - 1 that every warp has passed.
  uint32_t prefix = 0, mask = 0, kth = static_cast<uint32_t>(S);
  for (int pass = 0; pass < 4; ++pass) {
    const int shift = 24 - 8 * pass;
    uint32_t* hp = hist[pass % 3];
    // neighbouring slots mostly share a digit (the high digits of similar
    // scores): a thread adds runs of equal digits with one atomic each
    {
      uint32_t run_bin = 256u, run = 0u;
      for_keys([&](uint32_t key, int) {
        if ((key & mask) != prefix) return;
        const uint32_t bin = (key >> shift) & 255u;
        if (bin != run_bin) {
          if (run) atomicAdd(&hp[run_bin], run);
          run_bin = bin;
          run = 0u;
        }
        ++run;
      });
      if (run) atomicAdd(&hp[run_bin], run);
    }
    if (pass > 0)
      for (int x = tid; x < 256; x += kCThreads) hist[(pass + 1) % 3][x] = 0u;
    __syncthreads();
    if (pass == 0 && static_cast<uint32_t>(M) - hp[255] < static_cast<uint32_t>(S)) {
      if (tid == 0 && rank == 0) atomicOr(a.err, 2);
      // uniform over the cluster: every CTA computed the same histogram; the
      // rows loaded for the copies land before the CTA's shared memory goes
      if (prefetch && n_rows > 0) {
        volatile int never = 0;
        wait_bar(&rows_bar, 0, &never, kWaitLimitNs);
      }
      return;
    }
    // the bin holding the kth key: lane l sums bins 8l .. 8l + 7, a warp
    // scan of the sums, and the lane whose range holds kth finds the bin
    uint32_t c[8], sum = 0;
    const uint4 v0 = reinterpret_cast<const uint4*>(hp)[2 * lane];
    const uint4 v1 = reinterpret_cast<const uint4*>(hp)[2 * lane + 1];
    c[0] = v0.x; c[1] = v0.y; c[2] = v0.z; c[3] = v0.w;
    c[4] = v1.x; c[5] = v1.y; c[6] = v1.z; c[7] = v1.w;
#pragma unroll
    for (int x = 0; x < 8; ++x) sum += c[x];
    uint32_t incl = sum;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, incl, o);
      if (lane >= o) incl += y;
    }
    uint32_t run = incl - sum, bin = 0u, rem = 0u;
    const bool here = run < kth && kth <= incl;
#pragma unroll
    for (int x = 0; x < 8; ++x) {
      if (run < kth && kth <= run + c[x]) {
        bin = static_cast<uint32_t>(8 * lane + x);
        rem = kth - run;
      }
      run += c[x];
    }
    const int src = __ffs(__ballot_sync(0xffffffffu, here)) - 1;
    bin = __shfl_sync(0xffffffffu, bin, src);
    rem = __shfl_sync(0xffffffffu, rem, src);
    prefix |= bin << shift;
    mask |= 255u << shift;
    kth = rem;
  }
  const uint32_t T = prefix, take_eq = kth;

  // Phase 3: one scan of (keys < T, keys == T) per thread, packed in 16-bit
  // halves (M < 65536), gives each slot's eviction rank: the slots below T
  // before it plus the taken slots equal to T before it.
  uint32_t n_lt = 0, n_eq = 0;
  for_keys([&](uint32_t key, int) {
    n_lt += key < T;
    n_eq += key == T;
  });
  uint32_t tot;
  const uint32_t before = block_excl_scan(n_lt | (n_eq << 16), warp_tot, &tot);

  // Phase 4: evicted slots get ranks 0..S-1 (every CTA needs all of them for
  // its share of the row copies); the CTA whose share holds a thread's slots
  // writes their new state for every batch entry the cluster owns.
  {
    const bool mine = j0 >= lo && j0 < hi;
    uint32_t lt_b = before & 0xFFFFu, eq_b = before >> 16;
    for_keys([&](uint32_t key, int j) {
      const bool eq = key == T;
      const bool sel0 = key < T || (eq && eq_b < take_eq);
      const uint32_t c = lt_b + min(eq_b, take_eq);
      const bool sel = sel0 && c < static_cast<uint32_t>(S);
      lt_b += key < T;
      eq_b += eq;
      if (sel) elist[c] = j;
      if (mine) {
        for (int bi = 0; bi < nb; ++bi) {
          const int b = b0 + bi;
          const size_t g = static_cast<size_t>(b) * a.Hkv + h;
          if (sel) {
            pos_of(b)[j] = a.pos0 + static_cast<int>(c);
            if (a.evict_idx) a.evict_idx[g * S + c] = j;
          }
          if (orig) {
            scores_of(b)[j] = sel ? inc_group(a, inc_of(b) + M, NK, static_cast<int>(c))
                                  : slot_acc(a, b, h, j);
          } else if (sel) {
            accs[j] = nscore[c];
          }
        }
      }
    });
    if (mine && !orig) {
      float* sc = scores_of(b0);
      if (vec) {
        for (int j = j0; j < j1; j += 4)
          *reinterpret_cast<float4*>(sc + j) = *reinterpret_cast<const float4*>(accs + j);
      } else {
        for (int j = j0; j < j1; ++j) sc[j] = accs[j];
      }
    }
  }
  __syncthreads();

  const int n_sel = min(static_cast<int>((tot & 0xFFFFu) + min(tot >> 16, take_eq)), S);
  if (prefetch) {
    // Phase 5 (rows in shared memory): the ranks [c_lo, c_lo + n_rows) of
    // batch entry b0, 16-byte pieces from the rows loaded at the start
    if (n_rows <= 0) return;
    const bool landed = wait_bar(&rows_bar, 0, &abort_flag, kWaitLimitNs);
    if (!landed) {
      // the copies may still be in flight: give them time before the CTA's
      // shared memory goes away, and report
      const uint64_t t0 = global_timer_ns();
      while (global_timer_ns() - t0 < 1000000ull) {
      }
      if (tid == 0) atomicOr(a.err, H2O_DEVERR_TIMEOUT);
      return;
    }
    const int vecs = a.d / 8;  // 16-byte pieces per row
    const int n_cp = min(n_rows, n_sel - c_lo);
    const int pieces = n_cp * 2 * vecs;
    const size_t g = static_cast<size_t>(b0) * a.Hkv + h;
    for (int x = tid; x < pieces; x += kCThreads) {
      const int piece = x % vecs;
      const int rv = x / vecs;  // row * 2 + (0 = K, 1 = V)
      const int r = rv >> 1;
      const bool is_v = rv & 1;
      const uint4 v = reinterpret_cast<const uint4*>(
          rowbuf + (static_cast<size_t>(is_v ? c_per : 0) + r) * a.d)[piece];
      uint16_t* d = (is_v ? a.v_cache : a.k_cache) + (g * M + elist[c_lo + r]) * a.d;
      reinterpret_cast<uint4*>(d)[piece] = v;
    }
    return;
  }
  // Phase 5: this CTA's share of the K/V row copies (ranks c = rank mod C) of
  // every batch entry the cluster owns, 16-byte pieces, four loads in flight
  // per thread before their stores.
  const int rows = a.k_cache != nullptr && n_sel > rank ? (n_sel - 1 - rank) / C + 1 : 0;
  const int vecs = a.d / 8;  // 16-byte pieces per row
  const int per_b = rows * 2 * vecs;
  const int pieces = nb * per_b;
  for (int x0 = tid; x0 < pieces; x0 += 4 * kCThreads) {
    uint4 v[4];
    uint4* dst[4];
#pragma unroll
    for (int u = 0; u < 4; ++u) {
      const int x = x0 + u * kCThreads;
      dst[u] = nullptr;
      if (x < pieces) {
        const int b = b0 + x / per_b;
        const int xr = x % per_b;
        const int piece = xr % vecs;
        const int rv = xr / vecs;          // row index * 2 + (0 = K, 1 = V)
        const int cc = rank + C * (rv >> 1);
        const bool is_v = rv & 1;
        const size_t g = static_cast<size_t>(b) * a.Hkv + h;
        const uint16_t* src = (is_v ? a.v_new : a.k_new) + (g * S + cc) * a.d;
        uint16_t* d = (is_v ? a.v_cache : a.k_cache) + (g * M + elist[cc]) * a.d;
        v[u] = __ldg(reinterpret_cast<const uint4*>(src) + piece);
        dst[u] = reinterpret_cast<uint4*>(d) + piece;
      }
    }
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (dst[u]) *dst[u] = v[u];
  }
}

// ------------------------------------------------------ S = 1 (decode) --
// The selection is an argmin over (key, slot), so nothing is kept per slot:
// a cluster of C CTAs per (b, kv head) (h2o_orig: per kv head, every b) splits
// the M slots into C contiguous ranges.  Pass 1: each thread computes acc_j
// and the key of its slots with all loads of a batch in flight (the score_inc
// rows, M + 1 long, are not 16-byte aligned, so loads are 4-byte and
// coalesced) and keeps the smallest (key << 32 | j).  Every CTA sends its
// minimum to every CTA of the cluster; after a cluster barrier all know the
// evicted slot.  Pass 2 (nothing is written before it, so a (b, h) without a
// candidate stays unchanged): each CTA writes acc_j of its range (kept in
// shared memory by pass 1 when the range fits, recomputed otherwise), and
// the CTA holding the evicted slot writes the new token's score, position,
// evict_idx and K/V rows there.
constexpr int kDThreads = 512;
constexpr int kDBatch = 6;  // slots per thread per batch of loads

// acc_j of pass 1 kept for pass 2 when a CTA's range (x batch entries) fits
constexpr size_t kDStashBytes = 96 * 1024;

__global__ void __launch_bounds__(kDThreads, 2)
    update_decode_kernel(const UpdateArgs a, int C, int stash_ok) {
  grid_dependency_wait();  // score_inc of the attention kernels before it
  extern __shared__ float stash[];  // [nb][per] when stash_ok
  __shared__ unsigned long long wmin[kDThreads / 32];
  __shared__ unsigned long long cmin[8];
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int rank = static_cast<int>(cluster_rank());
  const bool orig = a.policy == H2O_POLICY_ORIG;
  const int gidx = static_cast<int>(blockIdx.x) / C;
  const int b0 = orig ? 0 : gidx / a.Hkv, h = orig ? gidx : gidx % a.Hkv;
  const int nb = orig ? a.B : 1;
  const int M = a.M, NK = M + 1, qg = a.qg;
  const int thr = a.pos0 + 1 - a.W;
  const int t_now = t_choice(a);
  const int qg_inc = a.insert ? 0 : qg;  // score_inc rows read per slot
  const int per = (M + C - 1) / C;
  const int jlo = min(M, rank * per), jhi = min(M, jlo + per);
  const int32_t* pos_b0 = a.slot_pos + (static_cast<size_t>(b0) * a.Hkv + h) * M;

  // acc_j (Eq. 3) of batch entry b for the slots base + u * kDThreads, heads
  // of the group added in ascending order, no fused multiply-add
  auto batch_acc = [&](int b, int base, float (&acc)[kDBatch]) {
    const float* sc = a.scores + (static_cast<size_t>(b) * a.Hkv + h) * M;
    const float* inc = a.score_inc + static_cast<size_t>(b * a.Hq + h * qg) * NK;
    float t[kDBatch], old[kDBatch];
#pragma unroll
    for (int u = 0; u < kDBatch; ++u) {
      const int j = base + u * kDThreads;
      old[u] = j < jhi ? sc[j] : 0.f;
      t[u] = j < jhi && qg_inc > 0 ? __ldg(inc + j) : 0.f;
    }
    for (int g = 1; g < qg_inc; ++g) {
      float x[kDBatch];
#pragma unroll
      for (int u = 0; u < kDBatch; ++u) {
        const int j = base + u * kDThreads;
        x[u] = j < jhi ? __ldg(inc + static_cast<size_t>(g) * NK + j) : 0.f;
      }
#pragma unroll
      for (int u = 0; u < kDBatch; ++u) t[u] = __fadd_rn(t[u], x[u]);
    }
#pragma unroll
    for (int u = 0; u < kDBatch; ++u) acc[u] = __fadd_rn(old[u], t[u]);
  };

  // ---- pass 1: the smallest (key, slot) of this CTA's range
  unsigned long long best = ~0ull;
  for (int base = jlo + tid; base < jhi; base += kDThreads * kDBatch) {
    int pos[kDBatch];
    float kacc[kDBatch];
#pragma unroll
    for (int u = 0; u < kDBatch; ++u) {
      const int j = base + u * kDThreads;
      pos[u] = j < jhi ? pos_b0[j] : 0;
    }
    for (int bi = 0; bi < nb; ++bi) {
      float acc[kDBatch];
      batch_acc(b0 + bi, base, acc);
#pragma unroll
      for (int u = 0; u < kDBatch; ++u) {
        kacc[u] = bi == 0 ? acc[u] : __fadd_rn(kacc[u], acc[u]);
        const int j = base + u * kDThreads;
        if (stash_ok && j < jhi) stash[bi * per + (j - jlo)] = acc[u];
      }
    }
#pragma unroll
    for (int u = 0; u < kDBatch; ++u) {
      const int j = base + u * kDThreads;
      if (j < jhi) {
        const uint32_t key = make_key(kacc[u], pos[u], thr, a.policy, t_now);
        const unsigned long long k64 =
            (static_cast<unsigned long long>(key) << 32) | static_cast<uint32_t>(j);
        best = k64 < best ? k64 : best;
      }
    }
  }
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
    best = other < best ? other : best;
  }
  if (lane == 0) wmin[warp] = best;
  __syncthreads();
  if (warp == 0) {
    best = lane < kDThreads / 32 ? wmin[lane] : ~0ull;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
      best = other < best ? other : best;
    }
    // this CTA's minimum into slot `rank` of every CTA of the cluster
    if (lane < C) {
      const uint32_t dst = cluster_addr(&cmin[rank], static_cast<uint32_t>(lane));
      asm volatile("st.shared::cluster.u64 [%0], %1;" ::"r"(dst), "l"(best) : "memory");
    }
  }
  cluster_sync_all();
  best = ~0ull;
  for (int r = 0; r < C; ++r) best = cmin[r] < best ? cmin[r] : best;
  if (static_cast<uint32_t>(best >> 32) == kProtected) {  // every slot inside the window
    if (rank == 0 && tid == 0) atomicOr(a.err, 2);
    return;
  }
  const int e = static_cast<int>(best & 0xFFFFFFFFu);

  // ---- pass 2: write acc_j of this range; the evicted slot takes the new token
  for (int base = jlo + tid; base < jhi; base += kDThreads * kDBatch) {
    for (int bi = 0; bi < nb; ++bi) {
      float acc[kDBatch];
      if (stash_ok) {
#pragma unroll
        for (int u = 0; u < kDBatch; ++u) {
          const int j = base + u * kDThreads;
          acc[u] = j < jhi ? stash[bi * per + (j - jlo)] : 0.f;
        }
      } else {
        batch_acc(b0 + bi, base, acc);
      }
      float* sc = a.scores + (static_cast<size_t>(b0 + bi) * a.Hkv + h) * M;
#pragma unroll
      for (int u = 0; u < kDBatch; ++u) {
        const int j = base + u * kDThreads;
        if (j < jhi && j != e) sc[j] = acc[u];
      }
    }
  }
  if (e < jlo || e >= jhi) return;
  for (int bi = warp; bi < nb; bi += kDThreads / 32) {
    const int b = b0 + bi;
    const int grp = b * a.Hkv + h;
    if (lane == 0) {
      const float* inc = a.score_inc + static_cast<size_t>(b * a.Hq + h * qg) * NK;
      a.scores[static_cast<size_t>(grp) * M + e] = inc_group(a, inc, NK, M);
      a.slot_pos[static_cast<size_t>(grp) * M + e] = a.pos0;
      if (a.evict_idx) a.evict_idx[grp] = e;
    }
    copy_row(a, grp, 0, e, lane);
  }
}

// Last part of the paper-order chunk step (Eq. 3): scores += the group sum of
// score_inc, in the same float32 order as the update kernels (one thread per
// slot; the kernel moves 4 (1 + q_g) bytes per slot and is bandwidth bound).
__global__ void __launch_bounds__(256) scores_add_kernel(const ScoresAddArgs a) {
  const size_t n = static_cast<size_t>(a.B) * a.Hkv * a.M;
  const size_t stride = static_cast<size_t>(gridDim.x) * blockDim.x;
  for (size_t x = blockIdx.x * static_cast<size_t>(blockDim.x) + threadIdx.x; x < n; x += stride) {
    const size_t grp = x / a.M;
    const int j = static_cast<int>(x % a.M);
    const size_t b = grp / a.Hkv, h = grp % a.Hkv;
    const float* inc = a.score_inc + (b * (a.Hkv * a.qg) + h * a.qg) * a.M;
    a.scores[x] = __fadd_rn(a.scores[x], group_sum(inc, a.M, a.qg, j));
  }
}

}  // namespace

cudaError_t launch_scores_add(const ScoresAddArgs& a, cudaStream_t stream) {
  const size_t n = static_cast<size_t>(a.B) * a.Hkv * a.M;
  const size_t blocks = std::min<size_t>((n + 255) / 256, 152 * 8);
  scores_add_kernel<<<static_cast<unsigned>(blocks), 256, 0, stream>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_update(const UpdateArgs& a, cudaStream_t stream) {
  const size_t smem = (2 * static_cast<size_t>(a.M) + 2 * static_cast<size_t>(a.S)) * sizeof(uint32_t);
  const bool smem_path = a.S > 1 && smem <= kMaxClusterSmem;
  if (a.S == 1) {
    int C = a.M / 8192;
    C = C < 1 ? 1 : (C > 8 ? 8 : C);
    const int groups = a.policy == H2O_POLICY_ORIG ? a.Hkv : a.B * a.Hkv;
    const size_t per = (static_cast<size_t>(a.M) + C - 1) / C;
    const size_t stash = per * (a.policy == H2O_POLICY_ORIG ? a.B : 1) * sizeof(float);
    const int stash_ok = stash <= kDStashBytes ? 1 : 0;
    static OncePerDevice dconf;
    cudaError_t e = dconf.run([](int) {
      return cudaFuncSetAttribute(update_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                  static_cast<int>(kDStashBytes));
    });
    if (e != cudaSuccess) return e;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(groups * C));
    cfg.blockDim = dim3(kDThreads);
    cfg.dynamicSmemBytes = stash_ok ? stash : 0;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = static_cast<unsigned>(C);
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, update_decode_kernel, a, C, stash_ok);
  }
  if (!smem_path) {
    const int groups = a.policy == H2O_POLICY_ORIG ? a.Hkv : a.B * a.Hkv;
    update_kernel<<<groups, kUpdThreads, 0, stream>>>(a);
    return cudaGetLastError();
  }
  static OncePerDevice configured;
  cudaError_t e = configured.run([](int) {
    return cudaFuncSetAttribute(update_cluster_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(kMaxClusterSmem));
  });
  if (e != cudaSuccess) return e;
  int C = (a.S + 63) / 64;
  C = C < 1 ? 1 : (C > 8 ? 8 : C);
  // the chunk rows a CTA writes are loaded into shared memory at its start
  // when they fit (one batch entry per cluster, rows to copy)
  const size_t rows_off = (smem + 15) / 16 * 16;
  const size_t rows_bytes = 2 * static_cast<size_t>((a.S + C - 1) / C) * a.d * sizeof(uint16_t);
  const int prefetch = a.k_cache != nullptr && a.policy != H2O_POLICY_ORIG &&
                       rows_off + rows_bytes <= kMaxClusterSmem;
  cudaLaunchConfig_t cfg = {};
  const int groups = a.policy == H2O_POLICY_ORIG ? a.Hkv : a.B * a.Hkv;
  cfg.gridDim = dim3(static_cast<unsigned>(groups * C));
  cfg.blockDim = dim3(kCThreads);
  cfg.dynamicSmemBytes = prefetch ? rows_off + rows_bytes : smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = static_cast<unsigned>(C);
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 2;
  return cudaLaunchKernelEx(&cfg, update_cluster_kernel, a, C, prefetch);
}

}  // namespace h2o
