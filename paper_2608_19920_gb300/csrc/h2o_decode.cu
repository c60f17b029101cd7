// Sparse SDPA with summed attention weights for one query token per sequence
// (S = 1, the decode regime of §3.3 with chunk size 1).
//
// What it computes is the S = 1 case of the chunk kernel: the token at
// position pos0 attends to the M cache slots it may see (0 <= slot_pos <=
// pos0, §3.1 Eq. 2 with the mask of §3.3.1) and to itself (chunk column M);
// score_inc[b, hq, j] = m_j = exp(a_j - lambda) (§3.3.1 / §A.6.1, one query row,
// so the column sum is the weight itself) and out = sum_j m_j v_j.
//
// The work is one dot product per (key, query head) and one weighted row sum,
// with every K and V row read once: HBM bound, so no tensor cores.  Per (b, kv
// head) the M slots are cut into splits of split_len slots (the last split also
// takes the new token), one CTA each:
//
//  * decode_split_kernel: a single thread streams the split's K rows, then its V
//    rows, in 16 KB bulk copies through a 4-stage shared-memory ring (mbarrier
//    completion, L2 evict-first).  All q_g query heads of the group share each
//    K/V row.  Q K^T: eight lanes per key, each holding 16 (d = 128) or 8
//    (d = 64) elements of every head's q in registers; a reduce-scatter over the
//    eight lanes leaves one head's logit per lane.  The logits (log2 units,
//    masked = -inf) go to score_inc and to shared memory; then p = exp2(a - m)
//    with the split's own max m, the split sum l, and P V with one warp per key
//    and lanes over d.  The partial (m, l, o) of every query head goes to the
//    workspace (the §A.6.1 merge of partial logsumexps, as in split-K decoding).
//  * decode_combine_kernel: per (b, hq) merges the splits' partials into lambda
//    and out (§A.6.1), then rewrites that row of score_inc as exp2(a - lambda).
//
// Bytes per step: K and V once (the algorithmic 2 B d per slot each), plus
// the score_inc row written as logits, read and written again as weights.
#include <algorithm>
#include <cstdint>

#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kDecThreads = 256;
constexpr int kDecWarps = kDecThreads / 32;
constexpr int kDecStages = 4;
constexpr int kDecTileBytes = 16384;
constexpr int kCombineThreads = 256;
constexpr int kCombineCols = 4096;  // score_inc columns normalised per combine CTA

template <int D, bool Q8 = false>
struct DecGeom {
  static constexpr int kRowBytes = Q8 ? D : D * 2;             // a cache row in the ring
  static constexpr int kTileKeys = kDecTileBytes / kRowBytes;  // bf16: 64 (d = 128) or 128;
                                                               // 8-bit: 128 or 256
  // A ring slot holds kTileKeys rows, or (8-bit) up to kTileKeys - 1 code rows
  // followed by the new token's bf16 row (2 D bytes) when that token ends the item.
  static constexpr int kSlotBytes = kDecTileBytes + (Q8 ? D : 0);
  static constexpr int kCh = D / 64;                           // 16-byte chunks per lane in Q K^T
  static constexpr int kVe = D / 32;                           // value elements per lane in P V
};

// Two 8-bit codes of a cache row, read back as the 8-bit format defines:
// bf16(code * scale), returned as fp32.  `wb` holds four codes with their sign
// bits flipped (code + 128 as unsigned bytes); byte i of it is placed under the
// exponent of 2^23, so the float is 2^23 + 128 + code exactly, and subtracting
// 2^23 + 128 leaves the code.  The product and its rounding are those of the
// read-back kernel (fp32 multiply, then round to nearest even bf16).
__device__ __forceinline__ float2 q8_pair(uint32_t wb, int i, float2 s2) {
  const float lo = __uint_as_float(__byte_perm(wb, 0x4B000000u, 0x7650u | i));
  const float hi = __uint_as_float(__byte_perm(wb, 0x4B000000u, 0x7650u | (i + 1)));
  const float2 c = __fadd2_rn(make_float2(lo, hi), make_float2(-8388736.f, -8388736.f));
  const float2 x = __fmul2_rn(c, s2);
  const uint32_t p = pack_bf16x2(x.x, x.y);
  return make_float2(__uint_as_float(p << 16), __uint_as_float(p & 0xFFFF0000u));
}

// Floats of the region that holds the warps' partial outputs at the end of an
// item and, with 8-bit buffers, the split's K and V scales before that.
template <int D, int QG, bool Q8>
__host__ __device__ constexpr int red_region_floats(int split_len) {
  const int o = kDecWarps * QG * D;
  const int sc = Q8 ? (2 * (split_len + 1) + 3) / 4 * 4 : 0;
  return o > sc ? o : sc;
}

struct alignas(16) DecHead {  // 16-byte size: the logits after it are read as float4
  uint64_t full[kDecStages];
  float red[kDecWarps][kDecodeMaxQg];   // per-warp maxima
  float red2[kDecWarps][kDecodeMaxQg];  // per-warp sums
  int abort;
};

__device__ __forceinline__ void bf16x8_to_f32(const uint4& u, float* f) {
  const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
  for (int x = 0; x < 4; ++x) {
    f[2 * x] = __uint_as_float(w[x] << 16);
    f[2 * x + 1] = __uint_as_float(w[x] & 0xFFFF0000u);
  }
}

// Sum over the eight lanes of a key group (lane bits 0-2) of QG values,
// scattered: afterwards lane bits (2, 1) [and 0 when QG = 8] name the head
// whose total the lane holds.  QG = 4 leaves the total in both lanes of a pair.
template <int QG>
__device__ __forceinline__ float reduce_scatter8(float (&v)[QG], uint32_t lane) {
  if constexpr (QG == 8) {
    float a[4];
    const bool h2 = (lane >> 2) & 1u;
#pragma unroll
    for (int x = 0; x < 4; ++x) {
      const float send = h2 ? v[x] : v[4 + x];
      const float keep = h2 ? v[4 + x] : v[x];
      a[x] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
    float c[2];
    const bool h1 = (lane >> 1) & 1u;
#pragma unroll
    for (int x = 0; x < 2; ++x) {
      const float send = h1 ? a[x] : a[2 + x];
      const float keep = h1 ? a[2 + x] : a[x];
      c[x] = keep + __shfl_xor_sync(0xffffffffu, send, 2);
    }
    const bool h0 = lane & 1u;
    const float send = h0 ? c[0] : c[1];
    const float keep = h0 ? c[1] : c[0];
    return keep + __shfl_xor_sync(0xffffffffu, send, 1);
  } else {
    static_assert(QG == 4, "QG is 4 or 8");
    float a[2];
    const bool h2 = (lane >> 2) & 1u;
#pragma unroll
    for (int x = 0; x < 2; ++x) {
      const float send = h2 ? v[x] : v[2 + x];
      const float keep = h2 ? v[2 + x] : v[x];
      a[x] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
    const bool h1 = (lane >> 1) & 1u;
    const float send = h1 ? a[0] : a[1];
    float c = (h1 ? a[1] : a[0]) + __shfl_xor_sync(0xffffffffu, send, 2);
    return c + __shfl_xor_sync(0xffffffffu, c, 1);
  }
}

template <int QG>
__device__ __forceinline__ int scatter_head(uint32_t lane) {
  return QG == 8 ? static_cast<int>(lane & 7u) : static_cast<int>((lane >> 1) & 3u);
}

// One (b, kv head, split) work item.
struct DecItem {
  int grp, s, j0, n_cache, n_loc, n_tiles;
  bool last;
};

template <int D, bool Q8>
__device__ __forceinline__ DecItem dec_item(const DecodeArgs& a, int it) {
  DecItem x;
  x.grp = it / a.n_split;
  x.s = it % a.n_split;
  x.j0 = x.s * a.split_len;
  x.n_cache = min(a.split_len, a.M - x.j0);  // >= 1: n_split = ceil(M / split_len)
  x.last = x.s == a.n_split - 1 && a.with_new;  // this item also takes the new token
  x.n_loc = x.n_cache + (x.last ? 1 : 0);        // local key n_cache is the new token
  x.n_tiles = (x.n_loc + DecGeom<D, Q8>::kTileKeys - 1) / DecGeom<D, Q8>::kTileKeys;
  return x;
}

// Keys per thread in the per-item passes over the split (256 threads).
constexpr int kKeysPerThread = (kDecodeMaxSplitLen + 1 + kDecThreads - 1) / kDecThreads;

// Reduces QG values per thread over the block: warp shuffles, then one row of
// `red` per warp; every thread then reads the 8 rows.
template <int QG, bool kMax>
__device__ __forceinline__ void block_reduce_qg(float (&v)[QG], float (*red)[kDecodeMaxQg],
                                                int warp, uint32_t lane) {
#pragma unroll
  for (int g = 0; g < QG; ++g)
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float y = __shfl_xor_sync(0xffffffffu, v[g], o);
      v[g] = kMax ? fmaxf(v[g], y) : v[g] + y;
    }
  if (lane == 0)
#pragma unroll
    for (int g = 0; g < QG; ++g) red[warp][g] = v[g];
}

template <int D, int QG, bool Q8>
__global__ void __launch_bounds__(kDecThreads, QG == 4 ? 2 : 1)
    decode_split_kernel(const DecodeArgs a) {
  using G = DecGeom<D, Q8>;
  extern __shared__ __align__(128) uint8_t dsm[];
  uint8_t* ring = dsm;
  static_assert(G::kSlotBytes % 16 == 0, "ring slots must stay 16-byte aligned");
  DecHead& hd = *reinterpret_cast<DecHead*>(dsm + kDecStages * G::kSlotBytes);
  static_assert(sizeof(DecHead) % 16 == 0, "logits must stay 16-byte aligned");
  float* lg = reinterpret_cast<float*>(dsm + kDecStages * G::kSlotBytes + sizeof(DecHead));
  float* red_o = lg + (a.split_len + 1) * QG;  // [warp][g][D]
  // 8-bit buffers: the item's K and V scales, in red_o's space until P V ends
  float* ksc = red_o;
  float* vsc = red_o + (a.split_len + 1);
  // q rows of the item whose first K tile sits in ring slot x: qbuf + x * QG * D
  uint16_t* qbuf = reinterpret_cast<uint16_t*>(red_o + red_region_floats<D, QG, Q8>(a.split_len));

  const int tid = threadIdx.x, warp = tid >> 5;
  const uint32_t lane = static_cast<uint32_t>(tid & 31);
  const int n_items = a.n_split * a.B * a.Hkv;
  if (tid == 0) launch_dependents();  // the combine may be placed (it waits for this grid)

  if (tid == 0) {
#pragma unroll
    for (int x = 0; x < kDecStages; ++x) bar_init(&hd.full[x], 1);
    hd.abort = 0;
    fence_bar_init();
  }
  __syncthreads();

  // Producer (thread 0): the CTA's items in order, each as its K tiles then
  // its V tiles, one tile per ring slot freed; the stream of tiles runs on
  // across items, so the ring never drains between them.
  int issued = 0;
  int p_it = blockIdx.x, p_t = 0;
  DecItem p_x;
  if (p_it < n_items) p_x = dec_item<D, Q8>(a, p_it);
  auto issue_next = [&]() {
    if (p_it >= n_items) return;
    const bool is_v = p_t >= p_x.n_tiles;
    const int k0 = (is_v ? p_t - p_x.n_tiles : p_t) * G::kTileKeys;
    const int k1 = min(k0 + G::kTileKeys, p_x.n_loc);
    const int rows_c = max(0, min(k1, p_x.n_cache) - k0);
    const bool has_new = p_x.last && k1 > p_x.n_cache;
    uint8_t* dst = ring + (issued % kDecStages) * G::kSlotBytes;
    uint64_t* bar = &hd.full[issued % kDecStages];
    const uint32_t q_bytes = p_t == 0 ? static_cast<uint32_t>(a.qg * D * 2) : 0u;
    // the new token's row is bf16 (2 D bytes) in both layouts
    bar_expect_tx(bar, static_cast<uint32_t>(rows_c * G::kRowBytes + (has_new ? 2 * D : 0)) +
                           q_bytes);
    if (q_bytes) {
      const int pb = p_x.grp / a.Hkv, ph = p_x.grp % a.Hkv;
      bulk_load_once(qbuf + (issued % kDecStages) * QG * D,
                     a.q + static_cast<size_t>(pb * a.Hq + ph * a.qg) * D, q_bytes, bar);
    }
    if (rows_c > 0) {
      const size_t row0 = static_cast<size_t>(p_x.grp) * a.M + p_x.j0 + k0;
      const void* base;
      if constexpr (Q8)
        base = (is_v ? a.v_codes : a.k_codes) + row0 * D;
      else
        base = (is_v ? a.v_cache : a.k_cache) + row0 * D;
      bulk_load_once(dst, base, static_cast<uint32_t>(rows_c * G::kRowBytes), bar);
    }
    if (has_new)
      bulk_load_once(dst + rows_c * G::kRowBytes,
                     (is_v ? a.v_new : a.k_new) + static_cast<size_t>(p_x.grp) * D, 2 * D, bar);
    ++issued;
    if (++p_t == 2 * p_x.n_tiles) {
      p_t = 0;
      p_it += gridDim.x;
      if (p_it < n_items) p_x = dec_item<D, Q8>(a, p_it);
    }
  };
  if (tid == 0)
    for (int x = 0; x < kDecStages; ++x) issue_next();

  volatile int* abort_flag = &hd.abort;
  const int c0 = static_cast<int>(lane & 7u);  // this lane's 16-byte chunks: c0 (+ 8)
  const int hg = scatter_head<QG>(lane);
  const bool dot_writer = (QG == 8 || (lane & 1u) == 0) && hg < a.qg;
  int g_t = 0;  // tiles consumed so far (ring slot and phase)

  for (int it = blockIdx.x; it < n_items; it += gridDim.x) {
    const DecItem x = dec_item<D, Q8>(a, it);
    const int b = x.grp / a.Hkv, h = x.grp % a.Hkv;
    const size_t row0 = static_cast<size_t>(b * a.Hq + h * a.qg);  // first query head's row

    // positions of the keys this thread masks below (in flight during Q K^T)
    const int32_t* sp = a.slot_pos + static_cast<size_t>(x.grp) * a.M + x.j0;
    int pos[kKeysPerThread];
#pragma unroll
    for (int u = 0; u < kKeysPerThread; ++u) {
      const int k = tid + u * kDecThreads;
      pos[u] = k < x.n_cache ? __ldg(sp + k) : 0;
    }
    if constexpr (Q8) {  // the item's row scales, read in Q K^T and P V
      const size_t sc0 = static_cast<size_t>(x.grp) * a.M + x.j0;
      for (int k = tid; k < x.n_cache; k += kDecThreads) {
        ksc[k] = __ldg(a.k_scales + sc0 + k);
        vsc[k] = __ldg(a.v_scales + sc0 + k);
      }
      __syncthreads();
    }
    // ---- Q K^T: raw dot products of the item's keys into lg
    float2 qr[QG][4 * G::kCh];  // this lane's slice of every head's query, element pairs
    for (int t = 0; t < x.n_tiles; ++t, ++g_t) {
      if (wait_bar(&hd.full[g_t % kDecStages], (g_t / kDecStages) & 1, abort_flag,
                   kWaitLimitNs)) {
        const uint8_t* tile = ring + (g_t % kDecStages) * G::kSlotBytes;
        if (t == 0) {  // the q rows arrived with this tile; read before its slot is reissued
          const uint16_t* qs = qbuf + (g_t % kDecStages) * QG * D;
#pragma unroll
          for (int g = 0; g < QG; ++g) {
#pragma unroll
            for (int ch = 0; ch < G::kCh; ++ch) {
              float f[8];
              // bf16 rows: chunks c0 and c0 + 8; 8-bit rows: the contiguous
              // chunks kCh c0 .. kCh c0 + kCh - 1 (the lane's code bytes)
              const int qc = Q8 ? G::kCh * c0 + ch : c0 + 8 * ch;
              if (g < a.qg) {
                bf16x8_to_f32(reinterpret_cast<const uint4*>(qs + g * D)[qc], f);
              } else {
#pragma unroll
                for (int e = 0; e < 8; ++e) f[e] = 0.f;
              }
#pragma unroll
              for (int e = 0; e < 4; ++e) qr[g][4 * ch + e] = make_float2(f[2 * e], f[2 * e + 1]);
            }
          }
        }
#pragma unroll 1
        for (int r = 0; r < G::kTileKeys / 32; ++r) {
          const int kk = r * 32 + warp * 4 + static_cast<int>(lane >> 3);  // key within the tile
          const int kl = t * G::kTileKeys + kk;                             // key within the item
          // packed fp32 FMAs over element pairs (even, odd), the two halves
          // added at the end
          float2 d2[QG];
#pragma unroll
          for (int g = 0; g < QG; ++g) d2[g] = make_float2(0.f, 0.f);
          // the new token's row is bf16 in both layouts (8-bit: it follows the
          // tile's code rows, at the offset its key index gives)
          const bool code_row = Q8 && !(x.last && kl == x.n_cache);
          if (kl < x.n_loc && code_row) {
            const uint8_t* crow = tile + kk * G::kRowBytes;
            const float sk = ksc[kl];
            const float2 s2 = make_float2(sk, sk);
            uint32_t w[2 * G::kCh];  // this lane's codes (elements kCh 8 c0 ..), sign-flipped
            if constexpr (D == 128) {
              const uint4 u = *reinterpret_cast<const uint4*>(crow + 16 * c0);
              w[0] = u.x; w[1] = u.y; w[2] = u.z; w[3] = u.w;
            } else {
              const uint2 u = *reinterpret_cast<const uint2*>(crow + 8 * c0);
              w[0] = u.x; w[1] = u.y;
            }
#pragma unroll
            for (int x2 = 0; x2 < 2 * G::kCh; ++x2) w[x2] ^= 0x80808080u;
#pragma unroll
            for (int ch = 0; ch < G::kCh; ++ch)
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 kf = q8_pair(w[2 * ch + (e >> 1)], 2 * (e & 1), s2);
#pragma unroll
                for (int g = 0; g < QG; ++g) d2[g] = __ffma2_rn(qr[g][4 * ch + e], kf, d2[g]);
              }
          } else if (kl < x.n_loc) {
            const uint4* krow = reinterpret_cast<const uint4*>(tile + kk * G::kRowBytes);
#pragma unroll
            for (int ch = 0; ch < G::kCh; ++ch) {
              const uint4 u = krow[Q8 ? G::kCh * c0 + ch : c0 + 8 * ch];
              const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
              for (int e = 0; e < 4; ++e) {
                const float2 kf = make_float2(__uint_as_float(w[e] << 16),
                                              __uint_as_float(w[e] & 0xFFFF0000u));
#pragma unroll
                for (int g = 0; g < QG; ++g) d2[g] = __ffma2_rn(qr[g][4 * ch + e], kf, d2[g]);
              }
            }
          }
          float dot[QG];
#pragma unroll
          for (int g = 0; g < QG; ++g) dot[g] = d2[g].x + d2[g].y;
          const float tot = reduce_scatter8<QG>(dot, lane);
          if (dot_writer && kl < x.n_loc) lg[kl * QG + hg] = tot;
        }
      }
      __syncthreads();  // every warp is done with the slot; lg rows complete
      if (*abort_flag) break;
      if (tid == 0) issue_next();
    }
    if (*abort_flag) break;

    // ---- mask, log2 scale, logits to score_inc (coalesced), split max
    float mx[QG];
#pragma unroll
    for (int g = 0; g < QG; ++g) mx[g] = -INFINITY;
#pragma unroll
    for (int u = 0; u < kKeysPerThread; ++u) {
      const int k = tid + u * kDecThreads;
      if (k < x.n_loc) {
        const bool vis = k < x.n_cache ? (pos[u] >= 0 && pos[u] <= a.pos0) : true;
        const size_t j = k < x.n_cache ? static_cast<size_t>(x.j0 + k) : static_cast<size_t>(a.M);
#pragma unroll
        for (int g4 = 0; g4 < QG; g4 += 4) {
          float4 v = *reinterpret_cast<const float4*>(lg + k * QG + g4);
          float w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            w[e] = vis ? w[e] * a.scale_log2 : -INFINITY;
            if (g4 + e < a.qg) {
              a.score_inc[(row0 + g4 + e) * static_cast<size_t>(a.nk) + j] = w[e];
              mx[g4 + e] = fmaxf(mx[g4 + e], w[e]);
            }
          }
          *reinterpret_cast<float4*>(lg + k * QG + g4) = make_float4(w[0], w[1], w[2], w[3]);
        }
      }
    }
    block_reduce_qg<QG, true>(mx, hd.red, warp, lane);
    __syncthreads();
    float m[QG];
#pragma unroll
    for (int g = 0; g < QG; ++g) {
      m[g] = hd.red[0][g];
#pragma unroll
      for (int w = 1; w < kDecWarps; ++w) m[g] = fmaxf(m[g], hd.red[w][g]);
    }
    // ---- p = exp2(a - m) in place, split sums
    float ls[QG];
#pragma unroll
    for (int g = 0; g < QG; ++g) ls[g] = 0.f;
#pragma unroll
    for (int u = 0; u < kKeysPerThread; ++u) {
      const int k = tid + u * kDecThreads;
      if (k < x.n_loc) {
#pragma unroll
        for (int g4 = 0; g4 < QG; g4 += 4) {
          float4 v = *reinterpret_cast<const float4*>(lg + k * QG + g4);
          float w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            const float mg = m[g4 + e];
            w[e] = mg > -INFINITY ? fast_exp2(w[e] - mg) : 0.f;
            ls[g4 + e] += w[e];
          }
          *reinterpret_cast<float4*>(lg + k * QG + g4) = make_float4(w[0], w[1], w[2], w[3]);
        }
      }
    }
    block_reduce_qg<QG, false>(ls, hd.red2, warp, lane);
    __syncthreads();  // p complete; hd.red2 holds the warps' sums

    // ---- P V: one warp per key, lanes over d
    float2 acc[QG][G::kVe / 2];  // (d element 2e, 2e + 1) of this lane, per head
#pragma unroll
    for (int g = 0; g < QG; ++g)
#pragma unroll
      for (int e = 0; e < G::kVe / 2; ++e) acc[g][e] = make_float2(0.f, 0.f);
    for (int t = 0; t < x.n_tiles; ++t, ++g_t) {
      if (wait_bar(&hd.full[g_t % kDecStages], (g_t / kDecStages) & 1, abort_flag,
                   kWaitLimitNs)) {
        const uint8_t* tile = ring + (g_t % kDecStages) * G::kSlotBytes;
        const int k0 = t * G::kTileKeys;
        const int kend = min(G::kTileKeys, x.n_loc - k0);
#pragma unroll 2
        for (int kk = warp; kk < kend; kk += kDecWarps) {
          float p[QG];
#pragma unroll
          for (int g4 = 0; g4 < QG; g4 += 4) {
            const float4 pv = *reinterpret_cast<const float4*>(lg + (k0 + kk) * QG + g4);
            p[g4] = pv.x;
            p[g4 + 1] = pv.y;
            p[g4 + 2] = pv.z;
            p[g4 + 3] = pv.w;
          }
          float2 vf[G::kVe / 2];
          if (Q8 && !(x.last && k0 + kk == x.n_cache)) {  // a code row (the warp's key)
            const float sv = vsc[k0 + kk];
            const float2 s2 = make_float2(sv, sv);
            if constexpr (D == 128) {
              const uint32_t wb =
                  *reinterpret_cast<const uint32_t*>(tile + kk * G::kRowBytes + lane * 4) ^
                  0x80808080u;
              vf[0] = q8_pair(wb, 0, s2);
              vf[G::kVe / 2 - 1] = q8_pair(wb, 2, s2);
            } else {
              const uint32_t wb =
                  static_cast<uint32_t>(
                      *reinterpret_cast<const uint16_t*>(tile + kk * G::kRowBytes + lane * 2)) ^
                  0x8080u;
              vf[0] = q8_pair(wb, 0, s2);
            }
          } else if constexpr (D == 128) {
            const uint2 uu = *reinterpret_cast<const uint2*>(tile + kk * G::kRowBytes + lane * 8);
            vf[0] = make_float2(__uint_as_float(uu.x << 16), __uint_as_float(uu.x & 0xFFFF0000u));
            vf[1] = make_float2(__uint_as_float(uu.y << 16), __uint_as_float(uu.y & 0xFFFF0000u));
          } else {
            const uint32_t uu =
                *reinterpret_cast<const uint32_t*>(tile + kk * G::kRowBytes + lane * 4);
            vf[0] = make_float2(__uint_as_float(uu << 16), __uint_as_float(uu & 0xFFFF0000u));
          }
#pragma unroll
          for (int g = 0; g < QG; ++g)
#pragma unroll
            for (int e = 0; e < G::kVe / 2; ++e)
              acc[g][e] = __ffma2_rn(make_float2(p[g], p[g]), vf[e], acc[g][e]);
        }
      }
      __syncthreads();
      if (*abort_flag) break;
      if (tid == 0) issue_next();
    }
    if (*abort_flag) break;

    // ---- the item's partials: (max, sum, unnormalised output) per query head
#pragma unroll
    for (int g = 0; g < QG; ++g)
#pragma unroll
      for (int e = 0; e < G::kVe / 2; ++e)
        *reinterpret_cast<float2*>(red_o + (warp * QG + g) * D + static_cast<int>(lane) * G::kVe +
                                   2 * e) = acc[g][e];
    __syncthreads();
    for (int y = tid; y < a.qg * D; y += kDecThreads) {
      const int g = y / D, dd = y % D;
      float o = 0.f;
#pragma unroll
      for (int w = 0; w < kDecWarps; ++w) o += red_o[(w * QG + g) * D + dd];
      a.part[((row0 + g) * a.n_split + x.s) * (2 + D) + 2 + dd] = o;
    }
    if (tid < a.qg) {
      float l = 0.f, mt = -INFINITY;
#pragma unroll
      for (int w = 0; w < kDecWarps; ++w) {
        l += hd.red2[w][tid];
        mt = fmaxf(mt, hd.red[w][tid]);
      }
      float* pm = a.part + ((row0 + tid) * a.n_split + x.s) * (2 + D);
      pm[0] = mt;
      pm[1] = l;
    }
    __syncthreads();  // red_o, hd.red and hd.red2 are free for the next item
  }

  if (*abort_flag) {
    // a wait ran out: report it, let the copies still in flight land, return
    if (tid == 0) {
      atomicOr(a.err, H2O_DEVERR_TIMEOUT);
      int never = 0;
      for (int y = g_t; y < issued; ++y)
        wait_bar(&hd.full[y % kDecStages], (y / kDecStages) & 1, &never, kWaitLimitNs / 16);
    }
  }
}

__device__ __forceinline__ float block_max(float v, float* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  const int w = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) sh[w] = v;
  __syncthreads();
  float r = sh[0];
  for (int x = 1; x < kCombineThreads / 32; ++x) r = fmaxf(r, sh[x]);
  return r;
}

__device__ __forceinline__ float block_sum(float v, float* sh) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  const int w = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) sh[w] = v;
  __syncthreads();
  float r = 0.f;
  for (int x = 0; x < kCombineThreads / 32; ++x) r += sh[x];
  return r;
}

// Per (b, hq) row and block of score_inc columns: merge the splits'
// partials into lambda (and, in the first column block, out), then rewrite
// the block's logits as weights.  The block's logits are loaded first, so
// that their round trip overlaps the merge.
template <int D>
__global__ void __launch_bounds__(kCombineThreads) decode_combine_kernel(const DecodeArgs a) {
  extern __shared__ float fac[];  // [max(n_split, threads)]: exp2(m_s - m) per split
  __shared__ float sh[kCombineThreads / 32];
  if (threadIdx.x == 0) launch_dependents();  // the S = 1 update may be placed now
  grid_dependency_wait();                      // the split kernel's partials and logits
  const int tid = threadIdx.x;
  const size_t row = blockIdx.x;  // b * Hq + hq
  float* inc = a.score_inc + row * static_cast<size_t>(a.nk);
  const int per = (a.nk + static_cast<int>(gridDim.y) - 1) / static_cast<int>(gridDim.y);
  const int c0 = static_cast<int>(blockIdx.y) * per;
  const int c1 = min(c0 + per, a.nk);
  constexpr int kPer = kCombineCols / kCombineThreads;  // per <= kCombineCols
  float lg[kPer];
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int j = c0 + tid + k * kCombineThreads;
    lg[k] = j < c1 ? inc[j] : 0.f;
  }
  const float* part = a.part + row * a.n_split * (2 + D);
  float m = -INFINITY;
  for (int s = tid; s < a.n_split; s += kCombineThreads) m = fmaxf(m, part[s * (2 + D)]);
  m = block_max(m, sh);
  float l = 0.f;
  for (int s = tid; s < a.n_split; s += kCombineThreads) {
    const float ms = part[s * (2 + D)];
    const float f = ms > -INFINITY ? fast_exp2(ms - m) : 0.f;
    fac[s] = f;
    l += part[s * (2 + D) + 1] * f;
  }
  l = block_sum(l, sh);  // (its barriers also publish fac)
  // every row sees its own token, so m is finite and l >= 1
  const float lam = m + fast_log2(l);
#pragma unroll
  for (int k = 0; k < kPer; ++k) {
    const int j = c0 + tid + k * kCombineThreads;
    if (j < c1) inc[j] = fast_exp2(lg[k] - lam);
  }
  if (blockIdx.y == 0) {
    const float inv = 1.0f / l;
    // thread (dd, q): output element dd, splits q, q + 2, ... (two halves)
    constexpr int kHalves = kCombineThreads / D;
    const int dd = tid % D, q = tid / D;
    float o0 = 0.f, o1 = 0.f;
    int s = q;
    for (; s + kHalves < a.n_split; s += 2 * kHalves) {
      o0 = fmaf(fac[s], part[s * (2 + D) + 2 + dd], o0);
      o1 = fmaf(fac[s + kHalves], part[(s + kHalves) * (2 + D) + 2 + dd], o1);
    }
    if (s < a.n_split) o0 = fmaf(fac[s], part[s * (2 + D) + 2 + dd], o0);
    const float o = o0 + o1;
    __syncthreads();  // every thread is done with fac
    fac[tid] = o;     // (fac holds at least kCombineThreads floats)
    __syncthreads();
    if (q == 0) {
      float t = fac[dd];
#pragma unroll
      for (int x = 1; x < kHalves; ++x) t += fac[x * D + dd];
      a.out[row * D + dd] = static_cast<uint16_t>(pack_bf16x2(t * inv, 0.f) & 0xFFFFu);
    }
  }
}

template <int D, int QG, bool Q8>
constexpr size_t split_smem(int split_len) {
  return kDecStages * DecGeom<D, Q8>::kSlotBytes + sizeof(DecHead) +
         static_cast<size_t>(split_len + 1) * QG * sizeof(float) +
         static_cast<size_t>(red_region_floats<D, QG, Q8>(split_len)) * sizeof(float) +
         static_cast<size_t>(kDecStages) * QG * D * sizeof(uint16_t);
}

template <int D, int QG, bool Q8>
cudaError_t launch_split(const DecodeArgs& a, cudaStream_t stream) {
  // Persistent grid: as many CTAs as fit on the GPU at once (sized once per
  // device for the largest split), each taking every gridDim-th work item.
  // One table per instantiation.
  static OncePerDevice once;
  static int resident[kMaxDevices];
  cudaError_t e = once.run([](int d) {
    const int smem_max = static_cast<int>(split_smem<D, QG, Q8>(kDecodeMaxSplitLen));
    cudaError_t r = cudaFuncSetAttribute(decode_split_kernel<D, QG, Q8>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, smem_max);
    if (r != cudaSuccess) return r;
    int per_sm = 0, sms = 0;
    r = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_split_kernel<D, QG, Q8>,
                                                      kDecThreads, smem_max);
    if (r != cudaSuccess) return r;
    r = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, d);
    if (r != cudaSuccess) return r;
    resident[d] = std::max(1, per_sm) * sms;
    return cudaSuccess;
  });
  if (e != cudaSuccess) return e;
  int dev = 0;
  e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  const int n_res = resident[dev];
  const int n_items = a.n_split * a.B * a.Hkv;
  const size_t smem = split_smem<D, QG, Q8>(a.split_len);
  decode_split_kernel<D, QG, Q8><<<std::min(n_items, n_res), kDecThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_d(const DecodeArgs& a, cudaStream_t stream) {
  cudaError_t e;
  if (a.tc)
    e = launch_decode_tc(a, stream);
  else if (a.q8)
    e = a.qg <= 4 ? launch_split<D, 4, true>(a, stream) : launch_split<D, 8, true>(a, stream);
  else
    e = a.qg <= 4 ? launch_split<D, 4, false>(a, stream) : launch_split<D, 8, false>(a, stream);
  if (e != cudaSuccess) return e;
  // launched as a programmatic dependent of the split kernel: its CTAs are
  // placed while the split kernel's last CTAs run and wait for its results
  // in grid_dependency_wait
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(a.B * a.Hq),
                     static_cast<unsigned>((a.nk + kCombineCols - 1) / kCombineCols));
  cfg.blockDim = dim3(kCombineThreads);
  cfg.dynamicSmemBytes = static_cast<size_t>(std::max(a.n_split, kCombineThreads)) * sizeof(float);
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, decode_combine_kernel<D>, a);
}

}  // namespace

bool decode_plan(int B, int Hq, int Hkv, int d, int S, int M, int* split_len, int* n_split,
                 size_t* ws_bytes) {
  if (S != 1 || M < 1 || Hq / Hkv > kDecodeMaxQg) return false;
  // Work items are (b, kv head, split); the persistent split kernel deals them
  // round-robin to its resident CTAs, so a step costs about ceil(items / CTAs)
  // items of (split_len + per-item overhead) keys.  Take the split length in
  // [128, 1536] that minimises that: a multiple of the tensor-core kernel's
  // 128-key tiles for d = 128 (one CTA per SM), of 16 otherwise (two CTAs per
  // SM).  A function of the sizes only, so that h2o_workspace_size and the
  // calls agree whichever kernel runs.
  const int64_t groups = static_cast<int64_t>(B) * Hkv;
  const int64_t gran = d == 128 ? kDecodeTcTileKeys : 16;
  const int64_t ctas = d == 128 ? kDecodeTcCtas : kDecodeResidentCtas;
  const int64_t max_len = d == 128 ? kDecodeTcMaxSplitLen : kDecodeMaxSplitLen;
  const int64_t min_len = d == 128 ? kDecodeTcMinSplitLen : kDecodeMinSplitLen;
  int64_t best_len = max_len, best_cost = INT64_MAX;
  for (int64_t len = min_len; len <= max_len; len += gran) {
    const int64_t n = (M + len - 1) / len;
    const int64_t rounds = (groups * n + ctas - 1) / ctas;
    const int64_t cost = rounds * (std::min<int64_t>(len, M) +
                                   (d == 128 ? kDecodeTcItemOverheadKeys : kDecodeItemOverheadKeys));
    if (cost < best_cost) {
      best_cost = cost;
      best_len = len;
    }
    if (len >= M) break;
  }
  const int64_t n = (M + best_len - 1) / best_len;
  *split_len = static_cast<int>(best_len);
  *n_split = static_cast<int>(n);
  *ws_bytes = static_cast<size_t>(B) * Hq * n * (2 + d) * sizeof(float);
  return true;
}

// The per-split partials of h2o_sdpa_decode_static live here instead of in a
// caller's workspace.  Every entry a call reads was written earlier in the
// same call, so nothing needs clearing between calls.
static __device__ __align__(256) unsigned char g_decode_static_scratch[kDecodeStaticScratchBytes];

cudaError_t decode_static_scratch(void** ptr) {
  return cudaGetSymbolAddress(ptr, g_decode_static_scratch);
}

cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t stream) {
  return a.d == 128 ? launch_d<128>(a, stream) : launch_d<64>(a, stream);
}

}  // namespace h2o
