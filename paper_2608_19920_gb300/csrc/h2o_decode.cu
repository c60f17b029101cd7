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

template <int D>
struct DecGeom {
  static constexpr int kRowBytes = D * 2;
  static constexpr int kTileKeys = kDecTileBytes / kRowBytes;  // 64 (d = 128) or 128
  static constexpr int kCh = D / 64;                           // 16-byte chunks per lane in Q K^T
  static constexpr int kVe = D / 32;                           // value elements per lane in P V
};

struct alignas(16) DecHead {  // 16-byte size: the logits after it are read as float4
  uint64_t full[kDecStages];
  float red[kDecWarps][kDecodeMaxQg];
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

template <int D, int QG>
__global__ void __launch_bounds__(kDecThreads, QG == 4 ? 2 : 1)
    decode_split_kernel(const DecodeArgs a) {
  using G = DecGeom<D>;
  extern __shared__ __align__(128) uint8_t dsm[];
  uint8_t* ring = dsm;
  DecHead& hd = *reinterpret_cast<DecHead*>(dsm + kDecStages * kDecTileBytes);
  static_assert(sizeof(DecHead) % 16 == 0, "logits must stay 16-byte aligned");
  float* lg = reinterpret_cast<float*>(dsm + kDecStages * kDecTileBytes + sizeof(DecHead));

  const int tid = threadIdx.x, warp = tid >> 5;
  const uint32_t lane = static_cast<uint32_t>(tid & 31);
  const int s = blockIdx.x;
  const int grp = blockIdx.y;  // b * Hkv + h
  const int b = grp / a.Hkv, h = grp % a.Hkv;
  const int j0 = s * a.split_len;
  const int n_cache = min(a.split_len, a.M - j0);  // >= 1: n_split = ceil(M / split_len)
  const bool last = s == a.n_split - 1;
  const int n_loc = n_cache + (last ? 1 : 0);       // local key n_cache is the new token
  const int n_tiles = (n_loc + G::kTileKeys - 1) / G::kTileKeys;
  const int n_all = 2 * n_tiles;                    // K tiles, then V tiles
  const uint16_t* kc = a.k_cache + (static_cast<size_t>(grp) * a.M + j0) * D;
  const uint16_t* vc = a.v_cache + (static_cast<size_t>(grp) * a.M + j0) * D;
  const uint16_t* kn = a.k_new + static_cast<size_t>(grp) * D;
  const uint16_t* vn = a.v_new + static_cast<size_t>(grp) * D;

  if (tid == 0) {
#pragma unroll
    for (int x = 0; x < kDecStages; ++x) bar_init(&hd.full[x], 1);
    hd.abort = 0;
    fence_bar_init();
  }
  __syncthreads();

  // tile t < n_tiles: K rows of local keys [t T, t T + T); then the same for V
  auto issue = [&](int t) {
    const bool is_v = t >= n_tiles;
    const int k0 = (is_v ? t - n_tiles : t) * G::kTileKeys;
    const int k1 = min(k0 + G::kTileKeys, n_loc);
    const int rows_c = max(0, min(k1, n_cache) - k0);
    const bool has_new = last && k1 > n_cache;
    uint8_t* dst = ring + (t % kDecStages) * kDecTileBytes;
    uint64_t* bar = &hd.full[t % kDecStages];
    bar_expect_tx(bar, static_cast<uint32_t>((rows_c + (has_new ? 1 : 0)) * G::kRowBytes));
    if (rows_c > 0)
      bulk_load_once(dst, (is_v ? vc : kc) + static_cast<size_t>(k0) * D,
                     static_cast<uint32_t>(rows_c * G::kRowBytes), bar);
    if (has_new)
      bulk_load_once(dst + rows_c * G::kRowBytes, is_v ? vn : kn, G::kRowBytes, bar);
  };
  int issued = 0;  // meaningful in thread 0 only
  if (tid == 0) {
    for (; issued < min(kDecStages, n_all); ++issued) issue(issued);
  }

  // this lane's slice of every head's query: chunks c0 (+ 8) of 8 elements
  const int c0 = static_cast<int>(lane & 7u);
  float qr[QG][8 * G::kCh];
#pragma unroll
  for (int g = 0; g < QG; ++g) {
    if (g < a.qg) {
      const uint16_t* qp = a.q + static_cast<size_t>(b * a.Hq + h * a.qg + g) * D;
#pragma unroll
      for (int ch = 0; ch < G::kCh; ++ch)
        bf16x8_to_f32(__ldg(reinterpret_cast<const uint4*>(qp) + c0 + 8 * ch), &qr[g][8 * ch]);
    } else {
#pragma unroll
      for (int e = 0; e < 8 * G::kCh; ++e) qr[g][e] = 0.f;
    }
  }

  const int hg = scatter_head<QG>(lane);
  const bool writer = (QG == 8 || (lane & 1u) == 0) && hg < a.qg;
  float* inc_row = a.score_inc + static_cast<size_t>(b * a.Hq + h * a.qg + (hg < a.qg ? hg : 0)) *
                                     (static_cast<size_t>(a.M) + 1);
  const int32_t* sp = a.slot_pos + static_cast<size_t>(grp) * a.M + j0;
  volatile int* abort_flag = &hd.abort;

  // ---- Q K^T: logits of the split's keys (log2 units, masked = -inf)
  float mx = -INFINITY;
  int t = 0;
  for (; t < n_tiles; ++t) {
    const bool ok = wait_bar(&hd.full[t % kDecStages], (t / kDecStages) & 1, abort_flag,
                             kWaitLimitNs);
    if (ok) {
      const uint8_t* tile = ring + (t % kDecStages) * kDecTileBytes;
#pragma unroll 1
      for (int r = 0; r < G::kTileKeys / 32; ++r) {
        const int kk = r * 32 + warp * 4 + static_cast<int>(lane >> 3);  // key within the tile
        const int kl = t * G::kTileKeys + kk;                             // key within the split
        float dot[QG];
#pragma unroll
        for (int g = 0; g < QG; ++g) dot[g] = 0.f;
        if (kl < n_loc) {
          const uint4* row = reinterpret_cast<const uint4*>(tile + kk * G::kRowBytes);
#pragma unroll
          for (int ch = 0; ch < G::kCh; ++ch) {
            float kf[8];
            bf16x8_to_f32(row[c0 + 8 * ch], kf);
#pragma unroll
            for (int e = 0; e < 8; ++e)
#pragma unroll
              for (int g = 0; g < QG; ++g) dot[g] = fmaf(qr[g][8 * ch + e], kf[e], dot[g]);
          }
        }
        const float tot = reduce_scatter8<QG>(dot, lane);
        if (writer && kl < n_loc) {
          bool vis = true;
          int j = a.M;  // the new token's column
          if (kl < n_cache) {
            const int pos = __ldg(sp + kl);
            vis = pos >= 0 && pos <= a.pos0;
            j = j0 + kl;
          }
          const float v = vis ? tot * a.scale_log2 : -INFINITY;
          lg[kl * QG + hg] = v;
          inc_row[j] = v;
          mx = fmaxf(mx, v);
        }
      }
    }
    __syncthreads();  // every warp is done with the slot
    if (*abort_flag) break;
    if (tid == 0 && issued < n_all) issue(issued++);
  }

  // ---- split max per head, then p = exp2(a - m) in place and the split sum
  const bool aborted_k = *abort_flag != 0;
  if (!aborted_k) {
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 8));
    mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
    if (QG == 4) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
    if (lane < 8u && (QG == 8 || (lane & 1u) == 0)) hd.red[warp][hg] = mx;
  }
  __syncthreads();
  const int gp = tid % QG;  // the head of every lg entry this thread converts
  float m_g = -INFINITY;
#pragma unroll
  for (int w = 0; w < kDecWarps; ++w) m_g = fmaxf(m_g, hd.red[w][gp]);
  float lsum = 0.f;
  if (!aborted_k && gp < a.qg) {
    for (int x = tid; x < n_loc * QG; x += kDecThreads) {
      const float p = m_g > -INFINITY ? fast_exp2(lg[x] - m_g) : 0.f;
      lg[x] = p;
      lsum += p;
    }
  }
  // lanes holding the same head: lane bits >= log2(QG)
#pragma unroll
  for (int o = QG; o < 32; o <<= 1) lsum += __shfl_xor_sync(0xffffffffu, lsum, o);
  __syncthreads();  // every thread has read hd.red (max) and written its p
  if (lane < static_cast<uint32_t>(QG)) hd.red[warp][lane] = lsum;

  // ---- P V: one warp per key, lanes over d
  float acc[QG][G::kVe];
#pragma unroll
  for (int g = 0; g < QG; ++g)
#pragma unroll
    for (int e = 0; e < G::kVe; ++e) acc[g][e] = 0.f;
  if (!aborted_k) {
    for (; t < n_all; ++t) {
      const bool ok = wait_bar(&hd.full[t % kDecStages], (t / kDecStages) & 1, abort_flag,
                               kWaitLimitNs);
      if (ok) {
        const uint8_t* tile = ring + (t % kDecStages) * kDecTileBytes;
        const int k0 = (t - n_tiles) * G::kTileKeys;
        const int kend = min(G::kTileKeys, n_loc - k0);
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
          float vf[G::kVe];
          if constexpr (D == 128) {
            const uint2 u = *reinterpret_cast<const uint2*>(tile + kk * G::kRowBytes + lane * 8);
            vf[0] = __uint_as_float(u.x << 16);
            vf[1] = __uint_as_float(u.x & 0xFFFF0000u);
            vf[2] = __uint_as_float(u.y << 16);
            vf[3] = __uint_as_float(u.y & 0xFFFF0000u);
          } else {
            const uint32_t u = *reinterpret_cast<const uint32_t*>(tile + kk * G::kRowBytes + lane * 4);
            vf[0] = __uint_as_float(u << 16);
            vf[1] = __uint_as_float(u & 0xFFFF0000u);
          }
#pragma unroll
          for (int g = 0; g < QG; ++g)
#pragma unroll
            for (int e = 0; e < G::kVe; ++e) acc[g][e] = fmaf(p[g], vf[e], acc[g][e]);
        }
      }
      __syncthreads();
      if (*abort_flag) break;
      if (tid == 0 && issued < n_all) issue(issued++);
    }
  }

  if (*abort_flag) {
    // a wait ran out: report it, let the copies still in flight land, return
    if (tid == 0) {
      atomicOr(a.err, H2O_DEVERR_TIMEOUT);
      int never = 0;
      for (int x = t; x < issued; ++x)
        wait_bar(&hd.full[x % kDecStages], (x / kDecStages) & 1, &never, kWaitLimitNs / 16);
    }
    return;
  }

  // ---- combine the warps' partial outputs (the ring is free: every copy landed)
  float* red_o = reinterpret_cast<float*>(ring);  // [warp][g][D]
#pragma unroll
  for (int g = 0; g < QG; ++g)
#pragma unroll
    for (int e = 0; e < G::kVe; ++e)
      red_o[(warp * QG + g) * D + static_cast<int>(lane) * G::kVe + e] = acc[g][e];
  __syncthreads();
  const size_t row0 = static_cast<size_t>(b * a.Hq + h * a.qg);
  for (int x = tid; x < a.qg * D; x += kDecThreads) {
    const int g = x / D, dd = x % D;
    float o = 0.f;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) o += red_o[(w * QG + g) * D + dd];
    a.part[((row0 + g) * a.n_split + s) * (2 + D) + 2 + dd] = o;
  }
  if (tid < a.qg) {
    // thread tid < QG converted head gp = tid: m_g is that head's split max;
    // hd.red now holds the warps' partial sums
    float l = 0.f;
#pragma unroll
    for (int w = 0; w < kDecWarps; ++w) l += hd.red[w][tid];
    float* pm = a.part + ((row0 + tid) * a.n_split + s) * (2 + D);
    pm[0] = m_g;
    pm[1] = l;
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

template <int D>
__global__ void __launch_bounds__(kCombineThreads) decode_combine_kernel(const DecodeArgs a) {
  __shared__ float sh[kCombineThreads / 32];
  const int tid = threadIdx.x;
  const size_t row = blockIdx.x;  // b * Hq + hq
  const float* part = a.part + row * a.n_split * (2 + D);
  float m = -INFINITY;
  for (int s = tid; s < a.n_split; s += kCombineThreads) m = fmaxf(m, part[s * (2 + D)]);
  m = block_max(m, sh);
  float l = 0.f;
  for (int s = tid; s < a.n_split; s += kCombineThreads) {
    const float ms = part[s * (2 + D)];
    if (ms > -INFINITY) l += part[s * (2 + D) + 1] * fast_exp2(ms - m);
  }
  l = block_sum(l, sh);
  // every row sees its own token, so m is finite and l >= 1
  const float lam = m + fast_log2(l);
  if (blockIdx.y == 0) {
    const float inv = 1.0f / l;
    for (int dp = tid; dp < D / 2; dp += kCombineThreads) {
      float o0 = 0.f, o1 = 0.f;
      for (int s = 0; s < a.n_split; ++s) {
        const float ms = part[s * (2 + D)];
        if (ms > -INFINITY) {
          const float f = fast_exp2(ms - m);
          o0 = fmaf(f, part[s * (2 + D) + 2 + 2 * dp], o0);
          o1 = fmaf(f, part[s * (2 + D) + 3 + 2 * dp], o1);
        }
      }
      reinterpret_cast<uint32_t*>(a.out + row * D)[dp] = pack_bf16x2(o0 * inv, o1 * inv);
    }
  }
  float* inc = a.score_inc + row * (static_cast<size_t>(a.M) + 1);
  const int c0 = static_cast<int>(blockIdx.y) * kCombineCols;
  const int c1 = min(c0 + kCombineCols, a.M + 1);
#pragma unroll 4
  for (int j = c0 + tid; j < c1; j += kCombineThreads) inc[j] = fast_exp2(inc[j] - lam);
}

template <int QG>
constexpr size_t split_smem(int split_len) {
  return kDecStages * kDecTileBytes + sizeof(DecHead) +
         static_cast<size_t>(split_len + 1) * QG * sizeof(float);
}

template <int D, int QG>
cudaError_t launch_split(const DecodeArgs& a, cudaStream_t stream) {
  // the attribute is set once per device, for the largest split
  static bool configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev >= 64 || !configured[dev]) {
    e = cudaFuncSetAttribute(decode_split_kernel<D, QG>,
                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                             static_cast<int>(split_smem<QG>(kDecodeMaxSplitLen)));
    if (e != cudaSuccess) return e;
    if (dev < 64) configured[dev] = true;
  }
  const size_t smem = split_smem<QG>(a.split_len);
  const dim3 grid(static_cast<unsigned>(a.n_split), static_cast<unsigned>(a.B * a.Hkv));
  decode_split_kernel<D, QG><<<grid, kDecThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

template <int D>
cudaError_t launch_d(const DecodeArgs& a, cudaStream_t stream) {
  cudaError_t e = a.qg <= 4 ? launch_split<D, 4>(a, stream) : launch_split<D, 8>(a, stream);
  if (e != cudaSuccess) return e;
  const dim3 grid(static_cast<unsigned>(a.B * a.Hq),
                  static_cast<unsigned>((a.M + 1 + kCombineCols - 1) / kCombineCols));
  decode_combine_kernel<D><<<grid, kCombineThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

bool decode_plan(int B, int Hq, int Hkv, int d, int S, int M, int* split_len, int* n_split,
                 size_t* ws_bytes) {
  if (S != 1 || M < 1 || Hq / Hkv > kDecodeMaxQg) return false;
  const int64_t groups = static_cast<int64_t>(B) * Hkv;
  int64_t len = (static_cast<int64_t>(M) * groups + kDecodeTargetCtas - 1) / kDecodeTargetCtas;
  len = (len + 63) / 64 * 64;
  len = std::min<int64_t>(std::max<int64_t>(len, kDecodeMinSplitLen), kDecodeMaxSplitLen);
  const int64_t n = (M + len - 1) / len;
  *split_len = static_cast<int>(len);
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
