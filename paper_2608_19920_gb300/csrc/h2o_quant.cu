// 8-bit K/V cache buffers (the setup of §4 keeps the KV cache buffers in 8
// bits).
//
// Format, per cache row of d elements (one token's key, or its value, in one KV
// head): d int8 codes c and one fp32 scale s, symmetric per row:
//   s = max_e |x_e| / 127,   c_e = round_half_even(x_e / s) clipped to [-127, 127],
// the division and the rounding in fp32 (IEEE division: __fdiv_rn), so the
// integer decisions are reproducible; an all-zero row has s = 0 and codes 0.
// A row is read back as bf16(fp32(c) * s): the attention computes in bf16 as
// it does on a bf16 cache.
//
//  * kv_quantize_kernel:   one warp per row, bf16 in, codes + scale out.
//  * kv_scatter_q8_kernel: the chunk's rows quantised into the slots an update
//                          chose (evict_idx): the 8-bit form of the K/V
//                          scatter of §3.2 / §A.1.1.
//  * kv_dequantize_kernel: codes + scales -> bf16 rows, 16 codes per thread
//                          (16 B read, 32 B written), for the chunk SDPA.
//
// All three are HBM bound; bytes per row: quantise 2d read + (d + 4) written,
// dequantise (d + 4) read + 2d written.
#include <cstdint>

#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kQThreads = 256;
constexpr int kQWarps = kQThreads / 32;
constexpr int kQMaxBlocks = 152 * 16;
constexpr float kQMax = 127.f;

// One row of D bf16 values, read and written by a warp: lane l takes elements
// [E l, E l + E), E = D / 32.
template <int D>
__device__ __forceinline__ void quantize_row(const uint16_t* src, int8_t* codes, float* scale,
                                             int lane) {
  constexpr int E = D / 32;  // 4 (d = 128) or 2 (d = 64)
  float x[E];
  if constexpr (E == 4) {
    const uint2 u = __ldg(reinterpret_cast<const uint2*>(src) + lane);
    x[0] = __uint_as_float(u.x << 16);
    x[1] = __uint_as_float(u.x & 0xFFFF0000u);
    x[2] = __uint_as_float(u.y << 16);
    x[3] = __uint_as_float(u.y & 0xFFFF0000u);
  } else {
    const uint32_t u = __ldg(reinterpret_cast<const uint32_t*>(src) + lane);
    x[0] = __uint_as_float(u << 16);
    x[1] = __uint_as_float(u & 0xFFFF0000u);
  }
  float amax = 0.f;
#pragma unroll
  for (int e = 0; e < E; ++e) amax = fmaxf(amax, fabsf(x[e]));
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) amax = fmaxf(amax, __shfl_xor_sync(0xffffffffu, amax, o));
  const float s = __fdiv_rn(amax, kQMax);
  uint32_t packed = 0;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    int c = 0;
    if (s > 0.f) c = max(-127, min(127, __float2int_rn(__fdiv_rn(x[e], s))));
    packed |= (static_cast<uint32_t>(c) & 0xFFu) << (8 * e);
  }
  if constexpr (E == 4)
    reinterpret_cast<uint32_t*>(codes)[lane] = packed;
  else
    reinterpret_cast<uint16_t*>(codes)[lane] = static_cast<uint16_t>(packed);
  if (lane == 0) *scale = s;
}

template <int D>
__global__ void __launch_bounds__(kQThreads) kv_quantize_kernel(const uint16_t* x, int8_t* codes,
                                                                float* scales, int64_t n_rows) {
  const int lane = threadIdx.x & 31;
  const int64_t step = static_cast<int64_t>(gridDim.x) * kQWarps;
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * kQWarps + (threadIdx.x >> 5); r < n_rows;
       r += step)
    quantize_row<D>(x + r * D, codes + r * D, scales + r, lane);
}

// One warp per (group, token c, K or V): the row goes to slot evict_idx; a
// slot of -1 (no selection was made for that group) leaves the buffers as
// they are; one outside [0, M) is recorded (H2O_DEVERR_INDEX) and skipped.
template <int D>
__global__ void __launch_bounds__(kQThreads) kv_scatter_q8_kernel(const Q8ScatterArgs a) {
  const int lane = threadIdx.x & 31;
  const int64_t items = static_cast<int64_t>(a.B) * a.Hkv * a.S * 2;
  const int64_t step = static_cast<int64_t>(gridDim.x) * kQWarps;
  for (int64_t it = static_cast<int64_t>(blockIdx.x) * kQWarps + (threadIdx.x >> 5); it < items;
       it += step) {
    const int64_t grp = it / (2 * a.S);
    const int rem = static_cast<int>(it % (2 * a.S));
    const int c = rem >> 1;
    const bool is_v = rem & 1;
    const int e = __ldg(a.evict_idx + grp * a.S + c);
    if (e < 0) continue;
    if (e >= a.M) {
      if (lane == 0) atomicOr(a.err, H2O_DEVERR_INDEX);
      continue;
    }
    const uint16_t* src = (is_v ? a.v_new : a.k_new) + (grp * a.S + c) * D;
    const int64_t slot = grp * a.M + e;
    quantize_row<D>(src, (is_v ? a.buf.v_codes : a.buf.k_codes) + slot * D,
                    (is_v ? a.buf.v_scales : a.buf.k_scales) + slot, lane);
  }
}

// 16 codes per thread: one 16-byte load, 16 products fp32(c) * s rounded to
// bf16, two 16-byte stores.  blockIdx.y picks the first or the second tensor.
template <int D>
__global__ void __launch_bounds__(kQThreads) kv_dequantize_kernel(
    const int8_t* codes0, const float* scales0, uint16_t* x0, const int8_t* codes1,
    const float* scales1, uint16_t* x1, int64_t n_rows) {
  constexpr int kPiecesPerRow = D / 16;
  const int8_t* codes = blockIdx.y ? codes1 : codes0;
  const float* scales = blockIdx.y ? scales1 : scales0;
  uint16_t* x = blockIdx.y ? x1 : x0;
  const int64_t pieces = n_rows * kPiecesPerRow;
  const int64_t step = static_cast<int64_t>(gridDim.x) * kQThreads;
  for (int64_t p = static_cast<int64_t>(blockIdx.x) * kQThreads + threadIdx.x; p < pieces;
       p += step) {
    const float s = __ldg(scales + p / kPiecesPerRow);
    const uint4 u = __ldcs(reinterpret_cast<const uint4*>(codes) + p);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
    uint32_t o[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) {
      const uint32_t word = w[k >> 1];
      const int sh = 16 * (k & 1);
      const float lo = __fmul_rn(static_cast<float>(static_cast<int8_t>((word >> sh) & 0xFFu)), s);
      const float hi =
          __fmul_rn(static_cast<float>(static_cast<int8_t>((word >> (sh + 8)) & 0xFFu)), s);
      o[k] = pack_bf16x2(lo, hi);
    }
    uint4* dst = reinterpret_cast<uint4*>(x) + 2 * p;
    dst[0] = make_uint4(o[0], o[1], o[2], o[3]);
    dst[1] = make_uint4(o[4], o[5], o[6], o[7]);
  }
}

unsigned grid_for(int64_t units, int per_block) {
  const int64_t b = (units + per_block - 1) / per_block;
  return static_cast<unsigned>(b < 1 ? 1 : b > kQMaxBlocks ? kQMaxBlocks : b);
}

}  // namespace

cudaError_t launch_kv_quantize(const uint16_t* x, int8_t* codes, float* scales, int64_t n_rows,
                               int d, cudaStream_t stream) {
  if (n_rows <= 0) return cudaSuccess;
  const unsigned grid = grid_for(n_rows, kQWarps);
  if (d == 128)
    kv_quantize_kernel<128><<<grid, kQThreads, 0, stream>>>(x, codes, scales, n_rows);
  else
    kv_quantize_kernel<64><<<grid, kQThreads, 0, stream>>>(x, codes, scales, n_rows);
  return cudaGetLastError();
}

cudaError_t launch_kv_dequantize(const int8_t* codes, const float* scales, uint16_t* x,
                                 const int8_t* codes2, const float* scales2, uint16_t* x2,
                                 int64_t n_rows, int d, cudaStream_t stream) {
  if (n_rows <= 0) return cudaSuccess;
  const dim3 grid(grid_for(n_rows * (d / 16), kQThreads), codes2 ? 2u : 1u);
  if (d == 128)
    kv_dequantize_kernel<128><<<grid, kQThreads, 0, stream>>>(codes, scales, x, codes2, scales2,
                                                              x2, n_rows);
  else
    kv_dequantize_kernel<64><<<grid, kQThreads, 0, stream>>>(codes, scales, x, codes2, scales2,
                                                             x2, n_rows);
  return cudaGetLastError();
}

cudaError_t launch_kv_scatter_q8(const Q8ScatterArgs& a, cudaStream_t stream) {
  const int64_t items = static_cast<int64_t>(a.B) * a.Hkv * a.S * 2;
  if (items <= 0) return cudaSuccess;
  const unsigned grid = grid_for(items, kQWarps);
  if (a.d == 128)
    kv_scatter_q8_kernel<128><<<grid, kQThreads, 0, stream>>>(a);
  else
    kv_scatter_q8_kernel<64><<<grid, kQThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace h2o
