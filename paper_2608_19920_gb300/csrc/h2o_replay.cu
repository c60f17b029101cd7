// Replay-cache row operations (§3.2 recurrence, §A.1.1 scatter / gather).
//
// A chunk's cache write is a scatter of its S rows into the slots `index`
// (B, Hkv, S) along the slot axis; the reverse recurrence of §3.2 restores
// the buffers from the rows that write replaced (delta_key = gather(keys,
// index), taken before it).  kv_rows_kernel does either direction for K, V
// and, when given, the slot positions: one warp per (b, h, c) row pair, lanes
// 0-15 the K row and 16-31 the V row in 16-byte pieces (a row is contiguous,
// the index is constant along d), the old row read before the new one is
// written.  Pure copies, bandwidth bound: 2 x 2 d bytes read and written per
// row pair (3 x with the delta).  An index outside [0, M) is recorded in the
// device error word and its row skipped.
#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kRowThreads = 256;
constexpr int kRowWarps = kRowThreads / 32;

__global__ void __launch_bounds__(kRowThreads) kv_rows_kernel(const ReplayArgs a) {
  const int lane = static_cast<int>(threadIdx.x & 31);
  const size_t n_rows = static_cast<size_t>(a.B) * a.Hkv * a.S;
  const int vec = a.d / 8;  // 16-byte pieces per row
  const bool is_v = lane >= 16;
  const int l = lane & 15;
  for (size_t r = blockIdx.x * static_cast<size_t>(kRowWarps) + (threadIdx.x >> 5); r < n_rows;
       r += static_cast<size_t>(gridDim.x) * kRowWarps) {
    const size_t grp = r / a.S;
    const int c = static_cast<int>(r % a.S);
    const int e = __ldg(a.index + r);
    if (e < 0 || e >= a.M) {
      if (lane == 0) atomicOr(a.err, H2O_DEVERR_INDEX);
      continue;
    }
    const size_t slot = grp * a.M + static_cast<size_t>(e);
    uint4* cache = reinterpret_cast<uint4*>((is_v ? a.v_cache : a.k_cache) + slot * a.d);
    if (a.restore) {
      const uint4* src = reinterpret_cast<const uint4*>((is_v ? a.delta_v : a.delta_k) + r * a.d);
      for (int x = l; x < vec; x += 16) cache[x] = __ldg(src + x);
      if (lane == 0 && a.slot_pos && a.delta_pos) a.slot_pos[slot] = __ldg(a.delta_pos + r);
    } else {
      const uint4* src = reinterpret_cast<const uint4*>((is_v ? a.v_new : a.k_new) + r * a.d);
      uint16_t* dptr = is_v ? a.delta_v : a.delta_k;
      uint4* delta = dptr ? reinterpret_cast<uint4*>(dptr + r * a.d) : nullptr;
      for (int x = l; x < vec; x += 16) {
        const uint4 fresh = __ldg(src + x);
        if (delta) delta[x] = cache[x];
        cache[x] = fresh;
      }
      if (lane == 0 && a.slot_pos) {
        if (a.delta_pos) a.delta_pos[r] = a.slot_pos[slot];
        a.slot_pos[slot] = a.pos0 + c;
      }
    }
  }
}

}  // namespace

cudaError_t launch_kv_rows(const ReplayArgs& a, cudaStream_t stream) {
  const size_t n_rows = static_cast<size_t>(a.B) * a.Hkv * a.S;
  size_t blocks = (n_rows + kRowWarps - 1) / kRowWarps;
  if (blocks > 152 * 16) blocks = 152 * 16;
  kv_rows_kernel<<<static_cast<unsigned>(blocks), kRowThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace h2o
