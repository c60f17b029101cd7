// C ABI of the H2O sparse-attention library: argument checking, tensor-map
// encoding and kernel launches.  Declarations and contracts: include/h2o.h.
#include <cuda.h>
#include <cuda_runtime.h>
#include <cudaTypedefs.h>

#include <cmath>
#include <cstdint>
#include <cstring>
#include <mutex>

#include "../../include/h2o.h"
#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {

// Device-side error bits (H2O_DEVERR_*), one word per device.
__device__ int g_device_errors;

namespace {

thread_local int t_last_cuda_error = 0;

struct DeviceInfo {
  std::once_flag once;
  cudaError_t status = cudaSuccess;
  bool supported = false;
  int* err_word = nullptr;
};
DeviceInfo g_dev[kMaxDevices];

std::once_flag g_encode_once;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;

int cuda_fail(cudaError_t e) {
  t_last_cuda_error = static_cast<int>(e);
  return H2O_ERR_CUDA;
}

// Resolves the current device once: architecture check and error-word address.
int current_device(DeviceInfo** out) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e == cudaErrorNoDevice || e == cudaErrorInsufficientDriver
                                   ? H2O_ERR_NODEVICE
                                   : cuda_fail(e);
  if (dev < 0 || dev >= kMaxDevices) return H2O_ERR_NODEVICE;
  DeviceInfo& di = g_dev[dev];
  std::call_once(di.once, [&di, dev] {
    cudaDeviceProp prop;
    di.status = cudaGetDeviceProperties(&prop, dev);
    if (di.status != cudaSuccess) return;
    di.supported = prop.major == 10;
    if (!di.supported) return;
    di.status = cudaGetSymbolAddress(reinterpret_cast<void**>(&di.err_word), g_device_errors);
  });
  if (di.status != cudaSuccess) return cuda_fail(di.status);
  if (!di.supported) return H2O_ERR_NODEVICE;
  *out = &di;
  return H2O_OK;
}

// Address of the decode kernels' fixed scratch on each device, resolved once.
struct StaticScratch {
  std::once_flag once;
  cudaError_t status = cudaSuccess;
  void* ptr = nullptr;
};
StaticScratch g_static_scratch[kMaxDevices];

int get_encoder() {
  std::call_once(g_encode_once, [] {
    cudaDriverEntryPointQueryResult q;
    void* fn = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  });
  return g_encode ? H2O_OK : H2O_ERR_NODEVICE;
}

bool misaligned(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; }

// Dense tensor map, dims/box innermost first, elements of `esize` bytes.
int encode_any(CUtensorMap* m, CUtensorMapDataType type, int esize, CUtensorMapSwizzle swizzle,
               const void* base, int rank, const uint64_t* dims, const uint32_t* box) {
  cuuint64_t gd[5], gs[4];
  cuuint32_t bx[5], es[5];
  uint64_t stride = static_cast<uint64_t>(esize);
  for (int r = 0; r < rank; ++r) {
    gd[r] = dims[r];
    bx[r] = box[r];
    es[r] = 1;
    if (r > 0) gs[r - 1] = stride;
    stride *= dims[r];
  }
  const CUresult res = g_encode(m, type, rank, const_cast<void*>(base), gd, gs, bx, es,
                                CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle,
                                CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                                CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return res == CUDA_SUCCESS ? H2O_OK : H2O_ERR_SHAPE;
}

// bf16 tensor map, 128-byte swizzle, dims/box innermost first.
int encode(CUtensorMap* m, const void* base, int rank, const uint64_t* dims, const uint32_t* box) {
  return encode_any(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, CU_TENSOR_MAP_SWIZZLE_128B, base, rank,
                    dims, box);
}

// The tensor-core decode kernel's TMA maps (d = 128): bf16 cache rows, or
// with 8-bit buffers the code rows (128 bytes, no swizzle) and the row
// scales (one flat fp32 array; a 128-scale tile starts 16-byte aligned only
// when M is a multiple of 4, else the CUDA-core kernel runs).  Otherwise a.tc
// stays 0 and the CUDA-core split kernel runs.
int decode_maps(DecodeArgs& a) {
  a.tc = 0;
  if (a.d != 128) return H2O_OK;
  if (a.q8 && (a.M % 4 != 0 || static_cast<int64_t>(a.B) * a.Hkv * a.M >= (int64_t(1) << 31)))
    return H2O_OK;
  int st = get_encoder();
  if (st != H2O_OK) return st;
  const uint64_t G = static_cast<uint64_t>(a.B) * a.Hkv;
  const uint64_t dq[3] = {128, static_cast<uint64_t>(a.Hq), static_cast<uint64_t>(a.B)};
  const uint32_t bq[3] = {64, 16, 1};
  if ((st = encode(&a.tm_q, a.q, 3, dq, bq)) != H2O_OK) return st;
  if (!a.q8) {
    const uint64_t dc[3] = {128, static_cast<uint64_t>(a.M), G};
    const uint32_t bc[3] = {64, static_cast<uint32_t>(kDecodeTcTileKeys), 1};
    if ((st = encode(&a.tm_kc, a.k_cache, 3, dc, bc)) != H2O_OK) return st;
    if ((st = encode(&a.tm_vc, a.v_cache, 3, dc, bc)) != H2O_OK) return st;
  } else {
    const uint64_t dc[3] = {128, static_cast<uint64_t>(a.M), G};
    const uint32_t bc[3] = {128, static_cast<uint32_t>(kDecodeTcTileKeys), 1};
    const uint64_t ds[1] = {G * static_cast<uint64_t>(a.M)};
    const uint32_t bs[1] = {static_cast<uint32_t>(kDecodeTcTileKeys)};
    if ((st = encode_any(&a.tm_kc, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, CU_TENSOR_MAP_SWIZZLE_NONE,
                         a.k_codes, 3, dc, bc)) != H2O_OK)
      return st;
    if ((st = encode_any(&a.tm_vc, CU_TENSOR_MAP_DATA_TYPE_UINT8, 1, CU_TENSOR_MAP_SWIZZLE_NONE,
                         a.v_codes, 3, dc, bc)) != H2O_OK)
      return st;
    if ((st = encode_any(&a.tm_ks, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, CU_TENSOR_MAP_SWIZZLE_NONE,
                         a.k_scales, 1, ds, bs)) != H2O_OK)
      return st;
    if ((st = encode_any(&a.tm_vs, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 4, CU_TENSOR_MAP_SWIZZLE_NONE,
                         a.v_scales, 1, ds, bs)) != H2O_OK)
      return st;
  }
  a.tc = 1;
  return H2O_OK;
}

int check_dims(const h2o_dims_t* d) {
  if (!d) return H2O_ERR_NULL;
  if (d->B < 1 || d->Hq < 1 || d->Hkv < 1 || d->S < 1 || d->M < 0 || d->d < 1) return H2O_ERR_SHAPE;
  if (d->Hq % d->Hkv != 0) return H2O_ERR_SHAPE;
  if (d->d != 64 && d->d != 128) return H2O_ERR_UNSUPPORTED;
  if (d->B * static_cast<int64_t>(d->Hkv) > 65535) return H2O_ERR_UNSUPPORTED;
  const int64_t tiles = (d->M + kTileN - 1) / kTileN + (d->S + kTileN - 1) / kTileN;
  if (tiles > kMaxKeyTiles) return H2O_ERR_UNSUPPORTED;
  const int64_t elems = static_cast<int64_t>(d->B) * d->Hq * (static_cast<int64_t>(d->M) + d->S);
  if (elems > (int64_t(1) << 40)) return H2O_ERR_SHAPE;
  return H2O_OK;
}

// h2o_sdpa_chunk (cache_only = false: keys are the M slots, then the chunk's
// S tokens) and h2o_sdpa_cache (cache_only = true: the M slots only, the
// chunk's keys already written there; k_new / v_new unused).  With q8 (the
// 8-bit buffer calls) the decode kernels read the codes themselves; the chunk
// kernel reads k_cache / v_cache = q8's bf16 read-back rows, filled from the
// codes on the stream just before it.
int sdpa_impl(const h2o_dims_t* dims, int64_t pos0, float softmax_scale, const h2o_bf16* q,
              const h2o_bf16* k_cache, const h2o_bf16* v_cache, const h2o_bf16* k_new,
              const h2o_bf16* v_new, const int32_t* slot_pos, h2o_bf16* out, float* score_inc,
              void* workspace, size_t workspace_bytes, void* stream, bool cache_only,
              const Q8Buffers* q8 = nullptr, const SdpaArgs* lse_req = nullptr,
              float* lse_out = nullptr) {
  // lse_req (the backward's recomputation): its lse, lse_stride, bwd_out,
  // bwd_dout and drow fields; the chunk kernel's pass 1 alone then writes the
  // rows' log-sum-exp and D, and neither out nor score_inc
  float* lse = lse_req ? lse_req->lse : nullptr;
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (!q || (!lse && (!out || !score_inc)) || (!cache_only && (!k_new || !v_new)))
    return H2O_ERR_NULL;
  // (q8: the codes were checked by the caller; the decode kernels need no rows)
  if (D.M > 0 && ((!q8 && (!k_cache || !v_cache)) || !slot_pos)) return H2O_ERR_NULL;
  if (misaligned(q) || misaligned(k_new) || misaligned(v_new) || misaligned(out) ||
      misaligned(score_inc) || (D.M > 0 && (misaligned(k_cache) || misaligned(v_cache) ||
                                            misaligned(slot_pos))))
    return H2O_ERR_ALIGN;
  const int nk = cache_only ? D.M : D.M + D.S;  // key columns of a score_inc row
  if (pos0 < 0 || pos0 + D.S >= (int64_t(1) << 31)) return H2O_ERR_ARG;
  if (!(softmax_scale <= 0.f) && !std::isfinite(softmax_scale)) return H2O_ERR_ARG;
  const int qg = D.Hq / D.Hkv;
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt(static_cast<float>(D.d));
  int split_len = 0, n_split = 0;
  size_t ws_need = 0;
  // lse_out (the forward's lse for a later backward): the chunk kernel, also
  // for S = 1, which writes each row's lambda as it enters its second pass
  if (lse_out && misaligned(lse_out)) return H2O_ERR_ALIGN;
  const bool decode = !lse && !lse_out &&
                      decode_plan(D.B, D.Hq, D.Hkv, D.d, D.S, D.M, &split_len, &n_split, &ws_need);
  if (!decode) ws_need = lse ? 0 : sdpa_colpart_bytes(D.B, D.Hq, D.S, D.M);
  if (ws_need > 0 && (!workspace || workspace_bytes < ws_need)) return H2O_ERR_WORKSPACE;
  if (ws_need > 0 && misaligned(workspace)) return H2O_ERR_ALIGN;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // the 8-bit buffers' rows, read back to bf16 ahead of the attention kernels
  auto read_back = [&]() -> cudaError_t {
    if (!q8) return cudaSuccess;
    return launch_kv_dequantize(q8->k_codes, q8->k_scales, q8->k_rows, q8->v_codes, q8->v_scales,
                                q8->v_rows, static_cast<int64_t>(D.B) * D.Hkv * D.M, D.d, s);
  };

  if (decode) {
    // one query token per sequence: split-K kernels (h2o_decode.cu)
    DecodeArgs a{};
    a.q = q; a.k_cache = k_cache; a.v_cache = v_cache; a.k_new = k_new; a.v_new = v_new;
    a.slot_pos = slot_pos; a.out = out; a.score_inc = score_inc;
    a.part = static_cast<float*>(workspace);
    a.err = di->err_word;
    a.B = D.B; a.Hq = D.Hq; a.Hkv = D.Hkv; a.d = D.d; a.M = D.M; a.qg = qg;
    a.pos0 = static_cast<int>(pos0);
    a.scale_log2 = scale * 1.4426950408889634f;
    a.split_len = split_len;
    a.n_split = n_split;
    a.with_new = cache_only ? 0 : 1;
    a.nk = nk;
    a.q8 = q8 ? 1 : 0;
    a.k_codes = q8 ? q8->k_codes : nullptr;
    a.k_scales = q8 ? q8->k_scales : nullptr;
    a.v_codes = q8 ? q8->v_codes : nullptr;
    a.v_scales = q8 ? q8->v_scales : nullptr;
    if ((st = decode_maps(a)) != H2O_OK) return st;
    const cudaError_t e = launch_decode(a, s);
    return e == cudaSuccess ? H2O_OK : cuda_fail(e);
  }
  if ((st = get_encoder()) != H2O_OK) return st;

  SdpaArgs a;
  std::memset(&a, 0, sizeof(a));
  a.B = D.B; a.Hq = D.Hq; a.Hkv = D.Hkv; a.d = D.d; a.S = D.S; a.M = D.M; a.qg = qg;
  a.pos0 = static_cast<int>(pos0);
  a.scale_log2 = scale * 1.4426950408889634f;
  if (D.S > kTileM) {
    a.rows_box = kTileM;
    a.heads_box = 1;
    a.tiles_per_head = (D.S + kTileM - 1) / kTileM;
    a.n_row_tiles = qg * a.tiles_per_head;
  } else {
    a.rows_box = (D.S + 31) / 32 * 32;
    a.heads_box = kTileM / a.rows_box;
    a.tiles_per_head = 0;
    a.n_row_tiles = (qg + a.heads_box - 1) / a.heads_box;
  }
  a.n_cache_tiles = (D.M + kTileN - 1) / kTileN;
  a.n_chunk_tiles = cache_only ? 0 : (D.S + kTileN - 1) / kTileN;
  a.nk = nk;
  a.slot_pos = slot_pos;
  a.out = out;
  a.score_inc = score_inc;
  a.err = di->err_word;
  a.colpart = ws_need > 0 ? static_cast<float*>(workspace) : nullptr;
  a.lse_out = lse_out;
  if (lse_req) {
    a.lse = lse_req->lse;
    a.lse_stride = lse_req->lse_stride;
    a.bwd_out = lse_req->bwd_out;
    a.bwd_dout = lse_req->bwd_dout;
    a.drow = lse_req->drow;
  }

  const uint64_t G = static_cast<uint64_t>(D.B) * D.Hkv;
  {
    const uint64_t dq[4] = {static_cast<uint64_t>(D.d), static_cast<uint64_t>(D.S),
                            static_cast<uint64_t>(qg), G};
    const uint32_t bq[4] = {64, static_cast<uint32_t>(a.rows_box), static_cast<uint32_t>(a.heads_box), 1};
    if ((st = encode(&a.tm_q, q, 4, dq, bq)) != H2O_OK) return st;
    // d = 128 runs on CTA pairs: each CTA loads 64 keys of a K tile and 64
    // columns of a V tile; d = 64 loads whole 128-key tiles.
    const uint64_t dn[3] = {static_cast<uint64_t>(D.d), static_cast<uint64_t>(D.S), G};
    const uint32_t bk[3] = {64, D.d == 128 ? kTileN / 2u : kTileN, 1};
    const uint32_t bv[3] = {64, kTileN, 1};
    const uint64_t dc[3] = {static_cast<uint64_t>(D.d), static_cast<uint64_t>(D.M), G};
    if (cache_only) {  // no chunk tiles: the chunk maps are never read
      if ((st = encode(&a.tm_kn, k_cache, 3, dc, bk)) != H2O_OK) return st;
      if ((st = encode(&a.tm_vn, v_cache, 3, dc, bv)) != H2O_OK) return st;
    } else {
      if ((st = encode(&a.tm_kn, k_new, 3, dn, bk)) != H2O_OK) return st;
      if ((st = encode(&a.tm_vn, v_new, 3, dn, bv)) != H2O_OK) return st;
    }
    if (D.M > 0) {
      if ((st = encode(&a.tm_kc, k_cache, 3, dc, bk)) != H2O_OK) return st;
      if ((st = encode(&a.tm_vc, v_cache, 3, dc, bv)) != H2O_OK) return st;
    }
  }
  const size_t inc_bytes = static_cast<size_t>(G) * qg * static_cast<size_t>(nk) * sizeof(float);
  cudaError_t e = read_back();
  if (e != cudaSuccess) return cuda_fail(e);
  if (a.colpart == nullptr && !lse) {
    e = cudaMemsetAsync(score_inc, 0, inc_bytes, s);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  e = launch_sdpa(a, s);
  if (e != cudaSuccess) return cuda_fail(e);
  if (a.colpart != nullptr) {
    e = launch_colsum_reduce(a.colpart, score_inc, D.B * D.Hq, a.tiles_per_head, nk, s);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  return H2O_OK;
}

// h2o_update_policy (insert = false) and h2o_evict_insert (insert = true:
// score_inc is not read and may be NULL).  With q8 (the 8-bit buffer calls)
// k_cache / v_cache are NULL: the update kernel writes scores, positions and
// evict_idx (set to -1 first), then kv_scatter_q8 quantises the chunk's rows
// into the chosen slots.
int update_impl(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
                const float* score_inc, const h2o_bf16* k_new, const h2o_bf16* v_new,
                h2o_bf16* k_cache, h2o_bf16* v_cache, int32_t budget, int32_t recent_window,
                int32_t policy, int32_t* evict_idx, void* stream, bool insert,
                const Q8Buffers* q8 = nullptr) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (!scores || !slot_pos || (!insert && !score_inc) || !k_new || !v_new ||
      (!q8 && (!k_cache || !v_cache)) || (q8 && !evict_idx))
    return H2O_ERR_NULL;
  if (misaligned(scores) || misaligned(slot_pos) || misaligned(score_inc) || misaligned(k_new) ||
      misaligned(v_new) || misaligned(k_cache) || misaligned(v_cache) ||
      (evict_idx && misaligned(evict_idx)))
    return H2O_ERR_ALIGN;
  if (budget != D.M) return H2O_ERR_ARG;
  if (policy != H2O_POLICY_H2O && policy != H2O_POLICY_NORM && policy != H2O_POLICY_ORIG)
    return H2O_ERR_ARG;
  if (D.M < 1 || D.S > D.M) return H2O_ERR_SHAPE;
  if (recent_window < 0 || recent_window > D.M) return H2O_ERR_ARG;
  if (D.M - std::max(0, recent_window - D.S) < D.S) return H2O_ERR_ARG;
  if (pos0 < 0 || pos0 + D.S >= (int64_t(1) << 31)) return H2O_ERR_ARG;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  UpdateArgs a;
  a.scores = scores; a.slot_pos = slot_pos; a.score_inc = insert ? nullptr : score_inc;
  a.k_new = k_new; a.v_new = v_new; a.k_cache = k_cache; a.v_cache = v_cache;
  a.evict_idx = evict_idx; a.err = di->err_word;
  a.B = D.B; a.Hq = D.Hq; a.Hkv = D.Hkv; a.d = D.d; a.S = D.S; a.M = D.M; a.qg = D.Hq / D.Hkv;
  a.pos0 = static_cast<int>(pos0);
  a.W = recent_window;
  a.policy = policy;
  a.insert = insert ? 1 : 0;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const size_t n_idx = static_cast<size_t>(D.B) * D.Hkv * D.S;
  cudaError_t e = cudaSuccess;
  if (q8) e = cudaMemsetAsync(evict_idx, 0xFF, n_idx * sizeof(int32_t), s);  // -1: no slot
  if (e == cudaSuccess) e = launch_update(a, s);
  if (e == cudaSuccess && q8) {
    Q8ScatterArgs qa;
    qa.evict_idx = evict_idx; qa.k_new = k_new; qa.v_new = v_new; qa.buf = *q8;
    qa.err = di->err_word;
    qa.B = D.B; qa.Hkv = D.Hkv; qa.d = D.d; qa.S = D.S; qa.M = D.M;
    e = launch_kv_scatter_q8(qa, s);
  }
  if (e != cudaSuccess) return cuda_fail(e);
  return H2O_OK;
}

// Bytes of one tensor of bf16 rows read back from 8-bit buffers (256-aligned);
// none when the decode kernels run (they read the codes themselves).
size_t q8_rows_bytes(const h2o_dims_t& D) {
  int split_len = 0, n_split = 0;
  size_t ws = 0;
  if (D.M == 0 || decode_plan(D.B, D.Hq, D.Hkv, D.d, D.S, D.M, &split_len, &n_split, &ws))
    return 0;
  const size_t b = static_cast<size_t>(D.B) * D.Hkv * static_cast<size_t>(D.M) * D.d * 2;
  return (b + 255) / 256 * 256;
}

bool q8_null(const int8_t* kc, const float* ks, const int8_t* vc, const float* vs) {
  return !kc || !ks || !vc || !vs;
}

bool q8_misaligned(const int8_t* kc, const float* ks, const int8_t* vc, const float* vs) {
  return misaligned(kc) || misaligned(ks) || misaligned(vc) || misaligned(vs);
}

// h2o_sdpa_chunk_q8 / h2o_sdpa_cache_q8: the head of the workspace takes the K
// and V rows read back to bf16, the rest is the attention's own workspace.
int sdpa_q8_impl(const h2o_dims_t* dims, int64_t pos0, float softmax_scale, const h2o_bf16* q,
                 const int8_t* k_codes, const float* k_scales, const int8_t* v_codes,
                 const float* v_scales, const h2o_bf16* k_new, const h2o_bf16* v_new,
                 const int32_t* slot_pos, h2o_bf16* out, float* score_inc, void* workspace,
                 size_t workspace_bytes, void* stream, bool cache_only) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (D.M > 0 && q8_null(k_codes, k_scales, v_codes, v_scales)) return H2O_ERR_NULL;
  if (D.M > 0 && q8_misaligned(k_codes, k_scales, v_codes, v_scales)) return H2O_ERR_ALIGN;
  size_t base = 0;
  if ((st = h2o_workspace_size(dims, &base)) != H2O_OK) return st;
  const size_t rows = q8_rows_bytes(D);
  const size_t need = 2 * rows + base;
  if (need > 0 && (!workspace || workspace_bytes < need)) return H2O_ERR_WORKSPACE;
  if (need > 0 && misaligned(workspace)) return H2O_ERR_ALIGN;
  uint8_t* w = static_cast<uint8_t*>(workspace);
  Q8Buffers b;
  b.k_codes = const_cast<int8_t*>(k_codes); b.k_scales = const_cast<float*>(k_scales);
  b.v_codes = const_cast<int8_t*>(v_codes); b.v_scales = const_cast<float*>(v_scales);
  b.k_rows = rows ? reinterpret_cast<uint16_t*>(w) : nullptr;
  b.v_rows = rows ? reinterpret_cast<uint16_t*>(w + rows) : nullptr;
  return sdpa_impl(dims, pos0, softmax_scale, q, b.k_rows, b.v_rows, k_new, v_new, slot_pos, out,
                   score_inc, base ? w + 2 * rows : nullptr, base ? workspace_bytes - 2 * rows : 0,
                   stream, cache_only, D.M > 0 ? &b : nullptr);
}

int update_q8_impl(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
                   const float* score_inc, const h2o_bf16* k_new, const h2o_bf16* v_new,
                   int8_t* k_codes, float* k_scales, int8_t* v_codes, float* v_scales,
                   int32_t budget, int32_t recent_window, int32_t policy, int32_t* evict_idx,
                   void* stream, bool insert) {
  const int st = check_dims(dims);
  if (st != H2O_OK) return st;
  if (q8_null(k_codes, k_scales, v_codes, v_scales)) return H2O_ERR_NULL;
  if (q8_misaligned(k_codes, k_scales, v_codes, v_scales)) return H2O_ERR_ALIGN;
  Q8Buffers b;
  b.k_codes = k_codes; b.k_scales = k_scales; b.v_codes = v_codes; b.v_scales = v_scales;
  b.k_rows = nullptr; b.v_rows = nullptr;
  return update_impl(dims, pos0, scores, slot_pos, score_inc, k_new, v_new, nullptr, nullptr,
                     budget, recent_window, policy, evict_idx, stream, insert, &b);
}

// Waits on an mbarrier nothing completes, with the bounded wait every kernel
// uses; when the limit runs out it records H2O_DEVERR_TIMEOUT and returns.
__global__ void selftest_wait_kernel(int* err, uint64_t limit_ns) {
  __shared__ uint64_t bar;
  __shared__ int abort_flag;
  if (threadIdx.x == 0) {
    bar_init(&bar, 1);  // one arrival expected; none ever comes
    abort_flag = 0;
    fence_bar_init();
  }
  __syncthreads();
  const bool ok = wait_bar(&bar, 0, &abort_flag, limit_ns);
  __syncthreads();
  if (threadIdx.x == 0 && !ok) atomicOr(err, H2O_DEVERR_TIMEOUT);
}

}  // namespace
}  // namespace h2o

using namespace h2o;

extern "C" {

int h2o_version(void) { return 100; }

const char* h2o_status_string(int s) {
  switch (s) {
    case H2O_OK: return "ok";
    case H2O_ERR_NULL: return "a required pointer is NULL";
    case H2O_ERR_SHAPE: return "inconsistent or out-of-range sizes";
    case H2O_ERR_ALIGN: return "a pointer is not 16-byte aligned";
    case H2O_ERR_UNSUPPORTED: return "unsupported configuration (head dim must be 64 or 128)";
    case H2O_ERR_WORKSPACE: return "workspace missing or too small";
    case H2O_ERR_ARG: return "bad scalar argument (position, budget or recent window)";
    case H2O_ERR_CUDA: return "a CUDA runtime call failed (see h2o_last_cuda_error)";
    case H2O_ERR_TIMEOUT: return "a device-side bounded wait ran out";
    case H2O_ERR_DEVICE: return "device-side error (fewer eviction candidates than S)";
    case H2O_ERR_NODEVICE: return "no usable sm_100-family GPU is current";
    case H2O_ERR_BLAS: return "reserved (no call returns it)";
    default: return "unknown status";
  }
}

int h2o_last_cuda_error(void) { return t_last_cuda_error; }

int h2o_workspace_size(const h2o_dims_t* dims, size_t* bytes) {
  const int st = check_dims(dims);
  if (st != H2O_OK) return st;
  if (!bytes) return H2O_ERR_NULL;
  int split_len = 0, n_split = 0;
  size_t ws = 0;
  const h2o_dims_t& D = *dims;
  *bytes = decode_plan(D.B, D.Hq, D.Hkv, D.d, D.S, D.M, &split_len, &n_split, &ws)
               ? ws
               : sdpa_colpart_bytes(D.B, D.Hq, D.S, D.M);
  return H2O_OK;
}

int h2o_sdpa_chunk(const h2o_dims_t* dims, int64_t pos0, float softmax_scale, const h2o_bf16* q,
                   const h2o_bf16* k_cache, const h2o_bf16* v_cache, const h2o_bf16* k_new,
                   const h2o_bf16* v_new, const int32_t* slot_pos, h2o_bf16* out,
                   float* score_inc, void* workspace, size_t workspace_bytes, void* stream) {
  return sdpa_impl(dims, pos0, softmax_scale, q, k_cache, v_cache, k_new, v_new, slot_pos, out,
                   score_inc, workspace, workspace_bytes, stream, false);
}

int h2o_sdpa_chunk_lse(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                       const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                       const h2o_bf16* k_new, const h2o_bf16* v_new, const int32_t* slot_pos,
                       h2o_bf16* out, float* score_inc, float* lse, void* workspace,
                       size_t workspace_bytes, void* stream) {
  if (!lse) return H2O_ERR_NULL;
  return sdpa_impl(dims, pos0, softmax_scale, q, k_cache, v_cache, k_new, v_new, slot_pos, out,
                   score_inc, workspace, workspace_bytes, stream, false, nullptr, nullptr, lse);
}

int h2o_sdpa_cache(const h2o_dims_t* dims, int64_t pos0, float softmax_scale, const h2o_bf16* q,
                   const h2o_bf16* k_cache, const h2o_bf16* v_cache, const int32_t* slot_pos,
                   h2o_bf16* out, float* score_inc, void* workspace, size_t workspace_bytes,
                   void* stream) {
  if (dims && dims->M < 1) return H2O_ERR_SHAPE;
  return sdpa_impl(dims, pos0, softmax_scale, q, k_cache, v_cache, nullptr, nullptr, slot_pos,
                   out, score_inc, workspace, workspace_bytes, stream, true);
}

int h2o_sdpa_decode_static(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                           const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                           const h2o_bf16* k_new, const h2o_bf16* v_new, const int32_t* slot_pos,
                           h2o_bf16* out, float* score_inc, void* stream) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (!q || !k_cache || !v_cache || !k_new || !v_new || !slot_pos || !out || !score_inc)
    return H2O_ERR_NULL;
  if (misaligned(q) || misaligned(k_cache) || misaligned(v_cache) || misaligned(k_new) ||
      misaligned(v_new) || misaligned(slot_pos) || misaligned(out) || misaligned(score_inc))
    return H2O_ERR_ALIGN;
  if (pos0 < 0 || pos0 + D.S >= (int64_t(1) << 31)) return H2O_ERR_ARG;
  if (!(softmax_scale <= 0.f) && !std::isfinite(softmax_scale)) return H2O_ERR_ARG;
  int split_len = 0, n_split = 0;
  size_t ws_need = 0;
  if (!decode_plan(D.B, D.Hq, D.Hkv, D.d, D.S, D.M, &split_len, &n_split, &ws_need))
    return H2O_ERR_UNSUPPORTED;
  if (ws_need > kDecodeStaticScratchBytes) return H2O_ERR_WORKSPACE;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  StaticScratch& ss = g_static_scratch[dev];  // dev < kMaxDevices: current_device checked it
  std::call_once(ss.once, [&ss] { ss.status = decode_static_scratch(&ss.ptr); });
  if (ss.status != cudaSuccess) return cuda_fail(ss.status);

  const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt(static_cast<float>(D.d));
  DecodeArgs a{};
  a.q = q; a.k_cache = k_cache; a.v_cache = v_cache; a.k_new = k_new; a.v_new = v_new;
  a.slot_pos = slot_pos; a.out = out; a.score_inc = score_inc;
  a.part = static_cast<float*>(ss.ptr);
  a.err = di->err_word;
  a.B = D.B; a.Hq = D.Hq; a.Hkv = D.Hkv; a.d = D.d; a.M = D.M; a.qg = D.Hq / D.Hkv;
  a.pos0 = static_cast<int>(pos0);
  a.scale_log2 = scale * 1.4426950408889634f;
  a.split_len = split_len;
  a.n_split = n_split;
  a.with_new = 1;
  a.nk = D.M + 1;
  if ((st = decode_maps(a)) != H2O_OK) return st;
  e = launch_decode(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_update(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
               const float* score_inc, const h2o_bf16* k_new, const h2o_bf16* v_new,
               h2o_bf16* k_cache, h2o_bf16* v_cache, int32_t budget, int32_t recent_window,
               int32_t* evict_idx, void* stream) {
  return h2o_update_policy(dims, pos0, scores, slot_pos, score_inc, k_new, v_new, k_cache,
                           v_cache, budget, recent_window, H2O_POLICY_H2O, evict_idx, stream);
}

int h2o_update_policy(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
                      const float* score_inc, const h2o_bf16* k_new, const h2o_bf16* v_new,
                      h2o_bf16* k_cache, h2o_bf16* v_cache, int32_t budget,
                      int32_t recent_window, int32_t policy, int32_t* evict_idx, void* stream) {
  return update_impl(dims, pos0, scores, slot_pos, score_inc, k_new, v_new, k_cache, v_cache,
                     budget, recent_window, policy, evict_idx, stream, false);
}

int h2o_evict_insert(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
                     const h2o_bf16* k_new, const h2o_bf16* v_new, h2o_bf16* k_cache,
                     h2o_bf16* v_cache, int32_t budget, int32_t recent_window, int32_t policy,
                     int32_t* evict_idx, void* stream) {
  return update_impl(dims, pos0, scores, slot_pos, nullptr, k_new, v_new, k_cache, v_cache,
                     budget, recent_window, policy, evict_idx, stream, true);
}

int h2o_scores_add(const h2o_dims_t* dims, float* scores, const float* score_inc, void* stream) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (D.M < 1) return H2O_ERR_SHAPE;
  if (!scores || !score_inc) return H2O_ERR_NULL;
  if (misaligned(scores) || misaligned(score_inc)) return H2O_ERR_ALIGN;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  ScoresAddArgs a;
  a.scores = scores;
  a.score_inc = score_inc;
  a.B = D.B; a.Hkv = D.Hkv; a.M = D.M; a.qg = D.Hq / D.Hkv;
  const cudaError_t e = launch_scores_add(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_kv_replace(const h2o_dims_t* dims, int64_t pos0, const int32_t* index,
                   const h2o_bf16* k_new, const h2o_bf16* v_new, h2o_bf16* k_cache,
                   h2o_bf16* v_cache, int32_t* slot_pos, h2o_bf16* delta_k, h2o_bf16* delta_v,
                   int32_t* delta_pos, void* stream) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (D.M < 1 || D.S > D.M) return H2O_ERR_SHAPE;
  if (!index || !k_new || !v_new || !k_cache || !v_cache) return H2O_ERR_NULL;
  if ((delta_k == nullptr) != (delta_v == nullptr)) return H2O_ERR_NULL;
  if (misaligned(index) || misaligned(k_new) || misaligned(v_new) || misaligned(k_cache) ||
      misaligned(v_cache) || misaligned(slot_pos) || misaligned(delta_k) ||
      misaligned(delta_v) || misaligned(delta_pos))
    return H2O_ERR_ALIGN;
  if (pos0 < 0 || pos0 + D.S >= (int64_t(1) << 31)) return H2O_ERR_ARG;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  ReplayArgs a;
  a.index = index; a.k_new = k_new; a.v_new = v_new; a.k_cache = k_cache; a.v_cache = v_cache;
  a.slot_pos = slot_pos; a.delta_k = delta_k; a.delta_v = delta_v;
  a.delta_pos = slot_pos ? delta_pos : nullptr;
  a.err = di->err_word;
  a.B = D.B; a.Hkv = D.Hkv; a.d = D.d; a.S = D.S; a.M = D.M;
  a.pos0 = static_cast<int>(pos0);
  a.restore = 0;
  const cudaError_t e = launch_kv_rows(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_kv_restore(const h2o_dims_t* dims, const int32_t* index, const h2o_bf16* delta_k,
                   const h2o_bf16* delta_v, const int32_t* delta_pos, h2o_bf16* k_cache,
                   h2o_bf16* v_cache, int32_t* slot_pos, void* stream) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (D.M < 1 || D.S > D.M) return H2O_ERR_SHAPE;
  if (!index || !delta_k || !delta_v || !k_cache || !v_cache) return H2O_ERR_NULL;
  if (misaligned(index) || misaligned(delta_k) || misaligned(delta_v) || misaligned(k_cache) ||
      misaligned(v_cache) || misaligned(slot_pos) || misaligned(delta_pos))
    return H2O_ERR_ALIGN;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  ReplayArgs a;
  a.index = index; a.k_new = nullptr; a.v_new = nullptr; a.k_cache = k_cache;
  a.v_cache = v_cache; a.slot_pos = slot_pos;
  a.delta_k = const_cast<h2o_bf16*>(delta_k); a.delta_v = const_cast<h2o_bf16*>(delta_v);
  a.delta_pos = const_cast<int32_t*>(delta_pos);
  a.err = di->err_word;
  a.B = D.B; a.Hkv = D.Hkv; a.d = D.d; a.S = D.S; a.M = D.M;
  a.pos0 = 0;
  a.restore = 1;
  const cudaError_t e = launch_kv_rows(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_kv_quantize(int64_t n_rows, int32_t d, const h2o_bf16* x, int8_t* codes, float* scales,
                    void* stream) {
  if (n_rows < 0) return H2O_ERR_SHAPE;
  if (d != 64 && d != 128) return H2O_ERR_UNSUPPORTED;
  if (n_rows == 0) return H2O_OK;
  if (!x || !codes || !scales) return H2O_ERR_NULL;
  if (misaligned(x) || misaligned(codes) || misaligned(scales)) return H2O_ERR_ALIGN;
  DeviceInfo* di = nullptr;
  const int st = current_device(&di);
  if (st != H2O_OK) return st;
  const cudaError_t e = launch_kv_quantize(x, codes, scales, n_rows, d,
                                           static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_kv_dequantize(int64_t n_rows, int32_t d, const int8_t* codes, const float* scales,
                      h2o_bf16* x, void* stream) {
  if (n_rows < 0) return H2O_ERR_SHAPE;
  if (d != 64 && d != 128) return H2O_ERR_UNSUPPORTED;
  if (n_rows == 0) return H2O_OK;
  if (!x || !codes || !scales) return H2O_ERR_NULL;
  if (misaligned(x) || misaligned(codes) || misaligned(scales)) return H2O_ERR_ALIGN;
  DeviceInfo* di = nullptr;
  const int st = current_device(&di);
  if (st != H2O_OK) return st;
  const cudaError_t e = launch_kv_dequantize(codes, scales, x, nullptr, nullptr, nullptr, n_rows,
                                             d, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_q8_workspace_size(const h2o_dims_t* dims, size_t* bytes) {
  const int st = h2o_workspace_size(dims, bytes);
  if (st != H2O_OK) return st;
  *bytes += 2 * q8_rows_bytes(*dims);
  return H2O_OK;
}

int h2o_sdpa_chunk_q8(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                      const h2o_bf16* q, const int8_t* k_codes, const float* k_scales,
                      const int8_t* v_codes, const float* v_scales, const h2o_bf16* k_new,
                      const h2o_bf16* v_new, const int32_t* slot_pos, h2o_bf16* out,
                      float* score_inc, void* workspace, size_t workspace_bytes, void* stream) {
  return sdpa_q8_impl(dims, pos0, softmax_scale, q, k_codes, k_scales, v_codes, v_scales, k_new,
                      v_new, slot_pos, out, score_inc, workspace, workspace_bytes, stream, false);
}

int h2o_sdpa_cache_q8(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                      const h2o_bf16* q, const int8_t* k_codes, const float* k_scales,
                      const int8_t* v_codes, const float* v_scales, const int32_t* slot_pos,
                      h2o_bf16* out, float* score_inc, void* workspace, size_t workspace_bytes,
                      void* stream) {
  if (dims && dims->M < 1) return H2O_ERR_SHAPE;
  return sdpa_q8_impl(dims, pos0, softmax_scale, q, k_codes, k_scales, v_codes, v_scales,
                      nullptr, nullptr, slot_pos, out, score_inc, workspace, workspace_bytes,
                      stream, true);
}

int h2o_update_q8(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
                  const float* score_inc, const h2o_bf16* k_new, const h2o_bf16* v_new,
                  int8_t* k_codes, float* k_scales, int8_t* v_codes, float* v_scales,
                  int32_t budget, int32_t recent_window, int32_t policy, int32_t* evict_idx,
                  void* stream) {
  return update_q8_impl(dims, pos0, scores, slot_pos, score_inc, k_new, v_new, k_codes, k_scales,
                        v_codes, v_scales, budget, recent_window, policy, evict_idx, stream,
                        false);
}

int h2o_evict_insert_q8(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
                        const h2o_bf16* k_new, const h2o_bf16* v_new, int8_t* k_codes,
                        float* k_scales, int8_t* v_codes, float* v_scales, int32_t budget,
                        int32_t recent_window, int32_t policy, int32_t* evict_idx,
                        void* stream) {
  return update_q8_impl(dims, pos0, scores, slot_pos, nullptr, k_new, v_new, k_codes, k_scales,
                        v_codes, v_scales, budget, recent_window, policy, evict_idx, stream,
                        true);
}

int h2o_backward_workspace_size(const h2o_dims_t* dims, size_t* bytes) {
  const int st = check_dims(dims);
  if (st != H2O_OK) return st;
  if (!bytes) return H2O_ERR_NULL;
  *bytes = backward_workspace_bytes(dims->B, dims->Hq, dims->Hkv, dims->S, dims->M);
  return H2O_OK;
}

// h2o_sdpa_chunk_backward (lse_saved = NULL: the rows' log-sum-exp is
// recomputed by the forward kernel's first pass, which also forms D) and
// h2o_sdpa_chunk_backward_lse (the forward's saved lse; a row kernel forms D).
static int backward_impl(const h2o_dims_t* dims, int64_t pos0, float softmax_scale, const h2o_bf16* q,
                  const h2o_bf16* k_cache, const h2o_bf16* v_cache, const h2o_bf16* k_new,
                  const h2o_bf16* v_new, const int32_t* slot_pos, const h2o_bf16* out,
                  const h2o_bf16* dout, const float* lse_saved, float* dq, float* dk_cache,
                  float* dv_cache, float* dk_new, float* dv_new, void* workspace,
                  size_t workspace_bytes, void* stream, bool with_lse) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  const h2o_dims_t& D = *dims;
  if (!q || !k_new || !v_new || !out || !dout || !dq || !dk_new || !dv_new) return H2O_ERR_NULL;
  if (with_lse && !lse_saved) return H2O_ERR_NULL;
  if (D.M > 0 && (!k_cache || !v_cache || !slot_pos || !dk_cache || !dv_cache))
    return H2O_ERR_NULL;
  if (misaligned(q) || misaligned(k_cache) || misaligned(v_cache) || misaligned(k_new) ||
      misaligned(v_new) || misaligned(slot_pos) || misaligned(out) || misaligned(dout) ||
      misaligned(dq) || misaligned(dk_cache) || misaligned(dv_cache) || misaligned(dk_new) ||
      misaligned(dv_new) || misaligned(workspace) || misaligned(lse_saved))
    return H2O_ERR_ALIGN;
  if (pos0 < 0 || pos0 + D.S >= (int64_t(1) << 31)) return H2O_ERR_ARG;
  if (!(softmax_scale <= 0.f) && !std::isfinite(softmax_scale)) return H2O_ERR_ARG;
  const int qg = D.Hq / D.Hkv;
  const int R = qg * D.S;                        // stacked query rows of a group
  if ((R + kTileM - 1) / kTileM > kMaxKeyTiles) return H2O_ERR_UNSUPPORTED;
  if (!workspace || workspace_bytes < backward_workspace_bytes(D.B, D.Hq, D.Hkv, D.S, D.M))
    return H2O_ERR_WORKSPACE;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  if ((st = get_encoder()) != H2O_OK) return st;
  const float scale = softmax_scale > 0.f ? softmax_scale : 1.0f / std::sqrt(static_cast<float>(D.d));
  BackwardArgs a;
  std::memset(&a, 0, sizeof(a));
  a.slot_pos = slot_pos;
  a.dq = dq; a.dk_cache = dk_cache; a.dv_cache = dv_cache; a.dk_new = dk_new; a.dv_new = dv_new;
  a.err = di->err_word;
  a.B = D.B; a.Hq = D.Hq; a.Hkv = D.Hkv; a.d = D.d; a.S = D.S; a.M = D.M; a.qg = qg;
  a.pos0 = static_cast<int>(pos0);
  a.scale = scale;
  a.scale_log2 = scale * 1.4426950408889634f;
  const int Rp = backward_row_stride(qg, D.S);
  const uint64_t G = static_cast<uint64_t>(D.B) * D.Hkv;
  a.lse = static_cast<float*>(workspace);
  a.drow = a.lse + G * Rp;
  {
    // 128-row boxes of the stacked query rows and of the key / value rows
    const uint32_t box[3] = {64, static_cast<uint32_t>(kTileM), 1};
    const uint64_t dr[3] = {static_cast<uint64_t>(D.d), static_cast<uint64_t>(R), G};
    const uint64_t dn[3] = {static_cast<uint64_t>(D.d), static_cast<uint64_t>(D.S), G};
    if ((st = encode(&a.tm_q, q, 3, dr, box)) != H2O_OK) return st;
    if ((st = encode(&a.tm_do, dout, 3, dr, box)) != H2O_OK) return st;
    if ((st = encode(&a.tm_kn, k_new, 3, dn, box)) != H2O_OK) return st;
    if ((st = encode(&a.tm_vn, v_new, 3, dn, box)) != H2O_OK) return st;
    if (D.M > 0) {
      const uint64_t dc[3] = {static_cast<uint64_t>(D.d), static_cast<uint64_t>(D.M), G};
      if ((st = encode(&a.tm_kc, k_cache, 3, dc, box)) != H2O_OK) return st;
      if ((st = encode(&a.tm_vc, v_cache, 3, dc, box)) != H2O_OK) return st;
    }
  }
  if (with_lse) {
    // the saved lse and D = dout . out, into the padded row layout
    cudaError_t e = launch_backward_rows(a, out, dout, lse_saved, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e);
    e = launch_backward(a, static_cast<cudaStream_t>(stream));
    return e == cudaSuccess ? H2O_OK : cuda_fail(e);
  }
  // each row's log-sum-exp and D = dout . out, from the forward kernel's
  // first pass
  SdpaArgs req;
  std::memset(&req, 0, sizeof(req));
  req.lse = a.lse;
  req.lse_stride = Rp;
  req.bwd_out = out;
  req.bwd_dout = dout;
  req.drow = a.drow;
  st = sdpa_impl(dims, pos0, softmax_scale, q, k_cache, v_cache, k_new, v_new, slot_pos, nullptr,
                 nullptr, nullptr, 0, stream, false, nullptr, &req);
  if (st != H2O_OK) return st;
  const cudaError_t e = launch_backward(a, static_cast<cudaStream_t>(stream));
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_sdpa_chunk_backward(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                            const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                            const h2o_bf16* k_new, const h2o_bf16* v_new,
                            const int32_t* slot_pos, const h2o_bf16* out,
                            const h2o_bf16* dout, float* dq, float* dk_cache, float* dv_cache,
                            float* dk_new, float* dv_new, void* workspace,
                            size_t workspace_bytes, void* stream) {
  return backward_impl(dims, pos0, softmax_scale, q, k_cache, v_cache, k_new, v_new, slot_pos, out,
                       dout, nullptr, dq, dk_cache, dv_cache, dk_new, dv_new, workspace,
                       workspace_bytes, stream, false);
}

int h2o_sdpa_chunk_backward_lse(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                                const h2o_bf16* q, const h2o_bf16* k_cache,
                                const h2o_bf16* v_cache, const h2o_bf16* k_new,
                                const h2o_bf16* v_new, const int32_t* slot_pos,
                                const h2o_bf16* out, const h2o_bf16* dout, const float* lse,
                                float* dq, float* dk_cache, float* dv_cache, float* dk_new,
                                float* dv_new, void* workspace, size_t workspace_bytes,
                                void* stream) {
  return backward_impl(dims, pos0, softmax_scale, q, k_cache, v_cache, k_new, v_new, slot_pos, out,
                       dout, lse, dq, dk_cache, dv_cache, dk_new, dv_new, workspace,
                       workspace_bytes, stream, true);
}

int h2o_cache_reset(const h2o_dims_t* dims, int32_t* slot_pos, float* scores, void* stream) {
  int st = check_dims(dims);
  if (st != H2O_OK) return st;
  if (dims->M < 1) return H2O_ERR_SHAPE;
  if (!slot_pos || !scores) return H2O_ERR_NULL;
  if (misaligned(slot_pos) || misaligned(scores)) return H2O_ERR_ALIGN;
  DeviceInfo* di = nullptr;
  if ((st = current_device(&di)) != H2O_OK) return st;
  const size_t n = static_cast<size_t>(dims->B) * dims->Hkv * dims->M;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  cudaError_t e = cudaMemsetAsync(slot_pos, 0xFF, n * sizeof(int32_t), s);
  if (e == cudaSuccess) e = cudaMemsetAsync(scores, 0, n * sizeof(float), s);
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_selftest_bounded_wait(int64_t limit_ns, void* stream) {
  if (limit_ns < 1000 || limit_ns > 100000000) return H2O_ERR_ARG;  // 1 us .. 100 ms
  DeviceInfo* di = nullptr;
  const int st = current_device(&di);
  if (st != H2O_OK) return st;
  selftest_wait_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(
      di->err_word, static_cast<uint64_t>(limit_ns));
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? H2O_OK : cuda_fail(e);
}

int h2o_device_errors(void) {
  DeviceInfo* di = nullptr;
  const int st = current_device(&di);
  if (st != H2O_OK) return st;
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e);
  int bits = 0;
  e = cudaMemcpy(&bits, di->err_word, sizeof(int), cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_fail(e);
  if (bits) {
    const int zero = 0;
    e = cudaMemcpy(di->err_word, &zero, sizeof(int), cudaMemcpyHostToDevice);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  return bits;
}

}  // extern "C"
