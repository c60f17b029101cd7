// Internal interface between the C-ABI layer (h2o_api.cu) and the kernels.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <mutex>

#include "../../include/h2o.h"

namespace h2o {

constexpr int kMaxDevices = 64;

// Runs a set-up step (a kernel attribute, an occupancy query) once per device,
// the first time any host thread needs it there, and remembers its status.
// The function receives the device ordinal and returns a cudaError_t.
struct OncePerDevice {
  std::once_flag once[kMaxDevices];
  cudaError_t status[kMaxDevices] = {};
  template <typename F>
  cudaError_t run(F&& f) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::call_once(once[dev], [&] { status[dev] = f(dev); });
    return status[dev];
  }
};

constexpr int kTileM = 128;        // query rows per CTA (tcgen05 M)
constexpr int kTileN = 128;        // keys per tile (tcgen05 N of Q K^T, K of P V)
constexpr int kMaxKeyTiles = 4096; // cache tiles + chunk tiles a CTA may visit
constexpr uint64_t kWaitLimitNs = 2000000000ull;  // bounded waits: 2 s

struct SdpaArgs {
  CUtensorMap tm_q;        // 4D {d, S, q_g, B*Hkv}, box {64, rows_box, heads_box, 1}
  CUtensorMap tm_kc;       // 3D {d, M, B*Hkv}, box {64, 64 (d = 128) or 128, 1}
  CUtensorMap tm_vc;       // 3D {d, M, B*Hkv}, box {64, 128, 1}
  CUtensorMap tm_kn;       // 3D {d, S, B*Hkv}, box as tm_kc
  CUtensorMap tm_vn;       // 3D {d, S, B*Hkv}, box as tm_vc
  const int32_t* slot_pos; // (B, Hkv, M)
  uint16_t* out;           // (B, Hq, S, d) bf16
  float* score_inc;        // (B, Hq, M + S)
  int* err;                // device error word
  int B, Hq, Hkv, d, S, M, qg;
  int pos0;
  float scale_log2;        // softmax scale * log2(e)
  int rows_box;            // query rows per head in a tile (S_pad when S <= 128, else 128)
  int heads_box;           // query heads per tile (1 when S > 128)
  int tiles_per_head;      // ceil(S / 128) when S > 128, else 0
  int n_row_tiles;         // CTAs per (b, kv head)
  int n_cache_tiles;       // ceil(M / 128)
  int n_chunk_tiles;       // ceil(S / 128); 0 for h2o_sdpa_cache (keys in the cache only)
  int nk;                  // key columns of a score_inc row: M + S, or M for h2o_sdpa_cache
  // Column-sum partials, one row per (b, query head, row tile of that head):
  // (B * Hq, tiles_per_head, nk) fp32 in the caller's workspace, or null.
  // With three or more row tiles per head the kernel stores each tile's
  // column sums here (zeros for tiles it skips) and colsum_reduce adds them
  // in row-tile order, so score_inc does not depend on the order the CTAs
  // finish in; otherwise it adds into the zeroed score_inc directly (at most
  // two addends per element onto an exact zero, which commute).
  float* colpart;
  // Non-null: pass 1 only.  The kernel writes every query row's log-sum-exp
  // of the scaled logits in log2 units, lse[(b Hkv + h) lse_stride + g S + i]
  // for query head h q_g + g, and nothing else (the backward's softmax
  // recomputation needs it).
  float* lse;
  int lse_stride;
  // With lse: when drow is non-null, also D = dout . out (fp32) of every
  // query row, at the same index as its log-sum-exp; out / dout (B, Hq, S, d)
  // bf16 are the forward output and the loss gradient the backward is given.
  const uint16_t* bwd_out;
  const uint16_t* bwd_dout;
  float* drow;
  // Full mode: when non-null, each query row's log-sum-exp of the scaled
  // logits (natural log), (B, Hq, S) fp32, as the forward's own lambda.
  float* lse_out;
};

// Row tiles per query head above which the column sums go through colpart.
constexpr int kColpartMinTiles = 3;

// Bytes of colpart for a chunk of S queries against M slots (0 when the
// column sums are added into score_inc directly).
size_t sdpa_colpart_bytes(int B, int Hq, int S, int M);

// score_inc[row, j] = sum over r = 0 .. tph-1 (in that order) of
// colpart[row, r, j], for rows = B * Hq and j < nk.
cudaError_t launch_colsum_reduce(const float* colpart, float* score_inc, int rows, int tph, int nk,
                                 cudaStream_t stream);

struct UpdateArgs {
  float* scores;
  int32_t* slot_pos;
  const float* score_inc;
  const uint16_t* k_new;
  const uint16_t* v_new;
  uint16_t* k_cache;
  uint16_t* v_cache;
  int32_t* evict_idx;      // may be null
  int* err;
  int B, Hq, Hkv, d, S, M, qg;
  int pos0;
  int W;
  int policy;              // H2O_POLICY_*
  int insert;              // 1: h2o_evict_insert (rank on scores as they are, no score_inc;
                           //    the new slots score 0; h2o_norm's t is pos0)
};

struct ScoresAddArgs {
  float* scores;           // (B, Hkv, M) in/out
  const float* score_inc;  // (B, Hq, M)
  int B, Hkv, M, qg;
};

// S = 1 (one query token per sequence): split-K decode kernels.
constexpr int kDecodeMaxQg = 8;         // larger GQA groups take the chunk kernel
constexpr int kDecodeMaxSplitLen = 1536;
constexpr int kDecodeMinSplitLen = 128;
constexpr int kDecodeResidentCtas = 304;     // split-kernel CTAs resident on a GB300 (2 x 152)
constexpr int kDecodeTcCtas = 152;           // tensor-core split kernel: one CTA per GB300 SM
constexpr int kDecodeTcTileKeys = 128;       // its K / V tiles (split lengths are multiples)
// its per-item cost, in keys of streaming (the items of a CTA overlap, K
// tiles of one with V tiles of the previous)
constexpr int kDecodeTcItemOverheadKeys = 16;
constexpr int kDecodeTcMaxSplitLen = 1024;   // its largest split (two items' logits in shared memory)
// and its smallest: the end of a phase costs ~1400 cycles that a phase of
// fewer than four tiles per stream no longer hides (measured)
constexpr int kDecodeTcMinSplitLen = 512;
constexpr int kDecodeItemOverheadKeys = 32;  // per-item cost, in keys, for choosing the split

struct DecodeArgs {
  // tensor-core path (d = 128): TMA maps of q {d, Hq, B} with box {64, 16, 1}
  // and of the cache K / V {d, M, B*Hkv} with box {64, 128, 1} (bf16, 128-byte
  // swizzle); with 8-bit buffers tm_kc / tm_vc map the codes {d, M, B*Hkv}
  // (uint8, box {128, 128, 1}, no swizzle) and tm_ks / tm_vs the scales
  // {B*Hkv*M} (fp32, box {128})
  CUtensorMap tm_q, tm_kc, tm_vc, tm_ks, tm_vs;
  int tc;                   // 1: decode_tc_kernel (maps valid); 0: decode_split_kernel
  const uint16_t* q;        // (B, Hq, 1, d)
  const uint16_t* k_cache;  // (B, Hkv, M, d)
  const uint16_t* v_cache;
  const uint16_t* k_new;    // (B, Hkv, 1, d)
  const uint16_t* v_new;
  const int32_t* slot_pos;  // (B, Hkv, M)
  uint16_t* out;            // (B, Hq, 1, d) bf16
  float* score_inc;         // (B, Hq, M + 1): logits (log2 units), then weights
  float* part;              // (B, Hq, n_split, 2 + d): max, sum, unnormalised output
  int* err;
  int B, Hq, Hkv, d, M, qg;
  int pos0;
  float scale_log2;
  int split_len;            // cache slots per split (multiple of 16)
  int n_split;              // ceil(M / split_len); the last split also takes the new token
  int with_new;             // 1: the new token is key column M; 0: h2o_sdpa_cache (none)
  int nk;                   // score_inc row length: M + with_new
  // 8-bit buffers (q8 = 1): the cache rows are int8 codes with a float32 scale
  // per row, read as bf16(code * scale); k_cache / v_cache are then unused
  int q8;
  const int8_t* k_codes;    // (B, Hkv, M, d)
  const float* k_scales;    // (B, Hkv, M)
  const int8_t* v_codes;
  const float* v_scales;
};

// Split of the M cache slots for the decode kernels (a function of the sizes
// only, so that h2o_workspace_size and h2o_sdpa_chunk agree).  Returns false
// when the decode kernels do not apply (S != 1, M == 0 or q_g too large).
bool decode_plan(int B, int Hq, int Hkv, int d, int S, int M, int* split_len, int* n_split,
                 size_t* ws_bytes);

// Fixed scratch of h2o_sdpa_decode_static (a file-scope device array in
// h2o_decode.cu, shared by every call on a device): its size and its address
// on the current device.
constexpr size_t kDecodeStaticScratchBytes = size_t(16) << 20;
cudaError_t decode_static_scratch(void** ptr);

// h2o_kv_replace / h2o_kv_restore (h2o_replay.cu)
struct ReplayArgs {
  const int32_t* index;      // (B, Hkv, S) slots, distinct per (b, h)
  const uint16_t* k_new;     // (B, Hkv, S, d) replace only
  const uint16_t* v_new;
  uint16_t* k_cache;         // (B, Hkv, M, d) in/out
  uint16_t* v_cache;
  int32_t* slot_pos;         // (B, Hkv, M) in/out, may be null
  uint16_t* delta_k;         // (B, Hkv, S, d): out (replace, may be null) or in (restore)
  uint16_t* delta_v;
  int32_t* delta_pos;        // (B, Hkv, S): likewise, may be null
  int* err;
  int B, Hkv, d, S, M;
  int pos0;
  int restore;               // 0: replace, 1: restore
};

cudaError_t launch_kv_rows(const ReplayArgs& a, cudaStream_t stream);

// 8-bit K/V buffers (h2o_quant.cu): per cache row d int8 codes and one fp32
// scale.  The q8 calls pass the buffers and, for the SDPA, the bf16 rows the
// codes are read back into.
struct Q8Buffers {
  int8_t* k_codes;           // (B, Hkv, M, d)
  float* k_scales;           // (B, Hkv, M)
  int8_t* v_codes;
  float* v_scales;
  uint16_t* k_rows;          // SDPA only: (B, Hkv, M, d) bf16 read-back of the codes
  uint16_t* v_rows;
};

struct Q8ScatterArgs {
  const int32_t* evict_idx;  // (B, Hkv, S): slot of token c, -1 = none (left as it is)
  const uint16_t* k_new;     // (B, Hkv, S, d) bf16
  const uint16_t* v_new;
  Q8Buffers buf;
  int* err;
  int B, Hkv, d, S, M;
};

cudaError_t launch_kv_quantize(const uint16_t* x, int8_t* codes, float* scales, int64_t n_rows,
                               int d, cudaStream_t stream);
cudaError_t launch_kv_dequantize(const int8_t* codes, const float* scales, uint16_t* x,
                                 const int8_t* codes2, const float* scales2, uint16_t* x2,
                                 int64_t n_rows, int d, cudaStream_t stream);
cudaError_t launch_kv_scatter_q8(const Q8ScatterArgs& a, cudaStream_t stream);

// h2o_sdpa_chunk_backward (h2o_backward.cu): fused tcgen05 kernels, no
// materialised score matrices.  The workspace holds, per stacked query row of
// each (b, kv head) group, the row's log-sum-exp (log2 units, from the
// forward kernel's pass 1) and D = dout . out.
struct BackwardArgs {
  // TMA maps (box {64, 128, 1}, 128-byte swizzle): the stacked query rows of
  // a group {d, q_g S, B Hkv} for q and dout, the keys and values {d, M or S,
  // B Hkv} of the cache and of the chunk
  CUtensorMap tm_q, tm_do, tm_kc, tm_vc, tm_kn, tm_vn;
  const int32_t* slot_pos;   // (B, Hkv, M)
  float* dq;                 // (B, Hq, S, d) fp32
  float* dk_cache;           // (B, Hkv, M, d) fp32
  float* dv_cache;
  float* dk_new;             // (B, Hkv, S, d) fp32
  float* dv_new;
  float* lse;                // (B Hkv, R_pad): per stacked row g S + i of a group, its
                             // log-sum-exp (log2 units); R_pad = q_g S rounded up to 128
  float* drow;               // (B Hkv, R_pad): D per stacked row
  int* err;
  int B, Hq, Hkv, d, S, M, qg;
  int pos0;
  float scale;               // softmax scale
  float scale_log2;          // scale * log2(e)
};
// Rows of a group in the lse / drow layout: q_g S rounded up to 128, so that
// every 128-row tile of them starts 16-byte aligned.
__host__ __device__ inline int backward_row_stride(int qg, int S) { return (qg * S + 127) / 128 * 128; }
size_t backward_workspace_bytes(int B, int Hq, int Hkv, int S, int M);
// The forward's pass 1 must have filled a.lse and a.drow first.
cudaError_t launch_backward(const BackwardArgs& a, cudaStream_t stream);
// Fills a.lse (from a saved natural-log lse, (B, Hq, S)) and a.drow (from out
// and dout) in the backward's padded row layout.
cudaError_t launch_backward_rows(const BackwardArgs& a, const uint16_t* out, const uint16_t* dout,
                                 const float* lse_saved, cudaStream_t stream);
cudaError_t launch_sdpa(const SdpaArgs& a, cudaStream_t stream);
cudaError_t launch_decode(const DecodeArgs& a, cudaStream_t stream);
// The tensor-core split kernel (h2o_decode_tc.cu): same partials as
// decode_split_kernel; launch_decode runs the combine after it.
cudaError_t launch_decode_tc(const DecodeArgs& a, cudaStream_t stream);
cudaError_t launch_update(const UpdateArgs& a, cudaStream_t stream);
cudaError_t launch_scores_add(const ScoresAddArgs& a, cudaStream_t stream);

}  // namespace h2o
