/*
 * h2o.h - C ABI of the GB300 (sm_103a) H2O sparse-attention library.
 *
 * One attention layer with a fixed-size KV cache of M slots per (batch, KV
 * head), processed chunk by chunk (paper §3.1: prefill, then chunks of S
 * tokens).  Two calls make up one chunk step:
 *
 *   h2o_sdpa_chunk  the chunk's S queries attend to the M cache slots and,
 *                   causally, to the chunk's own keys (§3.1 Eq. 2 with the
 *                   position mask of §3.3.1); besides the attention output it
 *                   returns the summed attention weights sum_i m_ij per key
 *                   column (§3.3.1, §A.6), shape (B, H_q, M + S).
 *   h2o_update      adds those weights into the per-(batch, KV head) H2O
 *                   scores (§3.1.1 Eq. 3, summed over the query heads of the
 *                   GQA group), evicts the S lowest-scoring slots outside the
 *                   recent window and writes the chunk's keys and values into
 *                   them (the scatter of §3.2 / §A.1.1).
 *
 * With one query token per sequence (S = 1) h2o_sdpa_chunk runs split-K decode
 * kernels that need a workspace (h2o_workspace_size).  Further calls:
 *   h2o_update_policy                the h2o_norm / h2o_orig variants (§3.1.1)
 *   h2o_evict_insert, h2o_sdpa_cache, h2o_scores_add
 *                                    the paper's own order of a chunk step
 *                                    (write first, then attend; §3.1, §3.3.1)
 *   h2o_kv_replace, h2o_kv_restore   replay-cache row writes and the reverse
 *                                    recurrence (§3.2, §A.1.1)
 *   h2o_sdpa_chunk_lse, h2o_sdpa_chunk_backward, h2o_sdpa_chunk_backward_lse
 *                                    the gradient of one chunk's SDPA (given
 *                                    the forward's lse, or recomputing it)
 *   h2o_sdpa_decode_static           S = 1 SDPA on a fixed internal scratch
 *   h2o_kv_quantize, h2o_kv_dequantize, h2o_update_q8, h2o_evict_insert_q8,
 *   h2o_sdpa_chunk_q8, h2o_sdpa_cache_q8, h2o_q8_workspace_size
 *                                    8-bit K/V cache buffers (§4 setup)
 *
 * Conventions for every call:
 *  - All array arguments are DEVICE pointers, allocated and owned by the
 *    caller.  No call allocates device memory (the scratch of
 *    h2o_sdpa_decode_static and the error word are static device arrays) or
 *    keeps per-call state; every kernel is this library's own (no cuBLAS).
 *    Every array is dense, row-major (C order) with the shape given, and must
 *    be 16-byte aligned.
 *  - The library resolves some per-device state on its first call on a
 *    device (the error word's and the static scratch's addresses, kernel
 *    shared-memory limits, resident CTA counts) and keeps it until exit.
 *    A cudaDeviceReset() destroys the context that state belongs to: after
 *    one, no call of this library may be made on that device in the same
 *    process.
 *  - bf16 arrays hold IEEE bfloat16 bit patterns (h2o_bf16 = uint16_t).
 *  - Calls only enqueue work on `stream` (a cudaStream_t; NULL = legacy
 *    default stream) and return without synchronising.  Arguments are
 *    validated on the host first; on any error nothing is enqueued.
 *  - Stream order holds as usual, with one refinement: the update kernels,
 *    and the reduction and combine steps of the attention calls, are
 *    launched as programmatic dependents of the kernel before them.  If that
 *    kernel allows an early start (only this library's attention kernels
 *    do), they may begin while it finishes, reading before its completion
 *    only what it does not write (scores, slot_pos, k_new, v_new), and
 *    everything else after it has completed.
 *  - Return value: H2O_OK (0) or a negative H2O_ERR_* code; h2o_status_string
 *    gives a message.  For H2O_ERR_CUDA, h2o_last_cuda_error() gives the
 *    cudaError_t of the failing runtime call on this host thread.
 *  - Device-side problems (a bounded wait that ran out, fewer eviction
 *    candidates than S found in slot_pos) are recorded in a per-device error
 *    word; h2o_device_errors() synchronises the device and reads and clears it.
 *  - Token positions are int32; pos0 + S must stay below 2^31.
 */
#ifndef H2O_GB300_H2O_H_
#define H2O_GB300_H2O_H_

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define H2O_API __attribute__((visibility("default")))
#else
#define H2O_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t h2o_bf16;

/* Problem sizes of one layer.  Hq % Hkv == 0 (GQA, §3.1: query head hq uses
 * KV head hq / (Hq / Hkv)); d is the head dimension (64 or 128); S >= 1 is
 * the chunk length; M >= 0 is the number of cache slots. */
typedef struct h2o_dims {
  int32_t B, Hq, Hkv, d, S, M;
} h2o_dims_t;

enum {
  H2O_OK = 0,
  H2O_ERR_NULL = -1,        /* a required pointer is NULL */
  H2O_ERR_SHAPE = -2,       /* inconsistent or out-of-range sizes */
  H2O_ERR_ALIGN = -3,       /* a pointer is not 16-byte aligned */
  H2O_ERR_UNSUPPORTED = -4, /* valid request the library does not handle (e.g. d) */
  H2O_ERR_WORKSPACE = -5,   /* workspace NULL or smaller than h2o_workspace_size */
  H2O_ERR_ARG = -6,         /* bad scalar argument (window, budget, position) */
  H2O_ERR_CUDA = -7,        /* a CUDA runtime call failed; see h2o_last_cuda_error */
  H2O_ERR_TIMEOUT = -8,     /* device: a bounded wait ran out (reported by h2o_device_errors) */
  H2O_ERR_DEVICE = -9,      /* device: fewer eviction candidates than S, etc. */
  H2O_ERR_NODEVICE = -10,   /* no usable sm_100-family GPU is current */
  H2O_ERR_BLAS = -11        /* reserved: no call returns it */
};

/* Device error bits reported by h2o_device_errors(). */
enum {
  H2O_DEVERR_TIMEOUT = 1,   /* a kernel's bounded wait on a barrier ran out */
  H2O_DEVERR_CANDIDATES = 2, /* h2o_update found fewer than S evictable slots */
  H2O_DEVERR_INDEX = 4       /* h2o_kv_replace / h2o_kv_restore met an index outside [0, M) */
};

/* Bytes of scratch memory h2o_sdpa_chunk needs for `dims` (may be 0). */
H2O_API int h2o_workspace_size(const h2o_dims_t* dims, size_t* bytes);

/*
 * One chunk of sparse SDPA with summed attention weights (§3.1 Eq. 2, mask of
 * §3.3.1, summed weights of §3.3.1 / §A.6.1).
 *
 *   q         (B, Hq, S, d) bf16   queries of tokens pos0 .. pos0+S-1
 *   k_cache   (B, Hkv, M, d) bf16  cache keys   (may be NULL when M == 0)
 *   v_cache   (B, Hkv, M, d) bf16  cache values (may be NULL when M == 0)
 *   k_new     (B, Hkv, S, d) bf16  the chunk's keys
 *   v_new     (B, Hkv, S, d) bf16  the chunk's values
 *   slot_pos  (B, Hkv, M) int32    token position held by each slot, -1 = empty
 *   out       (B, Hq, S, d) bf16   attention output (written)
 *   score_inc (B, Hq, M + S) f32   summed weights sum_i m_ij (written): columns
 *                                  0..M-1 are the cache slots, M..M+S-1 the
 *                                  chunk's own tokens in order
 *
 * Query row i (token pos0 + i) sees cache slot j iff 0 <= slot_pos[j] <=
 * pos0 + i, and chunk token c iff c <= i.  softmax_scale <= 0 selects
 * d^-1/2.  Every query row must see at least one key (it always sees its own
 * token).  `workspace` may be NULL when h2o_workspace_size reports 0.
 */
H2O_API int h2o_sdpa_chunk(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                   const h2o_bf16* k_new, const h2o_bf16* v_new, const int32_t* slot_pos,
                   h2o_bf16* out, float* score_inc, void* workspace, size_t workspace_bytes,
                   void* stream);

/*
 * h2o_sdpa_chunk that also writes, for a later h2o_sdpa_chunk_backward_lse,
 * each query row's log-sum-exp of the visible scaled logits (§3.1 Eq. 2's
 * normaliser, natural log):
 *
 *   lse  (B, Hq, S) f32, written: lse[b, hq, i] = log sum_{j visible} exp(scale q_i . k_j)
 *
 * Other arguments, results and the workspace as for h2o_sdpa_chunk.  S = 1
 * also runs the chunk kernel here (the decode kernels keep no lse).
 */
H2O_API int h2o_sdpa_chunk_lse(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                   const h2o_bf16* k_new, const h2o_bf16* v_new, const int32_t* slot_pos,
                   h2o_bf16* out, float* score_inc, float* lse, void* workspace,
                   size_t workspace_bytes, void* stream);

/*
 * h2o_sdpa_chunk for one query token per sequence (dims->S == 1, M >= 1,
 * Hq / Hkv <= 8), with no workspace argument: it allocates nothing.  The
 * paper has no counterpart; this entry point exists for callers that cannot
 * allocate device memory around the call.
 *
 * Its scratch (the per-split partial max, sum and output of every query head,
 * h2o_workspace_size(dims) bytes) is a fixed device array of 16 MiB inside the
 * library, one per device; dims needing more are rejected with
 * H2O_ERR_WORKSPACE and nothing runs.  Other sizes outside the decode case
 * give H2O_ERR_UNSUPPORTED.  Arguments, outputs and the other errors are
 * those of h2o_sdpa_chunk.
 *
 *  - The first call on a device looks up the array's address on that device
 *    (with the device current); make that first call before any stream capture.
 *  - Every call on a device shares the one array: calls whose kernels overlap
 *    on the GPU (different streams, no ordering between them) race on it.
 *    Nothing in it needs to start at zero; each call writes every entry it
 *    reads.
 */
H2O_API int h2o_sdpa_decode_static(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                   const h2o_bf16* k_new, const h2o_bf16* v_new, const int32_t* slot_pos,
                   h2o_bf16* out, float* score_inc, void* stream);

/*
 * H2O cache update after h2o_sdpa_chunk (§3.1.1 Eq. 3 and the eviction rule
 * that follows it; scatter of §3.2 / §A.1.1).  Per (b, kv head h):
 *
 *   t_j   = score_inc[b, h*qg + 0, j] + ... + score_inc[b, h*qg + qg-1, j]
 *           (float32, added in ascending g, no fused multiply-add)
 *   acc_j = scores[b,h,j] + t_j                       for cache slots j < M
 *   candidates: slots with slot_pos < pos0 + S - recent_window (empty slots,
 *   position -1, always qualify); the S smallest under the total order
 *   (empty first, then acc ascending, then slot index ascending) are evicted;
 *   the c-th smallest evicted slot e receives token pos0 + c:
 *   k_cache[b,h,e,:] = k_new[b,h,c,:], v_cache likewise, slot_pos = pos0 + c,
 *   scores = t_{M+c}; every other slot keeps its K/V/position and gets acc_j.
 *
 *   scores    (B, Hkv, M) f32      in/out
 *   slot_pos  (B, Hkv, M) int32    in/out
 *   score_inc (B, Hq, M + S) f32   in (from h2o_sdpa_chunk)
 *   k_new, v_new (B, Hkv, S, d) bf16 in
 *   k_cache, v_cache (B, Hkv, M, d) bf16 in/out
 *   budget    must equal dims->M (the cache length N_C of the paper)
 *   recent_window  0 <= W <= M; needs M - max(0, W - S) >= S
 *   evict_idx (B, Hkv, S) int32    out, optional (NULL = not written): the
 *             slot that received token pos0 + c; this is the content of the
 *             paper's replay log / scatter index (§3.2)
 *
 * If a (b, h) has fewer than S candidates at run time (slot_pos not produced
 * by this policy), that (b, h) is left unchanged and H2O_DEVERR_CANDIDATES is
 * recorded.
 */
H2O_API int h2o_update(const h2o_dims_t* dims, int64_t pos0, float* scores, int32_t* slot_pos,
               const float* score_inc, const h2o_bf16* k_new, const h2o_bf16* v_new,
               h2o_bf16* k_cache, h2o_bf16* v_cache, int32_t budget, int32_t recent_window,
               int32_t* evict_idx, void* stream);

/* Eviction policies of §3.1.1 (h2o_update_policy). */
enum {
  H2O_POLICY_H2O = 0,  /* rank by the H2O score acc_j (what h2o_update does) */
  H2O_POLICY_NORM = 1, /* rank by the normalized score acc_j / (t - slot_pos_j),
                          t = pos0 + S the tokens processed once the chunk is
                          in; the division is float32, rounded to nearest, of
                          acc_j by the nearest float32 to t - slot_pos_j.  The
                          stored scores stay the unnormalized acc_j. */
  H2O_POLICY_ORIG = 2  /* one selection per KV head h shared by every batch
                          entry, ranked by sum_b acc_{b,h,j} (float32, ascending
                          b); candidates, empties and the recent window are read
                          from slot_pos[0, h, :], which must be identical across
                          b (it stays so when every update of the cache since
                          h2o_cache_reset used this policy).  Each batch entry
                          writes its own rows, scores and positions. */
};

/*
 * h2o_update with an explicit eviction policy (§3.1.1: the paper's h2o,
 * h2o_norm and h2o_orig).  Same arguments, layouts, ordering and errors as
 * h2o_update; `policy` is one of H2O_POLICY_* (H2O_ERR_ARG otherwise).
 * h2o_update(...) is h2o_update_policy(..., H2O_POLICY_H2O, ...).
 */
H2O_API int h2o_update_policy(const h2o_dims_t* dims, int64_t pos0, float* scores,
                              int32_t* slot_pos, const float* score_inc, const h2o_bf16* k_new,
                              const h2o_bf16* v_new, h2o_bf16* k_cache, h2o_bf16* v_cache,
                              int32_t budget, int32_t recent_window, int32_t policy,
                              int32_t* evict_idx, void* stream);

/*
 * The paper's own order of a chunk step (§3.1 last paragraph, §3.3.1): the
 * chunk's keys and values are written into the cache first, then SDPA runs
 * over the M = N_C slots with the mask "row i sees slot j iff
 * 0 <= slot_pos[j] <= pos0 + i", then the chunk's summed weights are added to
 * the scores.  Three calls per chunk, in this order:
 *
 *   h2o_evict_insert  per (b, kv head), the S slots with the smallest score
 *                     (before this chunk attends) under the rules of
 *                     h2o_update_policy (candidates, total order, policies;
 *                     h2o_norm's age is pos0 - slot_pos) take the chunk's
 *                     K/V; the c-th smallest gets token pos0 + c, score 0.
 *                     Every other slot is left as it is.  Arguments and
 *                     errors as h2o_update_policy, without score_inc.
 *   h2o_sdpa_cache    SDPA of the chunk's queries over the M slots only:
 *                     out (B, Hq, S, d) bf16 and score_inc (B, Hq, M) f32;
 *                     k_cache / v_cache / slot_pos as left by
 *                     h2o_evict_insert (every query row then sees at least
 *                     its own token).  M >= 1.  Workspace as for
 *                     h2o_sdpa_chunk with the same dims
 *                     (h2o_workspace_size).  Errors as h2o_sdpa_chunk.
 *   h2o_scores_add    scores[b,h,j] += score_inc[b,h*qg+0,j] + ... +
 *                     score_inc[b,h*qg+qg-1,j] (float32, ascending g, then
 *                     added to the score) for every slot j < M.
 */
H2O_API int h2o_evict_insert(const h2o_dims_t* dims, int64_t pos0, float* scores,
                   int32_t* slot_pos, const h2o_bf16* k_new, const h2o_bf16* v_new,
                   h2o_bf16* k_cache, h2o_bf16* v_cache, int32_t budget,
                   int32_t recent_window, int32_t policy, int32_t* evict_idx, void* stream);
H2O_API int h2o_sdpa_cache(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                   const int32_t* slot_pos, h2o_bf16* out, float* score_inc, void* workspace,
                   size_t workspace_bytes, void* stream);
H2O_API int h2o_scores_add(const h2o_dims_t* dims, float* scores, const float* score_inc,
                   void* stream);

/*
 * Replay-cache row operations (§3.2 recurrence, §A.1.1 scatter / gather):
 *
 *   h2o_kv_replace  for every (b, h, c): delta_k[b,h,c,:] = k_cache[b,h,e,:],
 *                   then k_cache[b,h,e,:] = k_new[b,h,c,:], e = index[b,h,c];
 *                   v likewise; slot_pos[b,h,e] := pos0 + c with its old value
 *                   to delta_pos[b,h,c].  This is the cache write of a chunk
 *                   whose eviction decisions are replayed from a log, keeping
 *                   the rows it replaces (delta_key = gather(keys, index)).
 *   h2o_kv_restore  the reverse recurrence: k_cache[b,h,e,:] = delta_k[b,h,c,:],
 *                   v likewise, slot_pos[b,h,e] = delta_pos[b,h,c].
 *
 *   index      (B, Hkv, S) int32, distinct within each (b, h); an entry
 *              outside [0, M) skips its row and records H2O_DEVERR_INDEX
 *   k_new, v_new (B, Hkv, S, d) bf16 (replace)
 *   k_cache, v_cache (B, Hkv, M, d) bf16, in place
 *   slot_pos   (B, Hkv, M) int32 in place, or NULL (positions untouched)
 *   delta_k, delta_v (B, Hkv, S, d) bf16: out of replace (both NULL: no
 *              gather), in of restore; delta_pos (B, Hkv, S) int32 likewise
 *              (NULL: positions are not saved / restored)
 * dims->Hq only has to be a multiple of dims->Hkv.
 */
H2O_API int h2o_kv_replace(const h2o_dims_t* dims, int64_t pos0, const int32_t* index,
                   const h2o_bf16* k_new, const h2o_bf16* v_new, h2o_bf16* k_cache,
                   h2o_bf16* v_cache, int32_t* slot_pos, h2o_bf16* delta_k, h2o_bf16* delta_v,
                   int32_t* delta_pos, void* stream);
H2O_API int h2o_kv_restore(const h2o_dims_t* dims, const int32_t* index,
                   const h2o_bf16* delta_k, const h2o_bf16* delta_v, const int32_t* delta_pos,
                   h2o_bf16* k_cache, h2o_bf16* v_cache, int32_t* slot_pos, void* stream);

/*
 * 8-bit K/V cache buffers (§4 setup: the KV cache buffers are stored in 8
 * bits; the format below is this library's, the paper names none).
 *
 * Every cache row of d elements (one token's key, or its value, in one KV
 * head) is d signed codes and one scale, symmetric per row:
 *   s = max_e |x_e| / 127                      (float32, IEEE division)
 *   c_e = round_half_even(x_e / s), clipped to [-127, 127]  (float32 ratio)
 * An all-zero row has s = 0 and codes 0.  A row reads back as
 * bf16(float32(c) * s) (the product in float32, rounded to nearest even):
 * the attention computes on those bf16 values as it does on a bf16 cache.
 *
 * Buffers: k_codes / v_codes (B, Hkv, M, d) int8; k_scales / v_scales
 * (B, Hkv, M) float32; slot_pos and scores as for the bf16 calls.
 *
 *   h2o_kv_quantize    x (n_rows, d) bf16 -> codes (n_rows, d), scales (n_rows);
 *                      d is 64 or 128; n_rows == 0 enqueues nothing.
 *   h2o_kv_dequantize  codes, scales -> x (n_rows, d) bf16, the read-back above.
 *   h2o_update_q8, h2o_evict_insert_q8
 *                      h2o_update_policy / h2o_evict_insert on 8-bit buffers:
 *                      the same slots, scores and positions; the chosen slots
 *                      take the chunk's rows (k_new, v_new bf16) quantised.
 *                      evict_idx (B, Hkv, S) is required: the call sets it to
 *                      -1, the update writes the chosen slots, then a second
 *                      kernel quantises the rows into them.  A (b, h) left
 *                      unchanged (H2O_DEVERR_CANDIDATES) keeps -1 and its
 *                      buffers.  Errors as h2o_update_policy.
 *   h2o_sdpa_chunk_q8, h2o_sdpa_cache_q8
 *                      h2o_sdpa_chunk / h2o_sdpa_cache with the cache read
 *                      through the 8-bit buffers (the chunk's own k_new /
 *                      v_new stay bf16 in h2o_sdpa_chunk_q8).  S = 1 (the
 *                      decode kernels) reads the codes directly.  Otherwise
 *                      the workspace (h2o_q8_workspace_size bytes, 16-byte
 *                      aligned) holds the K and V rows read back to bf16
 *                      (2 B d per slot each; 8 MiB each for B = 1, Hkv = 8,
 *                      M = 4096, d = 128, which stays in L2) ahead of the
 *                      attention's own workspace.  Errors as h2o_sdpa_chunk /
 *                      h2o_sdpa_cache.
 */
H2O_API int h2o_kv_quantize(int64_t n_rows, int32_t d, const h2o_bf16* x, int8_t* codes,
                   float* scales, void* stream);
H2O_API int h2o_kv_dequantize(int64_t n_rows, int32_t d, const int8_t* codes,
                   const float* scales, h2o_bf16* x, void* stream);
H2O_API int h2o_q8_workspace_size(const h2o_dims_t* dims, size_t* bytes);
H2O_API int h2o_update_q8(const h2o_dims_t* dims, int64_t pos0, float* scores,
                   int32_t* slot_pos, const float* score_inc, const h2o_bf16* k_new,
                   const h2o_bf16* v_new, int8_t* k_codes, float* k_scales, int8_t* v_codes,
                   float* v_scales, int32_t budget, int32_t recent_window, int32_t policy,
                   int32_t* evict_idx, void* stream);
H2O_API int h2o_evict_insert_q8(const h2o_dims_t* dims, int64_t pos0, float* scores,
                   int32_t* slot_pos, const h2o_bf16* k_new, const h2o_bf16* v_new,
                   int8_t* k_codes, float* k_scales, int8_t* v_codes, float* v_scales,
                   int32_t budget, int32_t recent_window, int32_t policy, int32_t* evict_idx,
                   void* stream);
H2O_API int h2o_sdpa_chunk_q8(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const int8_t* k_codes, const float* k_scales,
                   const int8_t* v_codes, const float* v_scales, const h2o_bf16* k_new,
                   const h2o_bf16* v_new, const int32_t* slot_pos, h2o_bf16* out,
                   float* score_inc, void* workspace, size_t workspace_bytes, void* stream);
H2O_API int h2o_sdpa_cache_q8(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const int8_t* k_codes, const float* k_scales,
                   const int8_t* v_codes, const float* v_scales, const int32_t* slot_pos,
                   h2o_bf16* out, float* score_inc, void* workspace, size_t workspace_bytes,
                   void* stream);

/*
 * Gradient of one chunk of h2o_sdpa_chunk (§3.1 Eq. 2 with the mask of
 * §3.3.1), for the loss sum(out * dout): the backward pass the paper's
 * fine-tuning runs through every chunk (§3.2; the KV cache policy itself is not
 * differentiated).  Per (b, kv head) the probabilities are recomputed from q
 * and the keys; with D_i = dout_i . out_i and dS = P * (dout V^T - D):
 *
 *   dq = scale dS K,   d[k_cache; k_new] = scale dS^T Q,   d[v_cache; v_new] = P^T dout
 *
 * summed over the q_g query heads of the group for the keys and values.
 *
 *   q, k_cache, v_cache, k_new, v_new, slot_pos, pos0, softmax_scale: as for
 *              h2o_sdpa_chunk (the same call's inputs)
 *   out        (B, Hq, S, d) bf16, the output h2o_sdpa_chunk returned
 *   dout       (B, Hq, S, d) bf16, gradient of the loss w.r.t. out
 *   dq         (B, Hq, S, d) f32, written
 *   dk_cache, dv_cache (B, Hkv, M, d) f32, written (may be NULL when M == 0)
 *   dk_new, dv_new     (B, Hkv, S, d) f32, written
 *   workspace  at least h2o_backward_workspace_size(dims) bytes: two floats
 *              per query row (each group's q_g S rows padded to a multiple
 *              of 128), the rows' log-sum-exp and D
 *
 * Three kernels on the stream: the chunk SDPA's first pass (the rows'
 * log-sum-exp), D per row, and one fused tcgen05 kernel whose CTAs form
 * either 128 rows of dq or 128 keys of dk and dv.  Neither P nor dS is
 * stored: each is rebuilt tile by tile in tensor memory, rounded to bf16 for
 * the contractions (fp32 accumulation); no atomics, so results do not depend
 * on scheduling.  Cache slots no row sees get zero gradient.  A group may
 * hold at most 128 x 4096 query rows (q_g S), else H2O_ERR_UNSUPPORTED.
 */
H2O_API int h2o_backward_workspace_size(const h2o_dims_t* dims, size_t* bytes);
H2O_API int h2o_sdpa_chunk_backward(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                   const h2o_bf16* k_new, const h2o_bf16* v_new, const int32_t* slot_pos,
                   const h2o_bf16* out, const h2o_bf16* dout, float* dq, float* dk_cache,
                   float* dv_cache, float* dk_new, float* dv_new, void* workspace,
                   size_t workspace_bytes, void* stream);

/*
 * h2o_sdpa_chunk_backward given the forward's lse (h2o_sdpa_chunk_lse on the
 * same inputs), as a fine-tuning step that keeps it has it: the log-sum-exp
 * is read instead of recomputed (a row kernel forms D = dout . out and the
 * log2-unit copy the kernel uses), then the fused kernel runs.
 *
 *   lse  (B, Hq, S) f32, read
 *
 * Other arguments, results, workspace and errors as h2o_sdpa_chunk_backward.
 */
H2O_API int h2o_sdpa_chunk_backward_lse(const h2o_dims_t* dims, int64_t pos0, float softmax_scale,
                   const h2o_bf16* q, const h2o_bf16* k_cache, const h2o_bf16* v_cache,
                   const h2o_bf16* k_new, const h2o_bf16* v_new, const int32_t* slot_pos,
                   const h2o_bf16* out, const h2o_bf16* dout, const float* lse, float* dq,
                   float* dk_cache, float* dv_cache, float* dk_new, float* dv_new,
                   void* workspace, size_t workspace_bytes, void* stream);

/* Empties a cache before a new sequence: slot_pos (B, Hkv, M) int32 := -1 and
 * scores (B, Hkv, M) f32 := 0, enqueued on `stream` (the K/V buffers need no
 * clearing: empty slots are never attended and are overwritten first).  This
 * is the state of §3.1 before the first token: a cache filled left to right. */
H2O_API int h2o_cache_reset(const h2o_dims_t* dims, int32_t* slot_pos, float* scores,
                            void* stream);

/* Message for a status code (static storage). */
H2O_API const char* h2o_status_string(int status);

/* cudaError_t of the last failing CUDA runtime call on this host thread. */
H2O_API int h2o_last_cuda_error(void);

/* Synchronises the current device, returns the H2O_DEVERR_* bits recorded by
 * kernels since the last call (0 = none) and clears them.  Negative on a CUDA
 * failure. */
H2O_API int h2o_device_errors(void);

/* Self-test of device-side failure detection (no paper counterpart): one
 * small kernel waits on a barrier that nothing completes, with the same
 * bounded wait every kernel of the library uses, gives up after limit_ns
 * (1 us .. 100 ms, else H2O_ERR_ARG) and records H2O_DEVERR_TIMEOUT, which
 * h2o_device_errors() then reports.  The context stays usable. */
H2O_API int h2o_selftest_bounded_wait(int64_t limit_ns, void* stream);

/* Library version as major*10000 + minor*100 + patch. */
H2O_API int h2o_version(void);

#ifdef __cplusplus
}
#endif

#endif /* H2O_GB300_H2O_H_ */
