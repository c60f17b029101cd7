// Gradient of the chunk SDPA under the position mask (§3.1 Eq. 2, mask of
// §3.3.1), the backward pass the paper's fine-tuning runs through every chunk.
//
// For the loss sum(out * dout), per (b, kv head) group with its q_g query heads'
// rows stacked (R = q_g S rows, the layout of q) and the keys [k_cache; k_new]
// (N_k = M + S columns):
//
//   S  = Q K^T                      (GEMM)
//   P  = softmax(mask(scale S))     (masked row softmax, recomputed; bf16)
//   D  = rowsum(dout * out)         (per row)
//   dP = dout V^T                   (GEMM)
//   dS = P * (dP - D)               (elementwise; bf16)
//   dQ = scale dS K,  dK = scale dS^T Q,  dV = P^T dout   (GEMMs)
//
// dK and dV of a KV head sum over its q_g heads because Q, dS and P stack the
// heads' rows.  The five contractions are plain dense GEMMs, so they run on
// cuBLASLt (bf16 operands, fp32 accumulation and outputs), batched over the
// groups, in the caller's workspace; the mask, the softmax and dS run in the
// kernels below.  The S x N_k matrices are materialised (fp32 S / dP, bf16 P
// and dS), so the pass is bandwidth heavy; a fused kernel is future work.
#include <cublasLt.h>

#include <algorithm>
#include <cstdint>
#include <mutex>

#include "h2o_internal.h"
#include "sm100.cuh"

namespace h2o {
namespace {

constexpr int kRowThreads = 256;
constexpr size_t kLtWorkspace = size_t(32) << 20;

__device__ __forceinline__ uint16_t to_bf16(float x) {
  return static_cast<uint16_t>(pack_bf16x2(x, 0.f) & 0xFFFFu);
}

__device__ __forceinline__ float from_bf16(uint16_t x) {
  return __uint_as_float(static_cast<uint32_t>(x) << 16);
}

__device__ __forceinline__ float block_reduce(float v, float* sh, bool is_max) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float y = __shfl_xor_sync(0xffffffffu, v, o);
    v = is_max ? fmaxf(v, y) : v + y;
  }
  const int w = threadIdx.x >> 5;
  __syncthreads();
  if ((threadIdx.x & 31) == 0) sh[w] = v;
  __syncthreads();
  float r = sh[0];
  for (int x = 1; x < kRowThreads / 32; ++x) r = is_max ? fmaxf(r, sh[x]) : r + sh[x];
  return r;
}

// One CTA per stacked row: P (bf16) from the S row, and D.  (Measured against a
// register-resident one-read variant and a warp-per-row online variant: this
// plain three-pass form was the fastest of the three.)
__global__ void __launch_bounds__(kRowThreads) bwd_softmax_kernel(const BackwardArgs a) {
  __shared__ float sh[kRowThreads / 32];
  const size_t row = blockIdx.x;  // g * R + r
  const int R = a.qg * a.S;
  const size_t g = row / R;
  const int r = static_cast<int>(row % R);
  const int gg = r / a.S, i = r % a.S;
  const int NK = a.M + a.S;
  const float* srow = a.sbuf + row * NK;
  uint16_t* prow = a.pbuf + row * NK;
  const int32_t* sp = a.slot_pos + g * a.M;
  const int qpos = a.pos0 + i;
  auto visible = [&](int j) -> bool {
    if (j < a.M) {
      const int pos = __ldg(sp + j);
      return pos >= 0 && pos <= qpos;
    }
    return j - a.M <= i;
  };
  float mx = -INFINITY;
  for (int j = threadIdx.x; j < NK; j += kRowThreads)
    if (visible(j)) mx = fmaxf(mx, srow[j] * a.scale_log2);
  mx = block_reduce(mx, sh, true);
  float sum = 0.f;
  for (int j = threadIdx.x; j < NK; j += kRowThreads)
    if (visible(j)) sum += fast_exp2(srow[j] * a.scale_log2 - mx);
  sum = block_reduce(sum, sh, false);
  const float lam = mx + fast_log2(sum);  // every row sees its own token
  for (int j = threadIdx.x; j < NK; j += kRowThreads)
    prow[j] = to_bf16(visible(j) ? fast_exp2(srow[j] * a.scale_log2 - lam) : 0.f);
  // D = dout . out of this row (query head h q_g + gg, token i)
  const int b = static_cast<int>(g / a.Hkv), h = static_cast<int>(g % a.Hkv);
  const size_t orow = (static_cast<size_t>(b * a.Hq + h * a.qg + gg) * a.S + i) * a.d;
  float dsum = 0.f;
  for (int e = threadIdx.x; e < a.d; e += kRowThreads)
    dsum += from_bf16(a.dout[orow + e]) * from_bf16(a.out[orow + e]);
  dsum = block_reduce(dsum, sh, false);
  if (threadIdx.x == 0) a.drow[row] = dsum;
}

// dS = P * (dP - D), bf16, over every stacked row and key column; CTAs take
// whole rows.
__global__ void __launch_bounds__(kRowThreads) bwd_ds_kernel(const BackwardArgs a) {
  const int NK = a.M + a.S;
  const size_t rows = static_cast<size_t>(a.B) * a.Hkv * a.qg * a.S;
  for (size_t row = blockIdx.x; row < rows; row += gridDim.x) {
    const float dr = a.drow[row];
    const size_t base = row * NK;
    for (int j = threadIdx.x; j < NK; j += kRowThreads) {
      const float p = from_bf16(a.pbuf[base + j]);
      a.dsbuf[base + j] = to_bf16(p * (a.sbuf[base + j] - dr));
    }
  }
}

// ------------------------------------------------------------ cuBLASLt --
struct LtState {
  std::once_flag once;
  cublasStatus_t status = CUBLAS_STATUS_SUCCESS;
  cublasLtHandle_t handle = nullptr;
};
LtState g_lt[64];

int ptr_align(const void* p, size_t stride_bytes) {
  uintptr_t v = reinterpret_cast<uintptr_t>(p) | static_cast<uintptr_t>(stride_bytes) | 256u;
  return static_cast<int>(v & (~v + 1));  // lowest set bit, at most 256
}

// C[m x n] (col-major, ldc, fp32) = alpha op(A) op(B) + beta C, batched over
// `batch` with the given element strides; A and B bf16, stored col-major.
cublasStatus_t lt_gemm(cublasLtHandle_t lt, bool ta, bool tb, int m, int n, int k, float alpha,
                       const uint16_t* A, int lda, int64_t sa, const uint16_t* B, int ldb,
                       int64_t sb, float beta, float* C, int ldc, int64_t sc, int batch,
                       void* ws, size_t ws_bytes, cudaStream_t stream) {
  if (m == 0 || n == 0 || k == 0) return CUBLAS_STATUS_SUCCESS;  // callers never need C = beta C
  cublasLtMatmulDesc_t op = nullptr;
  cublasLtMatrixLayout_t la = nullptr, lb = nullptr, lc = nullptr;
  cublasLtMatmulPreference_t pref = nullptr;
  cublasStatus_t st = cublasLtMatmulDescCreate(&op, CUBLAS_COMPUTE_32F, CUDA_R_32F);
  const cublasOperation_t opa = ta ? CUBLAS_OP_T : CUBLAS_OP_N;
  const cublasOperation_t opb = tb ? CUBLAS_OP_T : CUBLAS_OP_N;
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulDescSetAttribute(op, CUBLASLT_MATMUL_DESC_TRANSA, &opa, sizeof(opa));
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulDescSetAttribute(op, CUBLASLT_MATMUL_DESC_TRANSB, &opb, sizeof(opb));
  // stored shapes: A is (ta ? k x m : m x k), B is (tb ? n x k : k x n)
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatrixLayoutCreate(&la, CUDA_R_16BF, ta ? k : m, ta ? m : k, lda);
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatrixLayoutCreate(&lb, CUDA_R_16BF, tb ? n : k, tb ? k : n, ldb);
  if (st == CUBLAS_STATUS_SUCCESS) st = cublasLtMatrixLayoutCreate(&lc, CUDA_R_32F, m, n, ldc);
  const int32_t nb = batch;
  for (auto [l, s] : {std::pair<cublasLtMatrixLayout_t, int64_t>{la, sa}, {lb, sb}, {lc, sc}}) {
    if (st != CUBLAS_STATUS_SUCCESS) break;
    st = cublasLtMatrixLayoutSetAttribute(l, CUBLASLT_MATRIX_LAYOUT_BATCH_COUNT, &nb, sizeof(nb));
    if (st == CUBLAS_STATUS_SUCCESS)
      st = cublasLtMatrixLayoutSetAttribute(l, CUBLASLT_MATRIX_LAYOUT_STRIDED_BATCH_OFFSET, &s,
                                            sizeof(s));
  }
  if (st == CUBLAS_STATUS_SUCCESS) st = cublasLtMatmulPreferenceCreate(&pref);
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MAX_WORKSPACE_BYTES,
                                              &ws_bytes, sizeof(ws_bytes));
  // the real alignment of every operand (base and batch stride), so that no
  // algorithm needing more is chosen
  const uint32_t al_a = static_cast<uint32_t>(ptr_align(A, sa * 2));
  const uint32_t al_b = static_cast<uint32_t>(ptr_align(B, sb * 2));
  const uint32_t al_c = static_cast<uint32_t>(ptr_align(C, sc * 4));
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_A_BYTES,
                                              &al_a, sizeof(al_a));
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_B_BYTES,
                                              &al_b, sizeof(al_b));
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_C_BYTES,
                                              &al_c, sizeof(al_c));
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulPreferenceSetAttribute(pref, CUBLASLT_MATMUL_PREF_MIN_ALIGNMENT_D_BYTES,
                                              &al_c, sizeof(al_c));
  cublasLtMatmulHeuristicResult_t heur = {};
  int found = 0;
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmulAlgoGetHeuristic(lt, op, la, lb, lc, lc, pref, 1, &heur, &found);
  if (st == CUBLAS_STATUS_SUCCESS && found == 0) st = CUBLAS_STATUS_NOT_SUPPORTED;
  if (st == CUBLAS_STATUS_SUCCESS)
    st = cublasLtMatmul(lt, op, &alpha, A, la, B, lb, &beta, C, lc, C, lc, &heur.algo, ws,
                        ws_bytes, stream);
  if (pref) cublasLtMatmulPreferenceDestroy(pref);
  if (lc) cublasLtMatrixLayoutDestroy(lc);
  if (lb) cublasLtMatrixLayoutDestroy(lb);
  if (la) cublasLtMatrixLayoutDestroy(la);
  if (op) cublasLtMatmulDescDestroy(op);
  return st;
}

size_t align256(size_t x) { return (x + 255) / 256 * 256; }

}  // namespace

size_t backward_workspace_bytes(int B, int Hq, int Hkv, int S, int M) {
  const size_t G = static_cast<size_t>(B) * Hkv, R = static_cast<size_t>(Hq / Hkv) * S;
  const size_t cells = G * R * (static_cast<size_t>(M) + S);
  return kLtWorkspace + align256(cells * 4) + 2 * align256(cells * 2) + align256(G * R * 4);
}

BackwardStatus launch_backward(BackwardArgs a, void* workspace, cudaStream_t stream) {
  BackwardStatus out;
  int dev = 0;
  cudaError_t ce = cudaGetDevice(&dev);
  if (ce != cudaSuccess) { out.cuda = ce; return out; }
  if (dev >= 64) { out.blas = CUBLAS_STATUS_NOT_SUPPORTED; return out; }
  LtState& ls = g_lt[dev];
  std::call_once(ls.once, [&ls] { ls.status = cublasLtCreate(&ls.handle); });
  if (ls.status != CUBLAS_STATUS_SUCCESS) { out.blas = ls.status; return out; }
  const int G = a.B * a.Hkv, R = a.qg * a.S, NK = a.M + a.S, M = a.M, S = a.S, d = a.d;
  const size_t cells = static_cast<size_t>(G) * R * NK;
  uint8_t* w = static_cast<uint8_t*>(workspace);
  void* lt_ws = w;
  w += kLtWorkspace;
  a.sbuf = reinterpret_cast<float*>(w);
  w += align256(cells * 4);
  a.pbuf = reinterpret_cast<uint16_t*>(w);
  w += align256(cells * 2);
  a.dsbuf = reinterpret_cast<uint16_t*>(w);
  w += align256(cells * 2);
  a.drow = reinterpret_cast<float*>(w);

  const int64_t sQ = static_cast<int64_t>(R) * d, sKc = static_cast<int64_t>(M) * d,
                sKn = static_cast<int64_t>(S) * d, sS = static_cast<int64_t>(R) * NK;
  cublasLtHandle_t lt = ls.handle;
  cublasStatus_t st = CUBLAS_STATUS_SUCCESS;
  auto gemm = [&](bool ta, bool tb, int m, int n, int k, float alpha, const uint16_t* A, int lda,
                  int64_t sa, const uint16_t* B, int ldb, int64_t sb, float beta, float* C,
                  int ldc, int64_t sc) {
    if (st == CUBLAS_STATUS_SUCCESS)
      st = lt_gemm(lt, ta, tb, m, n, k, alpha, A, lda, sa, B, ldb, sb, beta, C, ldc, sc, G, lt_ws,
                   kLtWorkspace, stream);
  };
  // S = Q K^T: per group, col-major C (N_k x R): cache block rows 0..M-1, chunk block M..
  gemm(true, false, M, R, d, 1.f, a.k_cache, d, sKc, a.q, d, sQ, 0.f, a.sbuf, NK, sS);
  gemm(true, false, S, R, d, 1.f, a.k_new, d, sKn, a.q, d, sQ, 0.f, a.sbuf + M, NK, sS);
  if (st != CUBLAS_STATUS_SUCCESS) { out.blas = st; return out; }
  bwd_softmax_kernel<<<static_cast<unsigned>(static_cast<size_t>(G) * R), kRowThreads, 0, stream>>>(a);
  if ((ce = cudaGetLastError()) != cudaSuccess) { out.cuda = ce; return out; }
  // dP = dout V^T into the same buffer
  gemm(true, false, M, R, d, 1.f, a.v_cache, d, sKc, a.dout, d, sQ, 0.f, a.sbuf, NK, sS);
  gemm(true, false, S, R, d, 1.f, a.v_new, d, sKn, a.dout, d, sQ, 0.f, a.sbuf + M, NK, sS);
  if (st != CUBLAS_STATUS_SUCCESS) { out.blas = st; return out; }
  {
    const size_t blocks = std::min<size_t>(static_cast<size_t>(G) * R, 152 * 8);
    bwd_ds_kernel<<<static_cast<unsigned>(blocks), kRowThreads, 0, stream>>>(a);
    if ((ce = cudaGetLastError()) != cudaSuccess) { out.cuda = ce; return out; }
  }
  // dQ^T (d x R) = K^T dS^T: cache block, then += chunk block
  gemm(false, false, d, R, M, a.scale, a.k_cache, d, sKc, a.dsbuf, NK, sS, 0.f, a.dq, d, sQ);
  gemm(false, false, d, R, S, a.scale, a.k_new, d, sKn, a.dsbuf + M, NK, sS, M > 0 ? 1.f : 0.f,
       a.dq, d, sQ);
  // dK^T (d x M) = Q^T dS (R x M); dV^T = dout^T P
  gemm(false, true, d, M, R, a.scale, a.q, d, sQ, a.dsbuf, NK, sS, 0.f, a.dk_cache, d, sKc);
  gemm(false, true, d, S, R, a.scale, a.q, d, sQ, a.dsbuf + M, NK, sS, 0.f, a.dk_new, d, sKn);
  gemm(false, true, d, M, R, 1.f, a.dout, d, sQ, a.pbuf, NK, sS, 0.f, a.dv_cache, d, sKc);
  gemm(false, true, d, S, R, 1.f, a.dout, d, sQ, a.pbuf + M, NK, sS, 0.f, a.dv_new, d, sKn);
  out.blas = st;
  return out;
}

}  // namespace h2o
