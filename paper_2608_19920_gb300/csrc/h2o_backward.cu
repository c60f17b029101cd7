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

// ---- vectorised forms: N_k and M multiples of 4, 16-byte aligned buffers ----
// A row of N_k fp32 scores is then a run of float4s, and no group of four
// columns straddles the cache / chunk boundary.  Each thread keeps four 16-byte
// loads in flight: one 4-byte load per thread (the scalar kernels above) holds
// too few bytes in flight per SM to cover the HBM latency.
constexpr int kVecUnroll = 4;

// Visibility of columns 4v .. 4v+3 of row (query i, position qpos) as a 4-bit
// mask: cache slots by their positions p (§3.3.1), chunk columns causally.
__device__ __forceinline__ unsigned vis_mask4(int v, int mv, int4 p, int qpos, int i, int M) {
  if (v < mv)
    return static_cast<unsigned>(p.x >= 0 && p.x <= qpos) |
           static_cast<unsigned>(p.y >= 0 && p.y <= qpos) << 1 |
           static_cast<unsigned>(p.z >= 0 && p.z <= qpos) << 2 |
           static_cast<unsigned>(p.w >= 0 && p.w <= qpos) << 3;
  const int n = i - (4 * v - M) + 1;  // chunk columns t .. t+3 visible while t <= i
  return n <= 0 ? 0u : n >= 4 ? 15u : (1u << n) - 1u;
}

// (m, l) <- the pair whose sum of 2^(y - m) covers both sets: the online
// softmax merge; an empty set is (-inf, 0).
__device__ __forceinline__ void merge_ml(float& m, float& l, float m2, float l2) {
  const float mn = fmaxf(m, m2);
  if (mn == -INFINITY) return;
  l = l * fast_exp2(m - mn) + l2 * fast_exp2(m2 - mn);
  m = mn;
}

// The softmax pass with one DRAM read of the S row, one CTA of kVecThreads per
// stacked row: a per-thread online (max, sum) over base-2 logits and D's dot
// product, merged across the CTA at one barrier.  kKeep (the row fits one trip
// of kVecUnroll float4s per thread, N_k <= 4096): the write pass takes the
// values still held in registers; otherwise it reads the row again while it is
// in L2 (streaming, its last use).  Four CTAs per SM: 512-thread CTAs (one trip
// up to N_k = 8192, two per SM) measured slower, having fewer rows in flight.
constexpr int kVecThreads = 256;

__device__ __forceinline__ void online4(float4 x, unsigned vm, float c, float& m, float& l) {
  if (vm == 0) return;
  const float y0 = (vm & 1u) ? x.x * c : -INFINITY;
  const float y1 = (vm & 2u) ? x.y * c : -INFINITY;
  const float y2 = (vm & 4u) ? x.z * c : -INFINITY;
  const float y3 = (vm & 8u) ? x.w * c : -INFINITY;
  const float mx = fmaxf(fmaxf(y0, y1), fmaxf(y2, y3));
  if (mx > m) {
    l *= fast_exp2(m - mx);
    m = mx;
  }
  l += (fast_exp2(y0 - m) + fast_exp2(y1 - m)) + (fast_exp2(y2 - m) + fast_exp2(y3 - m));
}

__device__ __forceinline__ uint2 probs4(float4 x, unsigned vm, float c, float lam) {
  const float e0 = (vm & 1u) ? fast_exp2(x.x * c - lam) : 0.f;
  const float e1 = (vm & 2u) ? fast_exp2(x.y * c - lam) : 0.f;
  const float e2 = (vm & 4u) ? fast_exp2(x.z * c - lam) : 0.f;
  const float e3 = (vm & 8u) ? fast_exp2(x.w * c - lam) : 0.f;
  return make_uint2(pack_bf16x2(e0, e1), pack_bf16x2(e2, e3));
}

template <bool kKeep>
__global__ void __launch_bounds__(kVecThreads, 4) bwd_softmax_vec_kernel(const BackwardArgs a) {
  constexpr int T = kVecThreads, U = kVecUnroll, W = kVecThreads / 32;
  __shared__ float sh_m[W], sh_l[W], sh_d[W];
  const size_t row = blockIdx.x;
  const int R = a.qg * a.S;
  const size_t g = row / R;
  const int r = static_cast<int>(row % R);
  const int gg = r / a.S, i = r % a.S;
  const int nv = (a.M + a.S) >> 2, mv = a.M >> 2;
  const float4* s4 = reinterpret_cast<const float4*>(a.sbuf) + row * nv;
  uint2* p4 = reinterpret_cast<uint2*>(a.pbuf) + row * nv;
  const int4* sp4 = reinterpret_cast<const int4*>(a.slot_pos + g * a.M);
  const int qpos = a.pos0 + i;
  const float c = a.scale_log2;

  // D = dout . out of this row (query head h q_g + gg, token i), d <= T: the
  // two loads go out ahead of the row's and are used after them
  const int b = static_cast<int>(g / a.Hkv), h = static_cast<int>(g % a.Hkv);
  const size_t orow = (static_cast<size_t>(b * a.Hq + h * a.qg + gg) * a.S + i) * a.d;
  uint16_t dv = 0, ov = 0;
  if (static_cast<int>(threadIdx.x) < a.d) {
    dv = a.dout[orow + threadIdx.x];
    ov = a.out[orow + threadIdx.x];
  }

  float m = -INFINITY, l = 0.f;
  float4 x[U];
  unsigned vm[U];
#pragma unroll
  for (int u = 0; u < U; ++u) vm[u] = 0u;
  for (int v0 = threadIdx.x; v0 < nv; v0 += U * T) {
    int4 p[U];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int v = v0 + u * T;
      x[u] = make_float4(0.f, 0.f, 0.f, 0.f);
      p[u] = make_int4(-1, -1, -1, -1);
      if (v < nv) x[u] = s4[v];
      if (v < mv) p[u] = __ldg(sp4 + v);
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int v = v0 + u * T;
      vm[u] = v < nv ? vis_mask4(v, mv, p[u], qpos, i, a.M) : 0u;
      online4(x[u], vm[u], c, m, l);
    }
  }
  float dsum = from_bf16(dv) * from_bf16(ov);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    merge_ml(m, l, __shfl_xor_sync(0xffffffffu, m, o), __shfl_xor_sync(0xffffffffu, l, o));
    dsum += __shfl_xor_sync(0xffffffffu, dsum, o);
  }
  if ((threadIdx.x & 31) == 0) {
    sh_m[threadIdx.x >> 5] = m;
    sh_l[threadIdx.x >> 5] = l;
    sh_d[threadIdx.x >> 5] = dsum;
  }
  __syncthreads();
  m = sh_m[0];
  l = sh_l[0];
  for (int w = 1; w < W; ++w) merge_ml(m, l, sh_m[w], sh_l[w]);
  const float lam = m + fast_log2(l);  // every row sees its own token
  if (threadIdx.x == 0) {
    float dr = 0.f;
    for (int w = 0; w < W; ++w) dr += sh_d[w];
    a.drow[row] = dr;
  }

  if constexpr (kKeep) {  // nv <= U T: x and vm hold this thread's whole share
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int v = threadIdx.x + u * T;
      if (v < nv) p4[v] = probs4(x[u], vm[u], c, lam);
    }
  } else {
    for (int v0 = threadIdx.x; v0 < nv; v0 += U * T) {
      int4 p[U];
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + u * T;
        x[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        p[u] = make_int4(-1, -1, -1, -1);
        if (v < nv) x[u] = __ldcs(s4 + v);
        if (v < mv) p[u] = __ldg(sp4 + v);
      }
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int v = v0 + u * T;
        if (v < nv) p4[v] = probs4(x[u], vis_mask4(v, mv, p[u], qpos, i, a.M), c, lam);
      }
    }
  }
}

// dS = P * (dP - D), one CTA per stacked row, four float4 / 8-byte loads in
// flight per thread; dP is read for the last time (streaming).
__global__ void __launch_bounds__(kRowThreads, 4) bwd_ds_vec_kernel(const BackwardArgs a) {
  const size_t row = blockIdx.x;
  const int nv = (a.M + a.S) >> 2;
  const float dr = a.drow[row];
  const float4* s4 = reinterpret_cast<const float4*>(a.sbuf) + row * nv;
  const uint2* p4 = reinterpret_cast<const uint2*>(a.pbuf) + row * nv;
  uint2* ds4 = reinterpret_cast<uint2*>(a.dsbuf) + row * nv;
  for (int v0 = threadIdx.x; v0 < nv; v0 += kVecUnroll * kRowThreads) {
    float4 x[kVecUnroll];
    uint2 p[kVecUnroll];
#pragma unroll
    for (int u = 0; u < kVecUnroll; ++u) {
      const int v = v0 + u * kRowThreads;
      if (v < nv) {
        x[u] = __ldcs(s4 + v);
        p[u] = p4[v];
      }
    }
#pragma unroll
    for (int u = 0; u < kVecUnroll; ++u) {
      const int v = v0 + u * kRowThreads;
      if (v >= nv) continue;
      const float d0 = __uint_as_float(p[u].x << 16) * (x[u].x - dr);
      const float d1 = __uint_as_float(p[u].x & 0xFFFF0000u) * (x[u].y - dr);
      const float d2 = __uint_as_float(p[u].y << 16) * (x[u].z - dr);
      const float d3 = __uint_as_float(p[u].y & 0xFFFF0000u) * (x[u].w - dr);
      ds4[v] = make_uint2(pack_bf16x2(d0, d1), pack_bf16x2(d2, d3));
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
  // the vectorised passes need float4 rows (N_k, M multiples of 4) and 16-byte
  // aligned workspace and slot positions; every other shape takes the scalar ones
  const bool vec = NK % 4 == 0 && M % 4 == 0 && d <= kVecThreads &&
                   (reinterpret_cast<uintptr_t>(workspace) & 15u) == 0 &&
                   (reinterpret_cast<uintptr_t>(a.slot_pos) & 15u) == 0;
  const unsigned rows = static_cast<unsigned>(static_cast<size_t>(G) * R);
  if (vec && NK / 4 <= kVecUnroll * kVecThreads)
    bwd_softmax_vec_kernel<true><<<rows, kVecThreads, 0, stream>>>(a);
  else if (vec)
    bwd_softmax_vec_kernel<false><<<rows, kVecThreads, 0, stream>>>(a);
  else
    bwd_softmax_kernel<<<rows, kRowThreads, 0, stream>>>(a);
  if ((ce = cudaGetLastError()) != cudaSuccess) { out.cuda = ce; return out; }
  // dP = dout V^T into the same buffer
  gemm(true, false, M, R, d, 1.f, a.v_cache, d, sKc, a.dout, d, sQ, 0.f, a.sbuf, NK, sS);
  gemm(true, false, S, R, d, 1.f, a.v_new, d, sKn, a.dout, d, sQ, 0.f, a.sbuf + M, NK, sS);
  if (st != CUBLAS_STATUS_SUCCESS) { out.blas = st; return out; }
  if (vec) {
    bwd_ds_vec_kernel<<<rows, kRowThreads, 0, stream>>>(a);
  } else {
    const size_t blocks = std::min<size_t>(static_cast<size_t>(G) * R, 152 * 8);
    bwd_ds_kernel<<<static_cast<unsigned>(blocks), kRowThreads, 0, stream>>>(a);
  }
  if ((ce = cudaGetLastError()) != cudaSuccess) { out.cuda = ce; return out; }
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
