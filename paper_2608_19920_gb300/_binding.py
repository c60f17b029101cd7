"""ctypes binding of libh2o_gb300.so (include/h2o.h): argument marshalling only.

Every step of the computation runs in the CUDA library; these wrappers check
tensor shapes, dtypes and devices, pass raw device pointers and the current
CUDA stream, and turn negative status codes into exceptions.  There is no CPU
or PyTorch fallback: without the built library every call raises.
"""
from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libh2o_gb300.so")

H2O_OK = 0
H2O_DEVERR_TIMEOUT = 1
H2O_DEVERR_CANDIDATES = 2
H2O_DEVERR_INDEX = 4

# Every symbol include/h2o.h declares.
EXPORTS = ("h2o_workspace_size", "h2o_sdpa_chunk", "h2o_sdpa_decode_static", "h2o_update",
           "h2o_update_policy", "h2o_evict_insert", "h2o_sdpa_cache", "h2o_scores_add",
           "h2o_kv_replace", "h2o_kv_restore", "h2o_backward_workspace_size",
           "h2o_sdpa_chunk_backward", "h2o_sdpa_chunk_lse", "h2o_sdpa_chunk_backward_lse",
           "h2o_selftest_bounded_wait",
           "h2o_kv_quantize", "h2o_kv_dequantize", "h2o_q8_workspace_size", "h2o_update_q8",
           "h2o_evict_insert_q8", "h2o_sdpa_chunk_q8", "h2o_sdpa_cache_q8",
           "h2o_cache_reset", "h2o_status_string", "h2o_last_cuda_error", "h2o_device_errors",
           "h2o_version")

# Eviction policies of h2o_update_policy (H2O_POLICY_* in include/h2o.h).
POLICY = {"h2o": 0, "h2o_norm": 1, "h2o_orig": 2}


class H2ODims(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("Hq", ctypes.c_int32), ("Hkv", ctypes.c_int32),
                ("d", ctypes.c_int32), ("S", ctypes.c_int32), ("M", ctypes.c_int32)]


class H2OError(RuntimeError):
    def __init__(self, fn: str, status: int, lib):
        msg = lib.h2o_status_string(status).decode()
        if status == -7:
            msg += f" (cudaError {lib.h2o_last_cuda_error()})"
        super().__init__(f"{fn} failed: {msg} [{status}]")
        self.status = status


_lib = None


def load(path: str = LIB_PATH):
    """Loads the library (once) and declares the C signatures."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(path):
        raise RuntimeError(
            f"CUDA library not built: {path} is missing. Build it with "
            "`python -m paper_2608_19920_gb300.build` (needs nvcc); there is no fallback.")
    lib = ctypes.CDLL(path)
    vp, i32, i64, f32 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float
    dims_p = ctypes.POINTER(H2ODims)
    lib.h2o_workspace_size.argtypes = [dims_p, ctypes.POINTER(ctypes.c_size_t)]
    lib.h2o_sdpa_chunk.argtypes = [dims_p, i64, f32, vp, vp, vp, vp, vp, vp, vp, vp, vp,
                                   ctypes.c_size_t, vp]
    lib.h2o_sdpa_decode_static.argtypes = [dims_p, i64, f32, vp, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.h2o_update.argtypes = [dims_p, i64, vp, vp, vp, vp, vp, vp, vp, i32, i32, vp, vp]
    lib.h2o_update_policy.argtypes = [dims_p, i64, vp, vp, vp, vp, vp, vp, vp, i32, i32, i32,
                                      vp, vp]
    lib.h2o_evict_insert.argtypes = [dims_p, i64, vp, vp, vp, vp, vp, vp, i32, i32, i32, vp, vp]
    lib.h2o_sdpa_cache.argtypes = [dims_p, i64, f32, vp, vp, vp, vp, vp, vp, vp, ctypes.c_size_t,
                                   vp]
    lib.h2o_scores_add.argtypes = [dims_p, vp, vp, vp]
    lib.h2o_kv_replace.argtypes = [dims_p, i64, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.h2o_kv_restore.argtypes = [dims_p, vp, vp, vp, vp, vp, vp, vp, vp]
    lib.h2o_backward_workspace_size.argtypes = [dims_p, ctypes.POINTER(ctypes.c_size_t)]
    lib.h2o_sdpa_chunk_backward.argtypes = [dims_p, i64, f32] + [vp] * 14 + [ctypes.c_size_t, vp]
    lib.h2o_sdpa_chunk_lse.argtypes = [dims_p, i64, f32] + [vp] * 10 + [ctypes.c_size_t, vp]
    lib.h2o_sdpa_chunk_backward_lse.argtypes = ([dims_p, i64, f32] + [vp] * 15 +
                                                [ctypes.c_size_t, vp])
    lib.h2o_selftest_bounded_wait.argtypes = [i64, vp]
    lib.h2o_kv_quantize.argtypes = [i64, i32, vp, vp, vp, vp]
    lib.h2o_kv_dequantize.argtypes = [i64, i32, vp, vp, vp, vp]
    lib.h2o_q8_workspace_size.argtypes = [dims_p, ctypes.POINTER(ctypes.c_size_t)]
    lib.h2o_update_q8.argtypes = [dims_p, i64] + [vp] * 9 + [i32, i32, i32, vp, vp]
    lib.h2o_evict_insert_q8.argtypes = [dims_p, i64] + [vp] * 8 + [i32, i32, i32, vp, vp]
    lib.h2o_sdpa_chunk_q8.argtypes = [dims_p, i64, f32] + [vp] * 11 + [ctypes.c_size_t, vp]
    lib.h2o_sdpa_cache_q8.argtypes = [dims_p, i64, f32] + [vp] * 9 + [ctypes.c_size_t, vp]
    lib.h2o_cache_reset.argtypes = [dims_p, vp, vp, vp]
    lib.h2o_status_string.argtypes = [ctypes.c_int]
    lib.h2o_status_string.restype = ctypes.c_char_p
    for fn in ("h2o_workspace_size", "h2o_sdpa_chunk", "h2o_sdpa_decode_static", "h2o_update",
               "h2o_update_policy", "h2o_evict_insert", "h2o_sdpa_cache", "h2o_scores_add",
               "h2o_kv_replace", "h2o_kv_restore", "h2o_backward_workspace_size",
               "h2o_sdpa_chunk_backward", "h2o_sdpa_chunk_lse", "h2o_sdpa_chunk_backward_lse",
               "h2o_selftest_bounded_wait", "h2o_cache_reset",
               "h2o_kv_quantize", "h2o_kv_dequantize", "h2o_q8_workspace_size",
               "h2o_update_q8", "h2o_evict_insert_q8", "h2o_sdpa_chunk_q8", "h2o_sdpa_cache_q8",
               "h2o_last_cuda_error",
               "h2o_device_errors", "h2o_version"):
        getattr(lib, fn).restype = ctypes.c_int
    _lib = lib
    return lib


def _check(fn: str, status: int):
    if status != H2O_OK:
        raise H2OError(fn, status, _lib)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _expect(t, name, shape, dtype, device):
    if t is None:
        raise ValueError(f"{name} is required")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")
    if t.dtype != dtype:
        raise ValueError(f"{name}: expected {dtype}, got {t.dtype}")
    if t.device != device:
        raise ValueError(f"{name}: expected device {device}, got {t.device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def dims_of(q, k_cache_or_M, k_new):
    B, Hq, S, d = q.shape
    Hkv = k_new.shape[1]
    M = k_cache_or_M if isinstance(k_cache_or_M, int) else k_cache_or_M.shape[2]
    return H2ODims(B, Hq, Hkv, d, S, M)


def h2o_workspace_size(dims: H2ODims) -> int:
    lib = load()
    n = ctypes.c_size_t(0)
    _check("h2o_workspace_size", lib.h2o_workspace_size(ctypes.byref(dims), ctypes.byref(n)))
    return n.value


def h2o_sdpa_chunk(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0: int, scale: float = 0.0,
                   out=None, score_inc=None, workspace=None, stream=None):
    """Sparse SDPA of one chunk + summed attention weights (see include/h2o.h).

    q (B,Hq,S,d) bf16; k_cache/v_cache (B,Hkv,M,d) bf16; k_new/v_new (B,Hkv,S,d)
    bf16; slot_pos (B,Hkv,M) int32.  Returns (out (B,Hq,S,d) bf16,
    score_inc (B,Hq,M+S) f32).  ``workspace`` (a device buffer of at least
    h2o_workspace_size bytes) is allocated here when it is needed and not given.
    """
    lib = load()
    dev = q.device
    B, Hq, S, d = q.shape
    Hkv = k_new.shape[1]
    M = k_cache.shape[2]
    bf = torch.bfloat16
    _expect(q, "q", (B, Hq, S, d), bf, dev)
    _expect(k_cache, "k_cache", (B, Hkv, M, d), bf, dev)
    _expect(v_cache, "v_cache", (B, Hkv, M, d), bf, dev)
    _expect(k_new, "k_new", (B, Hkv, S, d), bf, dev)
    _expect(v_new, "v_new", (B, Hkv, S, d), bf, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    if out is None:
        out = torch.empty((B, Hq, S, d), dtype=bf, device=dev)
    if score_inc is None:
        score_inc = torch.empty((B, Hq, M + S), dtype=torch.float32, device=dev)
    _expect(out, "out", (B, Hq, S, d), bf, dev)
    _expect(score_inc, "score_inc", (B, Hq, M + S), torch.float32, dev)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    if workspace is None:
        n = h2o_workspace_size(dims)
        if n:
            workspace = torch.empty(n, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.h2o_sdpa_chunk(ctypes.byref(dims), int(pos0), float(scale), _ptr(q), _ptr(k_cache),
                            _ptr(v_cache), _ptr(k_new), _ptr(v_new), _ptr(slot_pos), _ptr(out),
                            _ptr(score_inc), _ptr(workspace), ws_bytes, _stream(stream))
    _check("h2o_sdpa_chunk", st)
    return out, score_inc


def h2o_sdpa_chunk_lse(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0: int, scale: float = 0.0,
                       workspace=None, stream=None):
    """h2o_sdpa_chunk that also returns each query row's log-sum-exp (natural
    log), for h2o_sdpa_chunk_backward_lse.  Returns (out, score_inc, lse
    (B,Hq,S) f32)."""
    lib = load()
    dev = q.device
    B, Hq, S, d = q.shape
    Hkv, M = k_new.shape[1], k_cache.shape[2]
    bf = torch.bfloat16
    for t, n, shp, dt in ((q, "q", (B, Hq, S, d), bf), (k_cache, "k_cache", (B, Hkv, M, d), bf),
                          (v_cache, "v_cache", (B, Hkv, M, d), bf),
                          (k_new, "k_new", (B, Hkv, S, d), bf), (v_new, "v_new", (B, Hkv, S, d), bf),
                          (slot_pos, "slot_pos", (B, Hkv, M), torch.int32)):
        _expect(t, n, shp, dt, dev)
    out = torch.empty((B, Hq, S, d), dtype=bf, device=dev)
    score_inc = torch.empty((B, Hq, M + S), dtype=torch.float32, device=dev)
    lse = torch.empty((B, Hq, S), dtype=torch.float32, device=dev)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    if workspace is None:
        n = h2o_workspace_size(dims)
        if n:
            workspace = torch.empty(n, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.h2o_sdpa_chunk_lse(ctypes.byref(dims), int(pos0), float(scale), _ptr(q),
                                _ptr(k_cache), _ptr(v_cache), _ptr(k_new), _ptr(v_new),
                                _ptr(slot_pos), _ptr(out), _ptr(score_inc), _ptr(lse),
                                _ptr(workspace), ws_bytes, _stream(stream))
    _check("h2o_sdpa_chunk_lse", st)
    return out, score_inc, lse


def h2o_sdpa_decode_static(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0: int,
                           scale: float = 0.0, out=None, score_inc=None, stream=None):
    """h2o_sdpa_chunk for S = 1 on the library's fixed scratch (see include/h2o.h):
    the call itself allocates nothing on the device (``out`` and ``score_inc``
    are allocated here only when not given)."""
    lib = load()
    dev = q.device
    B, Hq, S, d = q.shape
    Hkv = k_new.shape[1]
    M = k_cache.shape[2]
    bf = torch.bfloat16
    _expect(q, "q", (B, Hq, S, d), bf, dev)
    _expect(k_cache, "k_cache", (B, Hkv, M, d), bf, dev)
    _expect(v_cache, "v_cache", (B, Hkv, M, d), bf, dev)
    _expect(k_new, "k_new", (B, Hkv, S, d), bf, dev)
    _expect(v_new, "v_new", (B, Hkv, S, d), bf, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    if out is None:
        out = torch.empty((B, Hq, S, d), dtype=bf, device=dev)
    if score_inc is None:
        score_inc = torch.empty((B, Hq, M + S), dtype=torch.float32, device=dev)
    _expect(out, "out", (B, Hq, S, d), bf, dev)
    _expect(score_inc, "score_inc", (B, Hq, M + S), torch.float32, dev)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    st = lib.h2o_sdpa_decode_static(ctypes.byref(dims), int(pos0), float(scale), _ptr(q),
                                    _ptr(k_cache), _ptr(v_cache), _ptr(k_new), _ptr(v_new),
                                    _ptr(slot_pos), _ptr(out), _ptr(score_inc), _stream(stream))
    _check("h2o_sdpa_decode_static", st)
    return out, score_inc


def h2o_update(scores, slot_pos, score_inc, k_new, v_new, k_cache, v_cache, pos0: int,
               recent_window: int, evict_idx=None, budget: int | None = None, stream=None,
               policy: str = "h2o"):
    """H2O score accumulation, eviction and K/V write, in place (see include/h2o.h).

    scores (B,Hkv,M) f32, slot_pos (B,Hkv,M) int32, score_inc (B,Hq,M+S) f32,
    k_new/v_new (B,Hkv,S,d) bf16, k_cache/v_cache (B,Hkv,M,d) bf16,
    evict_idx (B,Hkv,S) int32 or None.  ``policy`` "h2o" calls h2o_update,
    "h2o_norm" / "h2o_orig" call h2o_update_policy.  Returns evict_idx.
    """
    lib = load()
    dev = scores.device
    B, Hkv, M = scores.shape
    S, d = k_new.shape[2], k_new.shape[3]
    Hq = score_inc.shape[1]
    _expect(scores, "scores", (B, Hkv, M), torch.float32, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    _expect(score_inc, "score_inc", (B, Hq, M + S), torch.float32, dev)
    _expect(k_new, "k_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect(v_new, "v_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect(k_cache, "k_cache", (B, Hkv, M, d), torch.bfloat16, dev)
    _expect(v_cache, "v_cache", (B, Hkv, M, d), torch.bfloat16, dev)
    if evict_idx is not None:
        _expect(evict_idx, "evict_idx", (B, Hkv, S), torch.int32, dev)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    args = (ctypes.byref(dims), int(pos0), _ptr(scores), _ptr(slot_pos), _ptr(score_inc),
            _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache),
            int(M if budget is None else budget), int(recent_window))
    if policy == "h2o":
        st = lib.h2o_update(*args, _ptr(evict_idx), _stream(stream))
        _check("h2o_update", st)
    else:
        if policy not in POLICY:
            raise ValueError(f"unknown policy {policy!r}")
        st = lib.h2o_update_policy(*args, POLICY[policy], _ptr(evict_idx), _stream(stream))
        _check("h2o_update_policy", st)
    return evict_idx


def h2o_update_policy(scores, slot_pos, score_inc, k_new, v_new, k_cache, v_cache, pos0: int,
                      recent_window: int, policy: str, evict_idx=None, budget: int | None = None,
                      stream=None):
    """h2o_update with an explicit eviction policy of §3.1.1: "h2o", "h2o_norm"
    or "h2o_orig" (see include/h2o.h).  Returns evict_idx."""
    if policy not in POLICY:
        raise ValueError(f"unknown policy {policy!r}")
    return h2o_update(scores, slot_pos, score_inc, k_new, v_new, k_cache, v_cache, pos0,
                      recent_window, evict_idx=evict_idx, budget=budget, stream=stream,
                      policy=policy)


def h2o_evict_insert(scores, slot_pos, k_new, v_new, k_cache, v_cache, pos0: int,
                     recent_window: int, policy: str = "h2o", evict_idx=None,
                     budget: int | None = None, Hq: int | None = None, stream=None):
    """Paper-order step, part 1 (see include/h2o.h): the S lowest-scored
    candidate slots take the chunk's K/V, position pos0 + c and score 0, in
    place.  ``Hq`` only fills the size struct (default: Hkv).  Returns evict_idx."""
    lib = load()
    dev = scores.device
    B, Hkv, M = scores.shape
    S, d = k_new.shape[2], k_new.shape[3]
    if policy not in POLICY:
        raise ValueError(f"unknown policy {policy!r}")
    _expect(scores, "scores", (B, Hkv, M), torch.float32, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    _expect(k_new, "k_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect(v_new, "v_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect(k_cache, "k_cache", (B, Hkv, M, d), torch.bfloat16, dev)
    _expect(v_cache, "v_cache", (B, Hkv, M, d), torch.bfloat16, dev)
    if evict_idx is not None:
        _expect(evict_idx, "evict_idx", (B, Hkv, S), torch.int32, dev)
    dims = H2ODims(B, Hkv if Hq is None else Hq, Hkv, d, S, M)
    st = lib.h2o_evict_insert(ctypes.byref(dims), int(pos0), _ptr(scores), _ptr(slot_pos),
                              _ptr(k_new), _ptr(v_new), _ptr(k_cache), _ptr(v_cache),
                              int(M if budget is None else budget), int(recent_window),
                              POLICY[policy], _ptr(evict_idx), _stream(stream))
    _check("h2o_evict_insert", st)
    return evict_idx


def h2o_sdpa_cache(q, k_cache, v_cache, slot_pos, pos0: int, scale: float = 0.0, out=None,
                   score_inc=None, workspace=None, stream=None):
    """Paper-order step, part 2: SDPA of the chunk over the M cache slots only
    (the chunk's K/V already written there).  Returns (out (B,Hq,S,d) bf16,
    score_inc (B,Hq,M) f32)."""
    lib = load()
    dev = q.device
    B, Hq, S, d = q.shape
    Hkv, M = k_cache.shape[1], k_cache.shape[2]
    bf = torch.bfloat16
    _expect(q, "q", (B, Hq, S, d), bf, dev)
    _expect(k_cache, "k_cache", (B, Hkv, M, d), bf, dev)
    _expect(v_cache, "v_cache", (B, Hkv, M, d), bf, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    if out is None:
        out = torch.empty((B, Hq, S, d), dtype=bf, device=dev)
    if score_inc is None:
        score_inc = torch.empty((B, Hq, M), dtype=torch.float32, device=dev)
    _expect(out, "out", (B, Hq, S, d), bf, dev)
    _expect(score_inc, "score_inc", (B, Hq, M), torch.float32, dev)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    if workspace is None:
        n = h2o_workspace_size(dims)
        if n:
            workspace = torch.empty(n, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    st = lib.h2o_sdpa_cache(ctypes.byref(dims), int(pos0), float(scale), _ptr(q), _ptr(k_cache),
                            _ptr(v_cache), _ptr(slot_pos), _ptr(out), _ptr(score_inc),
                            _ptr(workspace), ws_bytes, _stream(stream))
    _check("h2o_sdpa_cache", st)
    return out, score_inc


def h2o_scores_add(scores, score_inc, stream=None):
    """Paper-order step, part 3: scores += the GQA-group sum of score_inc (B,Hq,M)."""
    lib = load()
    dev = scores.device
    B, Hkv, M = scores.shape
    Hq = score_inc.shape[1]
    _expect(scores, "scores", (B, Hkv, M), torch.float32, dev)
    _expect(score_inc, "score_inc", (B, Hq, M), torch.float32, dev)
    dims = H2ODims(B, Hq, Hkv, 64, 1, M)
    _check("h2o_scores_add", lib.h2o_scores_add(ctypes.byref(dims), _ptr(scores),
                                                _ptr(score_inc), _stream(stream)))


def h2o_kv_replace(index, k_new, v_new, k_cache, v_cache, pos0: int, slot_pos=None,
                   delta_k=None, delta_v=None, delta_pos=None, stream=None):
    """Replay-cache write (see include/h2o.h): the chunk's rows go to the slots
    ``index`` (B,Hkv,S) int32, in place; the replaced rows / positions go to the
    delta buffers when given.  Returns (delta_k, delta_v, delta_pos)."""
    lib = load()
    dev = k_cache.device
    B, Hkv, M, d = k_cache.shape
    S = index.shape[2]
    bf = torch.bfloat16
    _expect(index, "index", (B, Hkv, S), torch.int32, dev)
    for t, n, shp in ((k_new, "k_new", (B, Hkv, S, d)), (v_new, "v_new", (B, Hkv, S, d)),
                      (v_cache, "v_cache", (B, Hkv, M, d))):
        _expect(t, n, shp, bf, dev)
    if slot_pos is not None:
        _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    if delta_k is not None or delta_v is not None:
        _expect(delta_k, "delta_k", (B, Hkv, S, d), bf, dev)
        _expect(delta_v, "delta_v", (B, Hkv, S, d), bf, dev)
    if delta_pos is not None:
        _expect(delta_pos, "delta_pos", (B, Hkv, S), torch.int32, dev)
    dims = H2ODims(B, Hkv, Hkv, d, S, M)
    _check("h2o_kv_replace", lib.h2o_kv_replace(
        ctypes.byref(dims), int(pos0), _ptr(index), _ptr(k_new), _ptr(v_new), _ptr(k_cache),
        _ptr(v_cache), _ptr(slot_pos), _ptr(delta_k), _ptr(delta_v), _ptr(delta_pos),
        _stream(stream)))
    return delta_k, delta_v, delta_pos


def h2o_kv_restore(index, delta_k, delta_v, k_cache, v_cache, slot_pos=None, delta_pos=None,
                   stream=None):
    """The reverse recurrence: scatter the saved rows (and positions) back, in place."""
    lib = load()
    dev = k_cache.device
    B, Hkv, M, d = k_cache.shape
    S = index.shape[2]
    bf = torch.bfloat16
    _expect(index, "index", (B, Hkv, S), torch.int32, dev)
    _expect(delta_k, "delta_k", (B, Hkv, S, d), bf, dev)
    _expect(delta_v, "delta_v", (B, Hkv, S, d), bf, dev)
    _expect(v_cache, "v_cache", (B, Hkv, M, d), bf, dev)
    if slot_pos is not None:
        _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    if delta_pos is not None:
        _expect(delta_pos, "delta_pos", (B, Hkv, S), torch.int32, dev)
    dims = H2ODims(B, Hkv, Hkv, d, S, M)
    _check("h2o_kv_restore", lib.h2o_kv_restore(
        ctypes.byref(dims), _ptr(index), _ptr(delta_k), _ptr(delta_v), _ptr(delta_pos),
        _ptr(k_cache), _ptr(v_cache), _ptr(slot_pos), _stream(stream)))


def h2o_backward_workspace_size(dims: H2ODims) -> int:
    lib = load()
    n = ctypes.c_size_t(0)
    _check("h2o_backward_workspace_size",
           lib.h2o_backward_workspace_size(ctypes.byref(dims), ctypes.byref(n)))
    return n.value


def h2o_sdpa_chunk_backward(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0: int, out, dout,
                            scale: float = 0.0, workspace=None, stream=None, lse=None):
    """Gradient of sum(out * dout) for one h2o_sdpa_chunk call (see include/h2o.h).
    Returns fp32 (dq, dk_cache, dv_cache, dk_new, dv_new).  With ``lse`` (the
    forward's, from h2o_sdpa_chunk_lse) this calls h2o_sdpa_chunk_backward_lse."""
    lib = load()
    dev = q.device
    B, Hq, S, d = q.shape
    Hkv, M = k_new.shape[1], k_cache.shape[2]
    bf = torch.bfloat16
    for t, n, shp, dt in ((q, "q", (B, Hq, S, d), bf), (k_cache, "k_cache", (B, Hkv, M, d), bf),
                          (v_cache, "v_cache", (B, Hkv, M, d), bf),
                          (k_new, "k_new", (B, Hkv, S, d), bf), (v_new, "v_new", (B, Hkv, S, d), bf),
                          (slot_pos, "slot_pos", (B, Hkv, M), torch.int32),
                          (out, "out", (B, Hq, S, d), bf), (dout, "dout", (B, Hq, S, d), bf)):
        _expect(t, n, shp, dt, dev)
    f32 = torch.float32
    dq = torch.empty((B, Hq, S, d), dtype=f32, device=dev)
    dkc = torch.empty((B, Hkv, M, d), dtype=f32, device=dev)
    dvc = torch.empty_like(dkc)
    dkn = torch.empty((B, Hkv, S, d), dtype=f32, device=dev)
    dvn = torch.empty_like(dkn)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    if workspace is None:
        workspace = torch.empty(h2o_backward_workspace_size(dims), dtype=torch.uint8, device=dev)
    ws_bytes = workspace.numel() * workspace.element_size()
    head = (ctypes.byref(dims), int(pos0), float(scale), _ptr(q), _ptr(k_cache), _ptr(v_cache),
            _ptr(k_new), _ptr(v_new), _ptr(slot_pos), _ptr(out), _ptr(dout))
    tail = (_ptr(dq), _ptr(dkc if M else None), _ptr(dvc if M else None), _ptr(dkn), _ptr(dvn),
            _ptr(workspace), ws_bytes, _stream(stream))
    if lse is None:
        st = lib.h2o_sdpa_chunk_backward(*head, *tail)
        _check("h2o_sdpa_chunk_backward", st)
    else:
        _expect(lse, "lse", (B, Hq, S), torch.float32, dev)
        st = lib.h2o_sdpa_chunk_backward_lse(*head, _ptr(lse), *tail)
        _check("h2o_sdpa_chunk_backward_lse", st)
    return dq, dkc, dvc, dkn, dvn


def h2o_sdpa_chunk_backward_lse(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0: int, out, dout,
                                lse, scale: float = 0.0, workspace=None, stream=None):
    """h2o_sdpa_chunk_backward given the forward's lse (h2o_sdpa_chunk_lse):
    the log-sum-exp is not recomputed."""
    return h2o_sdpa_chunk_backward(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0, out, dout,
                                   scale, workspace, stream, lse=lse)


def h2o_cache_reset(slot_pos, scores, stream=None):
    """slot_pos := -1, scores := 0 (an empty cache), enqueued on the stream."""
    lib = load()
    B, Hkv, M = slot_pos.shape
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, slot_pos.device)
    _expect(scores, "scores", (B, Hkv, M), torch.float32, slot_pos.device)
    dims = H2ODims(B, Hkv, Hkv, 64, 1, M)
    _check("h2o_cache_reset", lib.h2o_cache_reset(ctypes.byref(dims), _ptr(slot_pos),
                                                  _ptr(scores), _stream(stream)))


def h2o_selftest_bounded_wait(limit_ns: int = 5_000_000, stream=None):
    """Runs the device-side bounded-wait self-test (see include/h2o.h)."""
    _check("h2o_selftest_bounded_wait",
           load().h2o_selftest_bounded_wait(int(limit_ns), _stream(stream)))


def h2o_device_errors() -> int:
    lib = load()
    r = lib.h2o_device_errors()
    if r < 0:
        _check("h2o_device_errors", r)
    return r


def h2o_status_string(status: int) -> str:
    return load().h2o_status_string(status).decode()


def h2o_version() -> int:
    return load().h2o_version()


# ---------------------------------------------------- 8-bit K/V buffers --

def h2o_kv_quantize(x, codes=None, scales=None, stream=None):
    """Rows (..., d) bf16 -> (codes (..., d) int8, scales (...) f32), per-row
    symmetric (see include/h2o.h)."""
    lib = load()
    dev = x.device
    d = x.shape[-1]
    _expect(x, "x", x.shape, torch.bfloat16, dev)
    if codes is None:
        codes = torch.empty(x.shape, dtype=torch.int8, device=dev)
    if scales is None:
        scales = torch.empty(x.shape[:-1], dtype=torch.float32, device=dev)
    _expect(codes, "codes", x.shape, torch.int8, dev)
    _expect(scales, "scales", x.shape[:-1], torch.float32, dev)
    n = x.numel() // d if d else 0
    _check("h2o_kv_quantize", lib.h2o_kv_quantize(int(n), int(d), _ptr(x), _ptr(codes),
                                                  _ptr(scales), _stream(stream)))
    return codes, scales


def h2o_kv_dequantize(codes, scales, out=None, stream=None):
    """codes (..., d) int8 + scales (...) f32 -> the bf16 rows they read back as."""
    lib = load()
    dev = codes.device
    d = codes.shape[-1]
    _expect(codes, "codes", codes.shape, torch.int8, dev)
    _expect(scales, "scales", codes.shape[:-1], torch.float32, dev)
    if out is None:
        out = torch.empty(codes.shape, dtype=torch.bfloat16, device=dev)
    _expect(out, "out", codes.shape, torch.bfloat16, dev)
    n = codes.numel() // d if d else 0
    _check("h2o_kv_dequantize", lib.h2o_kv_dequantize(int(n), int(d), _ptr(codes), _ptr(scales),
                                                      _ptr(out), _stream(stream)))
    return out


def h2o_q8_workspace_size(dims: H2ODims) -> int:
    lib = load()
    n = ctypes.c_size_t(0)
    _check("h2o_q8_workspace_size", lib.h2o_q8_workspace_size(ctypes.byref(dims), ctypes.byref(n)))
    return n.value


def _expect_q8(k_codes, k_scales, v_codes, v_scales, B, Hkv, M, d, dev):
    _expect(k_codes, "k_codes", (B, Hkv, M, d), torch.int8, dev)
    _expect(v_codes, "v_codes", (B, Hkv, M, d), torch.int8, dev)
    _expect(k_scales, "k_scales", (B, Hkv, M), torch.float32, dev)
    _expect(v_scales, "v_scales", (B, Hkv, M), torch.float32, dev)


def h2o_update_q8(scores, slot_pos, score_inc, k_new, v_new, k_codes, k_scales, v_codes,
                  v_scales, pos0: int, recent_window: int, policy: str = "h2o", evict_idx=None,
                  budget: int | None = None, stream=None):
    """h2o_update_policy on 8-bit buffers, in place.  Returns evict_idx (B,Hkv,S)."""
    lib = load()
    dev = scores.device
    B, Hkv, M = scores.shape
    S, d = k_new.shape[2], k_new.shape[3]
    Hq = score_inc.shape[1]
    if policy not in POLICY:
        raise ValueError(f"unknown policy {policy!r}")
    _expect(scores, "scores", (B, Hkv, M), torch.float32, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    _expect(score_inc, "score_inc", (B, Hq, M + S), torch.float32, dev)
    _expect(k_new, "k_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect(v_new, "v_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect_q8(k_codes, k_scales, v_codes, v_scales, B, Hkv, M, d, dev)
    if evict_idx is None:
        evict_idx = torch.empty((B, Hkv, S), dtype=torch.int32, device=dev)
    _expect(evict_idx, "evict_idx", (B, Hkv, S), torch.int32, dev)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    st = lib.h2o_update_q8(ctypes.byref(dims), int(pos0), _ptr(scores), _ptr(slot_pos),
                           _ptr(score_inc), _ptr(k_new), _ptr(v_new), _ptr(k_codes),
                           _ptr(k_scales), _ptr(v_codes), _ptr(v_scales),
                           int(M if budget is None else budget), int(recent_window),
                           POLICY[policy], _ptr(evict_idx), _stream(stream))
    _check("h2o_update_q8", st)
    return evict_idx


def h2o_evict_insert_q8(scores, slot_pos, k_new, v_new, k_codes, k_scales, v_codes, v_scales,
                        pos0: int, recent_window: int, policy: str = "h2o", evict_idx=None,
                        budget: int | None = None, Hq: int | None = None, stream=None):
    """h2o_evict_insert on 8-bit buffers, in place.  Returns evict_idx (B,Hkv,S)."""
    lib = load()
    dev = scores.device
    B, Hkv, M = scores.shape
    S, d = k_new.shape[2], k_new.shape[3]
    if policy not in POLICY:
        raise ValueError(f"unknown policy {policy!r}")
    _expect(scores, "scores", (B, Hkv, M), torch.float32, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    _expect(k_new, "k_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect(v_new, "v_new", (B, Hkv, S, d), torch.bfloat16, dev)
    _expect_q8(k_codes, k_scales, v_codes, v_scales, B, Hkv, M, d, dev)
    if evict_idx is None:
        evict_idx = torch.empty((B, Hkv, S), dtype=torch.int32, device=dev)
    _expect(evict_idx, "evict_idx", (B, Hkv, S), torch.int32, dev)
    dims = H2ODims(B, Hkv if Hq is None else Hq, Hkv, d, S, M)
    st = lib.h2o_evict_insert_q8(ctypes.byref(dims), int(pos0), _ptr(scores), _ptr(slot_pos),
                                 _ptr(k_new), _ptr(v_new), _ptr(k_codes), _ptr(k_scales),
                                 _ptr(v_codes), _ptr(v_scales),
                                 int(M if budget is None else budget), int(recent_window),
                                 POLICY[policy], _ptr(evict_idx), _stream(stream))
    _check("h2o_evict_insert_q8", st)
    return evict_idx


def _sdpa_q8(fn, q, k_codes, k_scales, v_codes, v_scales, k_new, v_new, slot_pos, pos0, scale,
             out, score_inc, workspace, stream):
    lib = load()
    dev = q.device
    B, Hq, S, d = q.shape
    Hkv, M = k_codes.shape[1], k_codes.shape[2]
    bf = torch.bfloat16
    cache_only = k_new is None
    nk = M if cache_only else M + S
    _expect(q, "q", (B, Hq, S, d), bf, dev)
    _expect_q8(k_codes, k_scales, v_codes, v_scales, B, Hkv, M, d, dev)
    _expect(slot_pos, "slot_pos", (B, Hkv, M), torch.int32, dev)
    if not cache_only:
        _expect(k_new, "k_new", (B, Hkv, S, d), bf, dev)
        _expect(v_new, "v_new", (B, Hkv, S, d), bf, dev)
    if out is None:
        out = torch.empty((B, Hq, S, d), dtype=bf, device=dev)
    if score_inc is None:
        score_inc = torch.empty((B, Hq, nk), dtype=torch.float32, device=dev)
    _expect(out, "out", (B, Hq, S, d), bf, dev)
    _expect(score_inc, "score_inc", (B, Hq, nk), torch.float32, dev)
    dims = H2ODims(B, Hq, Hkv, d, S, M)
    if workspace is None:
        n = h2o_q8_workspace_size(dims)
        if n:
            workspace = torch.empty(n, dtype=torch.uint8, device=dev)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    head = [ctypes.byref(dims), int(pos0), float(scale), _ptr(q), _ptr(k_codes), _ptr(k_scales),
            _ptr(v_codes), _ptr(v_scales)]
    mid = [] if cache_only else [_ptr(k_new), _ptr(v_new)]
    st = getattr(lib, fn)(*head, *mid, _ptr(slot_pos), _ptr(out), _ptr(score_inc),
                          _ptr(workspace), ws_bytes, _stream(stream))
    _check(fn, st)
    return out, score_inc


def h2o_sdpa_chunk_q8(q, k_codes, k_scales, v_codes, v_scales, k_new, v_new, slot_pos,
                      pos0: int, scale: float = 0.0, out=None, score_inc=None, workspace=None,
                      stream=None):
    """h2o_sdpa_chunk with the cache read through 8-bit buffers (k_new / v_new
    bf16).  Returns (out (B,Hq,S,d) bf16, score_inc (B,Hq,M+S) f32)."""
    return _sdpa_q8("h2o_sdpa_chunk_q8", q, k_codes, k_scales, v_codes, v_scales, k_new, v_new,
                    slot_pos, pos0, scale, out, score_inc, workspace, stream)


def h2o_sdpa_cache_q8(q, k_codes, k_scales, v_codes, v_scales, slot_pos, pos0: int,
                      scale: float = 0.0, out=None, score_inc=None, workspace=None, stream=None):
    """h2o_sdpa_cache with the cache read through 8-bit buffers.  Returns
    (out (B,Hq,S,d) bf16, score_inc (B,Hq,M) f32)."""
    return _sdpa_q8("h2o_sdpa_cache_q8", q, k_codes, k_scales, v_codes, v_scales, None, None,
                    slot_pos, pos0, scale, out, score_inc, workspace, stream)
