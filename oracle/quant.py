"""Oracle for 8-bit K/V cache buffers (the setup of §4 stores the KV cache
buffers in 8 bits; the paper names the library it used and nothing more).

TEST INFRASTRUCTURE ONLY (see oracle/h2o_oracle.py): only tests/, smoke() and
bench.py's CPU-baseline leg use it.  It shares no code with the CUDA library.

Readings where the paper is silent (also listed in the design notes):

* Format: every cache row of d elements (one token's key, or its value, in one
  KV head) is stored as d signed 8-bit codes c and one float32 scale s,
  symmetric and per row: s = max_e |x_e| / 127 and c_e = round(x_e / s),
  rounded half to even and clipped to [-127, 127].  An all-zero row has s = 0
  and codes 0.  The division and the rounding are done in float32 (the inputs
  are bf16 values, exact in float32), so both implementations take the same
  integer decisions.
* Reading a row back: x_hat = bf16(float32(c) * s), the product in float32,
  rounded to bf16 (nearest, ties to even).  The SDPA then attends to x_hat
  exactly as it attends to a bf16 cache: it computes in the model's dtype.
* The chunk's own new keys and values are bf16 (they come from the current
  projection); they are quantised when they are written into the buffers.
  In the paper's order (write first, then attend) the SDPA therefore reads
  every row, the chunk's included, through x_hat.
* Selection of the slots to overwrite is the same as with bf16 buffers: it
  depends on scores and positions only.

Parity: pinned by the not-gpu tests (hand rows with known codes, the
round-trip bound |x - s c| <= s / 2, sign symmetry, brute-force nearest code,
exact dequantisation when s is a power of two, and the SDPA / update paths
reducing to the pinned bf16 oracle on the dequantised rows).
"""
from __future__ import annotations

import numpy as np

from . import h2o_oracle

__all__ = ["quantize_rows", "dequantize_rows", "round_to_bf16", "sdpa_cache_q8",
           "sdpa_chunk_q8", "evict_insert_q8", "update_q8"]

QMAX = 127


def round_to_bf16(x):
    """float32 values rounded to the nearest bfloat16 (ties to even), returned
    as float32.  Finite inputs only."""
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    lsb = (u >> 16) & 1
    r = ((u + 0x7FFF + lsb) >> 16) << 16
    return r.astype(np.uint32).view(np.float32)


def quantize_rows(x):
    """Rows (..., d) of bf16-exact values -> (codes int8 (..., d), scales
    float32 (...)): s = max|x| / 127 in float32, c = rint(x / s) in float32,
    clipped to [-127, 127]; s = 0 gives codes 0."""
    x = np.asarray(x, np.float32)
    amax = np.abs(x).max(axis=-1)
    s = (amax / np.float32(QMAX)).astype(np.float32)
    codes = np.zeros(x.shape, np.int8)
    nz = s > 0
    ratio = (x[nz] / s[nz][..., None]).astype(np.float32)
    codes[nz] = np.clip(np.rint(ratio), -QMAX, QMAX).astype(np.int8)
    return codes, s


def dequantize_rows(codes, scales):
    """The bf16 values the SDPA reads back: bf16(float32(c) * s), as float32."""
    prod = (np.asarray(codes, np.float32) * np.asarray(scales, np.float32)[..., None])
    return round_to_bf16(prod.astype(np.float32))


def sdpa_cache_q8(q, k_codes, k_scales, v_codes, v_scales, slot_pos, pos0: int,
                  scale: float | None = None, rows=None):
    """``h2o_oracle.sdpa_cache`` over the dequantised buffers."""
    return h2o_oracle.sdpa_cache(q, dequantize_rows(k_codes, k_scales),
                                 dequantize_rows(v_codes, v_scales), slot_pos, pos0, scale, rows)


def sdpa_chunk_q8(q, k_codes, k_scales, v_codes, v_scales, k_new, v_new, slot_pos, pos0: int,
                  scale: float | None = None, rows=None):
    """``h2o_oracle.sdpa_chunk`` with the cache read through the 8-bit buffers and
    the chunk's own keys and values in bf16."""
    return h2o_oracle.sdpa_chunk(q, dequantize_rows(k_codes, k_scales),
                                 dequantize_rows(v_codes, v_scales), k_new, v_new, slot_pos,
                                 pos0, scale, rows)


def _write_q8(sel, k_new, v_new, k_codes, k_scales, v_codes, v_scales):
    """Quantises the chunk's rows into the slots ``sel`` (B, H_kv, S) of copies
    of the buffers."""
    kc, ks = np.array(k_codes, copy=True), np.array(k_scales, np.float32, copy=True)
    vc, vs = np.array(v_codes, copy=True), np.array(v_scales, np.float32, copy=True)
    qk, sk = quantize_rows(k_new)
    qv, sv = quantize_rows(v_new)
    B, Hkv, S = sel.shape
    for b in range(B):
        for h in range(Hkv):
            for c in range(S):
                e = sel[b, h, c]
                kc[b, h, e], ks[b, h, e] = qk[b, h, c], sk[b, h, c]
                vc[b, h, e], vs[b, h, e] = qv[b, h, c], sv[b, h, c]
    return kc, ks, vc, vs


def evict_insert_q8(scores, slot_pos, k_new, v_new, k_codes, k_scales, v_codes, v_scales,
                    pos0: int, recent_window: int, precision: str = "fp32", policy: str = "h2o"):
    """``h2o_oracle.evict_insert`` on 8-bit buffers: the same slots, scores and
    positions; the chosen slots take the chunk's rows quantised."""
    B, Hkv, M = slot_pos.shape
    S, d = k_new.shape[2], k_new.shape[3]
    blank = np.zeros((B, Hkv, M, d), np.float32)
    res = h2o_oracle.evict_insert(scores, slot_pos, k_new, v_new, blank, blank, pos0,
                                  recent_window, precision, policy)
    kc, ks, vc, vs = _write_q8(res["evict_idx"], k_new, v_new, k_codes, k_scales, v_codes,
                               v_scales)
    return dict(scores=res["scores"], slot_pos=res["slot_pos"], evict_idx=res["evict_idx"],
                k_codes=kc, k_scales=ks, v_codes=vc, v_scales=vs)


def update_q8(scores, slot_pos, score_inc, k_new, v_new, k_codes, k_scales, v_codes, v_scales,
              pos0: int, recent_window: int, precision: str = "fp32", policy: str = "h2o"):
    """``h2o_oracle.update`` on 8-bit buffers: the same selection, scores and
    positions; the evicted slots take the chunk's rows quantised."""
    B, Hkv, M = slot_pos.shape
    d = k_new.shape[3]
    blank = np.zeros((B, Hkv, M, d), np.float32)
    res = h2o_oracle.update(scores, slot_pos, score_inc, k_new, v_new, blank, blank, pos0,
                            recent_window, precision, policy)
    kc, ks, vc, vs = _write_q8(res["evict_idx"], k_new, v_new, k_codes, k_scales, v_codes,
                               v_scales)
    return dict(scores=res["scores"], slot_pos=res["slot_pos"], evict_idx=res["evict_idx"],
                k_codes=kc, k_scales=ks, v_codes=vc, v_scales=vs)
