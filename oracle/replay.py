"""Exact oracle for the replay-cache row operations of §3.2 / §A.1.1.

TEST INFRASTRUCTURE ONLY (see oracle/h2o_oracle.py): only tests/ use it.

A chunk's cache write is a scatter along the slot axis,
``keys' = scatter(keys, index, key_new)``, and it is undone by the reverse
recurrence (§3.2): ``delta_key = gather(keys, index)`` taken before the write,
then ``keys = scatter(keys', index, delta_key)``.  The slot positions follow
the same recurrence (the c-th row of a chunk at position pos0 + c).  These are
bit copies: no arithmetic, so every check is exact.
"""
from __future__ import annotations

import numpy as np

__all__ = ["kv_replace", "kv_restore"]


def kv_replace(k_cache, v_cache, slot_pos, index, k_new, v_new, pos0: int):
    """Writes the chunk's rows into the slots ``index`` (B, H_kv, S), distinct per
    (b, h), and returns the rows and positions they replace.

    Returns a dict: k_cache, v_cache, slot_pos (new buffers; inputs unchanged),
    delta_k, delta_v (B, H_kv, S, d) and delta_pos (B, H_kv, S).
    """
    index = np.asarray(index)
    B, Hkv, S = index.shape
    out_k = np.array(k_cache, copy=True)
    out_v = np.array(v_cache, copy=True)
    out_pos = np.array(slot_pos, dtype=np.int32, copy=True)
    d = out_k.shape[-1]
    delta_k = np.zeros((B, Hkv, S, d), out_k.dtype)
    delta_v = np.zeros((B, Hkv, S, d), out_v.dtype)
    delta_pos = np.zeros((B, Hkv, S), np.int32)
    for b in range(B):
        for h in range(Hkv):
            assert len(set(index[b, h].tolist())) == S, "index must be distinct per (b, h)"
            for c in range(S):
                e = index[b, h, c]
                delta_k[b, h, c] = k_cache[b, h, e]      # gather before the write
                delta_v[b, h, c] = v_cache[b, h, e]
                delta_pos[b, h, c] = slot_pos[b, h, e]
                out_k[b, h, e] = k_new[b, h, c]          # scatter
                out_v[b, h, e] = v_new[b, h, c]
                out_pos[b, h, e] = pos0 + c
    return dict(k_cache=out_k, v_cache=out_v, slot_pos=out_pos, delta_k=delta_k,
                delta_v=delta_v, delta_pos=delta_pos)


def kv_restore(k_cache, v_cache, slot_pos, index, delta_k, delta_v, delta_pos):
    """The reverse recurrence: scatter the saved rows and positions back."""
    index = np.asarray(index)
    B, Hkv, S = index.shape
    out_k = np.array(k_cache, copy=True)
    out_v = np.array(v_cache, copy=True)
    out_pos = np.array(slot_pos, dtype=np.int32, copy=True)
    for b in range(B):
        for h in range(Hkv):
            for c in range(S):
                e = index[b, h, c]
                out_k[b, h, e] = delta_k[b, h, c]
                out_v[b, h, e] = delta_v[b, h, c]
                out_pos[b, h, e] = delta_pos[b, h, c]
    return dict(k_cache=out_k, v_cache=out_v, slot_pos=out_pos)
