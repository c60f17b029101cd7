"""Chunk-loop driver for one attention layer with an H2O cache (§3.1, §A.4.1).

The layer state (cache buffers, slot positions, scores) lives in torch tensors
on the GPU; every step runs the library's calls on the current stream:
``h2o_sdpa_chunk`` then ``h2o_update`` (the default order), or, in the
paper's order, ``h2o_evict_insert``, ``h2o_sdpa_cache`` and ``h2o_scores_add``;
with 8-bit K/V buffers (the setup of §4) the ``_q8`` forms of the same calls.
A sequence is a prefill of M tokens (attending to an empty cache) followed by
chunks of S tokens.
"""
from __future__ import annotations

import torch

from . import _binding as lib


def chunk_bounds(T: int, M: int, S: int):
    """[(start, end)]: the prefill [0, min(T, M)) then chunks of S (last one ragged)."""
    p0 = min(T, M)
    out = [(0, p0)] if p0 else []
    p = p0
    while p < T:
        out.append((p, min(T, p + S)))
        p += S
    return out


class H2OLayer:
    """Device-resident H2O cache state of one layer: M slots per (b, KV head)."""

    def __init__(self, B: int, Hq: int, Hkv: int, d: int, M: int, S: int, W: int,
                 device="cuda", scale: float = 0.0, keep_evictions: bool = True,
                 policy: str = "h2o", order: str = "chunk", kv_bits: int = 16):
        """``policy``: eviction rule of §3.1.1, "h2o", "h2o_norm" or "h2o_orig".
        ``order``: "chunk" (attend to the cache and the chunk, then update) or
        "paper" (§3.1 / §3.3.1: evict and write first, attend to the cache,
        then add the scores).  ``kv_bits``: 16 (bf16 cache rows) or 8 (int8
        codes and a float32 scale per row: k_codes / k_scales / v_codes /
        v_scales instead of k_cache / v_cache)."""
        if order not in ("chunk", "paper"):
            raise ValueError(f"unknown order {order!r}")
        if kv_bits not in (8, 16):
            raise ValueError(f"kv_bits must be 8 or 16, not {kv_bits!r}")
        self.kv_bits = kv_bits
        self.order = order
        self.B, self.Hq, self.Hkv, self.d, self.M, self.S, self.W = B, Hq, Hkv, d, M, S, W
        self.policy = policy
        self.scale = scale
        dev = torch.device(device)
        if kv_bits == 16:
            self.k_cache = torch.zeros((B, Hkv, M, d), dtype=torch.bfloat16, device=dev)
            self.v_cache = torch.zeros_like(self.k_cache)
        else:
            self.k_cache = self.v_cache = None
            self.k_codes = torch.zeros((B, Hkv, M, d), dtype=torch.int8, device=dev)
            self.v_codes = torch.zeros_like(self.k_codes)
            self.k_scales = torch.zeros((B, Hkv, M), dtype=torch.float32, device=dev)
            self.v_scales = torch.zeros_like(self.k_scales)
        self.slot_pos = torch.full((B, Hkv, M), -1, dtype=torch.int32, device=dev)
        self.scores = torch.zeros((B, Hkv, M), dtype=torch.float32, device=dev)
        self._inc = {}
        self._evict = {}
        self._ws = {}
        self.keep_evictions = keep_evictions
        self.device = dev

    def reset(self, stream=None):
        """Empty cache for a new sequence (slot positions -1, scores 0)."""
        lib.h2o_cache_reset(self.slot_pos, self.scores, stream=stream)

    def _buf(self, s: int):
        if s not in self._inc:
            nk = self.M if self.order == "paper" else self.M + s
            self._inc[s] = torch.empty((self.B, self.Hq, nk), dtype=torch.float32,
                                       device=self.device)
            self._evict[s] = torch.empty((self.B, self.Hkv, s), dtype=torch.int32,
                                         device=self.device)
            dims = lib.H2ODims(self.B, self.Hq, self.Hkv, self.d, s, self.M)
            n = (lib.h2o_workspace_size if self.kv_bits == 16 else lib.h2o_q8_workspace_size)(dims)
            self._ws[s] = torch.empty(n, dtype=torch.uint8, device=self.device) if n else None
        return self._inc[s], self._evict[s], self._ws[s]

    def step(self, q, k_new, v_new, pos0: int, out=None, stream=None):
        """One chunk: attend (writes out, score_inc), then update the cache in place.

        Returns (out, score_inc, evict_idx); the last two are reused buffers.
        """
        s = q.shape[2]
        inc, ev, ws = self._buf(s)
        if self.kv_bits == 8:
            return self._step_q8(q, k_new, v_new, pos0, out, stream, inc, ev, ws)
        if self.order == "paper":
            lib.h2o_evict_insert(self.scores, self.slot_pos, k_new, v_new, self.k_cache,
                                 self.v_cache, pos0, self.W, policy=self.policy,
                                 evict_idx=ev if self.keep_evictions else None, Hq=self.Hq,
                                 stream=stream)
            out, inc = lib.h2o_sdpa_cache(q, self.k_cache, self.v_cache, self.slot_pos, pos0,
                                          self.scale, out=out, score_inc=inc, workspace=ws,
                                          stream=stream)
            lib.h2o_scores_add(self.scores, inc, stream=stream)
            return out, inc, ev
        out, inc = lib.h2o_sdpa_chunk(q, self.k_cache, self.v_cache, k_new, v_new, self.slot_pos,
                                      pos0, self.scale, out=out, score_inc=inc, workspace=ws,
                                      stream=stream)
        lib.h2o_update(self.scores, self.slot_pos, inc, k_new, v_new, self.k_cache, self.v_cache,
                       pos0, self.W, evict_idx=ev if self.keep_evictions else None, stream=stream,
                       policy=self.policy)
        return out, inc, ev

    def _step_q8(self, q, k_new, v_new, pos0, out, stream, inc, ev, ws):
        buf = (self.k_codes, self.k_scales, self.v_codes, self.v_scales)
        if self.order == "paper":
            lib.h2o_evict_insert_q8(self.scores, self.slot_pos, k_new, v_new, *buf, pos0, self.W,
                                    policy=self.policy, evict_idx=ev, Hq=self.Hq, stream=stream)
            out, inc = lib.h2o_sdpa_cache_q8(q, *buf, self.slot_pos, pos0, self.scale, out=out,
                                             score_inc=inc, workspace=ws, stream=stream)
            lib.h2o_scores_add(self.scores, inc, stream=stream)
            return out, inc, ev
        out, inc = lib.h2o_sdpa_chunk_q8(q, *buf, k_new, v_new, self.slot_pos, pos0, self.scale,
                                         out=out, score_inc=inc, workspace=ws, stream=stream)
        lib.h2o_update_q8(self.scores, self.slot_pos, inc, k_new, v_new, *buf, pos0, self.W,
                          policy=self.policy, evict_idx=ev, stream=stream)
        return out, inc, ev
