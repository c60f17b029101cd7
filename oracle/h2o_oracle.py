"""Float64 CPU oracle for the H2O sparse-attention chunk step and cache update.

TEST INFRASTRUCTURE ONLY.  Nothing on the product path may import or call
this module: only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline
leg of ``bench.py`` use it.  It shares no code with the CUDA library.

It is a plain, slow, literal restatement of what the paper defines:

* ``sdpa_chunk``: scaled dot product attention of §3.1, Eq. 2, with the
  position-based causal mask of §3.1 / §3.3.1 (a key with token position t(j)
  is hidden from query row i iff P + i < t(j)), plus the summed attention
  weights sum_i m_ij that §3.3.1 and §A.6 ask the kernel to return, shape
  (B, H_q, N_k).  Empty cache slots (position -1) are hidden as well.
* ``update``: the H2O policy of §3.1.1: the score of Eq. 3 is the running sum
  of attention weights a slot received since its token entered the cache; the
  S slots with the smallest score are overwritten by the chunk's keys and
  values (the scatter of §3.2 / §A.1.1), with the readings listed below.
* ``run_sequence``: prefill then chunks (§3.1 last paragraph, §A.4.1).

Readings where the paper is silent (each is also listed in the design notes):

* Order within a chunk step: the chunk attends to the M cache slots plus,
  causally, to itself (N_k = M + S); its attention weights are added to the
  scores; then S slots are evicted and overwritten.
* GQA: query head hq belongs to KV head hq // q_g; the score of a KV-head slot
  is the sum of its q_g query heads' summed weights.
* Recent window W: a slot whose token position is >= P + S - W is not a
  candidate for eviction.  Empty slots rank before every occupied slot.
* Total order for eviction: (empty first, score ascending, slot ascending);
  the c-th smallest evicted slot index receives the chunk's c-th token.
* The new slot's score is the summed weight its own column received in this
  chunk (Eq. 3 sums over s >= t(j), and the chunk's queries are s >= t(j)).
* Policy variants of §3.1.1 (``policy``): ``"h2o"`` ranks occupied slots by
  their score; ``"h2o_norm"`` by the normalized score, score / (t - t(j)) with
  t = P + S the number of tokens processed once the chunk is in (the stored
  scores stay unnormalized); ``"h2o_orig"`` ranks the slots of KV head h by the
  score summed over the batch (ascending b) and evicts the same slots in every
  batch entry, whose positions are read from batch entry 0 (they are identical
  across the batch when every update used this policy since a reset).
* Scores accumulate in one of two precisions: ``"fp64"`` (the oracle's own
  trajectory) or ``"fp32"``, which adds, in float32, the q_g query heads in
  ascending order (t = inc_0; t = t + inc_g) and then ``scores + t``; that is
  the order any implementation must follow to be compared bit for bit.

The paper's own order of a chunk step (§3.1 last paragraph, §3.3.1: the new
keys and values are written into the cache first, then SDPA runs over the
N_C = M slots under the position mask) is the second path here:
``evict_insert`` (the S slots with the smallest score phi^P, before this
chunk's attention, take the chunk's tokens; their scores restart at 0),
``sdpa_cache`` (N_k = M) and ``scores_add`` (Eq. 3 with this chunk's weights),
chained by ``step_paper_order`` and ``run_sequence(order="paper")``.  Its
readings: the same candidate rule (positions >= P + S - W protected, empty
first, score, slot) and token-to-slot assignment as ``update``; h2o_norm
divides by t - t(j) with t = P, the tokens processed when the choice is made.

Parity: every function here is pinned by the not-gpu tests against dense
causal attention, closed forms, the summed-weights identity of §A.6.2,
invariants of §3.1-§3.3 and brute-force enumeration.
"""
from __future__ import annotations

import math

import numpy as np

__all__ = ["sdpa_chunk", "update", "run_sequence", "SequenceState", "lse_merge",
           "chunk_bounds", "POLICIES", "sdpa_cache", "evict_insert", "scores_add",
           "step_paper_order"]


def _token_positions(slot_pos_bh: np.ndarray, pos0: int, S: int) -> np.ndarray:
    """Token position of every key column: cache slots first, then the chunk's S tokens."""
    return np.concatenate([slot_pos_bh.astype(np.int64), pos0 + np.arange(S, dtype=np.int64)])


def sdpa_chunk(q, k_cache, v_cache, k_new, v_new, slot_pos, pos0: int, scale: float | None = None,
               rows=None):
    """One chunk of H2O sparse SDPA (§3.1 Eq. 2 + summed weights of §3.3.1 / §A.6).

    Args:
      q: (B, H_q, S, d) queries of tokens pos0 .. pos0+S-1.
      k_cache, v_cache: (B, H_kv, M, d) cache buffers.
      k_new, v_new: (B, H_kv, S, d) keys/values of the chunk's tokens.
      slot_pos: (B, H_kv, M) int token position per slot, -1 = empty.
      pos0: P, the number of tokens processed before this chunk.
      scale: softmax scale, default d**-0.5 (Eq. 2).

    Returns (out (B,H_q,S,d), score_inc (B,H_q,M+S), lse (B,H_q,S)), float64.
    Key columns are ordered cache slots 0..M-1, then chunk tokens 0..S-1.
    ``rows`` (optional) restricts the computation to those query rows i: out and
    lse then have len(rows) rows and score_inc sums over those rows only.
    """
    q = np.asarray(q, np.float64)
    B, Hq, S, d = q.shape
    ridx = np.arange(S) if rows is None else np.asarray(rows, np.int64)
    Hkv, M = slot_pos.shape[1], slot_pos.shape[2]
    assert Hq % Hkv == 0
    qg = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    out = np.zeros((B, Hq, len(ridx), d))
    score_inc = np.zeros((B, Hq, M + S))
    lse = np.zeros((B, Hq, len(ridx)))
    for b in range(B):
        for hq in range(Hq):
            h = hq // qg
            keys = np.concatenate([np.asarray(k_cache[b, h], np.float64),
                                   np.asarray(k_new[b, h], np.float64)])
            vals = np.concatenate([np.asarray(v_cache[b, h], np.float64),
                                   np.asarray(v_new[b, h], np.float64)])
            t = _token_positions(slot_pos[b, h], pos0, S)
            # mask: hidden iff the slot is empty or P + i < t(j)  (§3.3.1)
            qpos = pos0 + ridx[:, None]
            visible = (t[None, :] >= 0) & (t[None, :] <= qpos)
            a = scale * (q[b, hq][ridx] @ keys.T)
            a = np.where(visible, a, -np.inf)
            amax = a.max(axis=1, keepdims=True)
            lam = amax + np.log(np.exp(a - amax).sum(axis=1, keepdims=True))
            m = np.where(visible, np.exp(a - lam), 0.0)
            out[b, hq] = m @ vals
            score_inc[b, hq] = m.sum(axis=0)
            lse[b, hq] = lam[:, 0]
    return out, score_inc, lse


def lse_merge(l1, l2):
    """Combine log-sum-exp values of two disjoint column sets (§A.6.1)."""
    l1 = np.asarray(l1, np.float64)
    l2 = np.asarray(l2, np.float64)
    return np.maximum(l1, l2) + np.log1p(np.exp(-np.abs(l1 - l2)))


POLICIES = ("h2o", "h2o_norm", "h2o_orig")


def update(scores, slot_pos, score_inc, k_new, v_new, k_cache, v_cache, pos0: int,
           recent_window: int, precision: str = "fp32", policy: str = "h2o"):
    """H2O score accumulation, eviction and K/V write (§3.1.1 Eq. 3, §3.2, §A.1.1).

    ``policy`` selects the ranking of §3.1.1 (see the module notes).  Inputs
    are not modified.  Returns a dict with new ``scores`` (float32 or float64),
    ``slot_pos``, ``k_cache``, ``v_cache`` and ``evict_idx`` (B, H_kv, S)
    int32: slot receiving token pos0 + c, ascending in c.
    """
    if policy not in POLICIES:
        raise ValueError(f"unknown policy {policy!r}")
    B, Hkv, M = slot_pos.shape
    Bq, Hq, N = score_inc.shape
    S = N - M
    assert Bq == B and Hq % Hkv == 0 and 1 <= S <= M
    qg = Hq // Hkv
    W = recent_window
    if W < 0 or W > M:
        raise ValueError("recent_window must lie in [0, M]")
    ft = np.float32 if precision == "fp32" else np.float64
    inc = np.asarray(score_inc, ft)
    out_scores = np.array(scores, dtype=ft, copy=True)
    out_pos = np.array(slot_pos, dtype=np.int32, copy=True)
    out_k = np.array(k_cache, copy=True)
    out_v = np.array(v_cache, copy=True)
    evict = np.zeros((B, Hkv, S), np.int32)
    acc = np.zeros((B, Hkv, M), ft)
    new = np.zeros((B, Hkv, S), ft)
    for b in range(B):
        for h in range(Hkv):
            # group sum over the q_g query heads of KV head h, ascending order
            t = inc[b, h * qg].copy()
            for g in range(1, qg):
                t = t + inc[b, h * qg + g]
            acc[b, h] = out_scores[b, h] + t[:M]    # Eq. 3: accumulate this chunk
            new[b, h] = t[M:]                        # scores of the chunk's own tokens

    def choose(rank_score, pos):
        """S smallest candidates under (empty first, rank_score, slot)."""
        cand = np.nonzero(pos < pos0 + S - W)[0]    # the recent window is protected
        if cand.size < S:
            raise ValueError("fewer eviction candidates than chunk tokens")
        occupied = pos[cand] >= 0
        rank0 = occupied.astype(np.int64)                   # 0 = empty: ranks first
        rank1 = np.where(occupied, rank_score[cand], 0)     # empties tie, broken by slot
        order = np.lexsort((cand, rank1, rank0))
        return np.sort(cand[order[:S]])

    for h in range(Hkv):
        if policy == "h2o_orig":
            tot = acc[0, h].copy()
            for b in range(1, B):
                tot = tot + acc[b, h]
            shared = choose(tot, out_pos[0, h])
        for b in range(B):
            pos = out_pos[b, h]
            if policy == "h2o":
                chosen = choose(acc[b, h], pos)
            elif policy == "h2o_norm":
                age = np.maximum(pos0 + S - pos.astype(np.int64), 1).astype(ft)
                chosen = choose(acc[b, h] / age, pos)
            else:
                chosen = shared
            evict[b, h] = chosen
            out_scores[b, h] = acc[b, h]
            for c, e in enumerate(chosen):            # scatter along the slot axis
                out_k[b, h, e] = k_new[b, h, c]
                out_v[b, h, e] = v_new[b, h, c]
                out_pos[b, h, e] = pos0 + c
                out_scores[b, h, e] = new[b, h, c]
    return dict(scores=out_scores, slot_pos=out_pos, k_cache=out_k, v_cache=out_v,
                evict_idx=evict)


def sdpa_cache(q, k_cache, v_cache, slot_pos, pos0: int, scale: float | None = None, rows=None):
    """SDPA over the M cache slots only, the chunk's own keys already written
    there (the paper's order: §3.1 Eq. 2 with N_k = N_C, mask of §3.3.1).

    Query row i (token pos0 + i) sees slot j iff 0 <= slot_pos[j] <= pos0 + i.
    Returns (out (B,H_q,S,d), score_inc (B,H_q,M), lse (B,H_q,S)), float64;
    ``rows`` as in ``sdpa_chunk``.
    """
    q = np.asarray(q, np.float64)
    B, Hq, S, d = q.shape
    ridx = np.arange(S) if rows is None else np.asarray(rows, np.int64)
    Hkv, M = slot_pos.shape[1], slot_pos.shape[2]
    assert Hq % Hkv == 0
    qg = Hq // Hkv
    if scale is None:
        scale = 1.0 / math.sqrt(d)
    out = np.zeros((B, Hq, len(ridx), d))
    score_inc = np.zeros((B, Hq, M))
    lse = np.zeros((B, Hq, len(ridx)))
    for b in range(B):
        for hq in range(Hq):
            h = hq // qg
            keys = np.asarray(k_cache[b, h], np.float64)
            vals = np.asarray(v_cache[b, h], np.float64)
            t = slot_pos[b, h].astype(np.int64)
            qpos = pos0 + ridx[:, None]
            visible = (t[None, :] >= 0) & (t[None, :] <= qpos)
            a = scale * (q[b, hq][ridx] @ keys.T)
            a = np.where(visible, a, -np.inf)
            amax = a.max(axis=1, keepdims=True)
            lam = amax + np.log(np.exp(a - amax).sum(axis=1, keepdims=True))
            m = np.where(visible, np.exp(a - lam), 0.0)
            out[b, hq] = m @ vals
            score_inc[b, hq] = m.sum(axis=0)
            lse[b, hq] = lam[:, 0]
    return out, score_inc, lse


def evict_insert(scores, slot_pos, k_new, v_new, k_cache, v_cache, pos0: int,
                 recent_window: int, precision: str = "fp32", policy: str = "h2o"):
    """First part of the paper-order chunk step (§3.1, §3.1.1, scatter of §3.2):
    per (b, kv head) the S slots with the smallest score phi^P (this chunk has
    not attended yet) receive the chunk's keys and values; the c-th smallest
    evicted slot gets token pos0 + c and a score of 0.  Candidates, total
    order and policies as in ``update``, with t = pos0 for h2o_norm.

    Inputs are not modified.  Returns a dict like ``update``'s.
    """
    if policy not in POLICIES:
        raise ValueError(f"unknown policy {policy!r}")
    B, Hkv, M = slot_pos.shape
    S = k_new.shape[2]
    assert 1 <= S <= M
    W = recent_window
    if W < 0 or W > M:
        raise ValueError("recent_window must lie in [0, M]")
    ft = np.float32 if precision == "fp32" else np.float64
    out_scores = np.array(scores, dtype=ft, copy=True)
    out_pos = np.array(slot_pos, dtype=np.int32, copy=True)
    out_k = np.array(k_cache, copy=True)
    out_v = np.array(v_cache, copy=True)
    evict = np.zeros((B, Hkv, S), np.int32)

    def choose(rank_score, pos):
        cand = np.nonzero(pos < pos0 + S - W)[0]
        if cand.size < S:
            raise ValueError("fewer eviction candidates than chunk tokens")
        occupied = pos[cand] >= 0
        rank0 = occupied.astype(np.int64)
        rank1 = np.where(occupied, rank_score[cand], 0)
        order = np.lexsort((cand, rank1, rank0))
        return np.sort(cand[order[:S]])

    for h in range(Hkv):
        if policy == "h2o_orig":
            tot = out_scores[0, h].copy()
            for b in range(1, B):
                tot = tot + out_scores[b, h]
            shared = choose(tot, out_pos[0, h])
        for b in range(B):
            pos = out_pos[b, h]
            if policy == "h2o":
                chosen = choose(out_scores[b, h], pos)
            elif policy == "h2o_norm":
                age = np.maximum(pos0 - pos.astype(np.int64), 1).astype(ft)
                chosen = choose(out_scores[b, h] / age, pos)
            else:
                chosen = shared
            evict[b, h] = chosen
            for c, e in enumerate(chosen):
                out_k[b, h, e] = k_new[b, h, c]
                out_v[b, h, e] = v_new[b, h, c]
                out_pos[b, h, e] = pos0 + c
                out_scores[b, h, e] = 0
    return dict(scores=out_scores, slot_pos=out_pos, k_cache=out_k, v_cache=out_v,
                evict_idx=evict)


def scores_add(scores, score_inc, precision: str = "fp32"):
    """Last part of the paper-order chunk step: Eq. 3 adds this chunk's summed
    weights, summed over the GQA group (ascending g), to every slot's score.

    scores (B, H_kv, M), score_inc (B, H_q, M).  Returns the new scores.
    """
    ft = np.float32 if precision == "fp32" else np.float64
    B, Hkv, M = scores.shape
    inc = np.asarray(score_inc, ft)
    qg = inc.shape[1] // Hkv
    out = np.array(scores, dtype=ft, copy=True)
    for b in range(B):
        for h in range(Hkv):
            t = inc[b, h * qg].copy()
            for g in range(1, qg):
                t = t + inc[b, h * qg + g]
            out[b, h] = out[b, h] + t
    return out


def step_paper_order(scores, slot_pos, k_cache, v_cache, q, k_new, v_new, pos0: int,
                     recent_window: int, precision: str = "fp32", policy: str = "h2o",
                     scale: float | None = None):
    """One chunk in the paper's order: evict_insert, sdpa_cache, scores_add.
    Returns (out, score_inc (B,H_q,M), state dict after the step)."""
    st = evict_insert(scores, slot_pos, k_new, v_new, k_cache, v_cache, pos0, recent_window,
                      precision, policy)
    out, inc, _ = sdpa_cache(q, st["k_cache"], st["v_cache"], st["slot_pos"], pos0, scale)
    st["scores"] = scores_add(st["scores"], inc, precision)
    return out, inc, st


class SequenceState:
    """Cache state of one attention layer: buffers of fixed length M (§3.1)."""

    def __init__(self, B, Hkv, M, d, dtype=np.float32, score_dtype=np.float64):
        self.k_cache = np.zeros((B, Hkv, M, d), dtype)
        self.v_cache = np.zeros((B, Hkv, M, d), dtype)
        self.slot_pos = -np.ones((B, Hkv, M), np.int32)
        self.scores = np.zeros((B, Hkv, M), score_dtype)


def chunk_bounds(T: int, M: int, S: int, prefill: int | None = None):
    """[(start, end)] of the prefill chunk (default length M) then chunks of S (§A.4.1)."""
    P0 = min(T, M if prefill is None else prefill)
    bounds = [(0, P0)] if P0 > 0 else []
    p = P0
    while p < T:
        bounds.append((p, min(T, p + S)))
        p += S
    return bounds


def run_sequence(q, k, v, M: int, S: int, W: int, prefill: int | None = None,
                 scale: float | None = None, precision: str = "fp64", on_step=None,
                 policy: str = "h2o", order: str = "chunk"):
    """Sparse-attention pass over whole sequences: prefill, then chunks of S.

    q (B,H_q,T,d), k/v (B,H_kv,T,d).  Returns (out (B,H_q,T,d), final state).
    ``order``: "chunk" (attend to the cache plus the chunk, then update) or
    "paper" (evict and write first, then attend to the cache, then add scores).
    ``on_step(i, bounds, state_before, result)`` is called after every chunk.
    """
    if order not in ("chunk", "paper"):
        raise ValueError(f"unknown order {order!r}")
    B, Hq, T, d = q.shape
    Hkv = k.shape[1]
    st = SequenceState(B, Hkv, M, d, score_dtype=np.float64 if precision == "fp64" else np.float32)
    out = np.zeros((B, Hq, T, d))
    for i, (p, e) in enumerate(chunk_bounds(T, M, S, prefill)):
        if order == "paper":
            o, inc, res = step_paper_order(st.scores, st.slot_pos, st.k_cache, st.v_cache,
                                           q[:, :, p:e], k[:, :, p:e], v[:, :, p:e], p, W,
                                           precision, policy, scale)
        else:
            o, inc, _ = sdpa_chunk(q[:, :, p:e], st.k_cache, st.v_cache, k[:, :, p:e],
                                   v[:, :, p:e], st.slot_pos, p, scale)
            res = update(st.scores, st.slot_pos, inc, k[:, :, p:e], v[:, :, p:e],
                         st.k_cache, st.v_cache, p, W, precision, policy)
        out[:, :, p:e] = o
        before = (st.scores, st.slot_pos, st.k_cache, st.v_cache)
        st.scores, st.slot_pos = res["scores"], res["slot_pos"]
        st.k_cache, st.v_cache = res["k_cache"], res["v_cache"]
        if on_step is not None:
            on_step(i, (p, e), before, dict(out=o, score_inc=inc, **res))
    return out, st
