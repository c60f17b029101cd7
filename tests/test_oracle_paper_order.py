"""Pins of the oracle's paper-order chunk step (§3.1 last paragraph, §3.3.1):
evict on the scores before the chunk attends, write the chunk's K/V into the
freed slots, run SDPA over the M cache slots under the position mask, then add
the chunk's summed weights to the scores (Eq. 3).

Each check ties the oracle to something other than itself: dense causal
attention, the independently pinned default-order oracle (attend, then evict) where no eviction
happens, closed forms, invariants and brute-force enumeration.
"""
import itertools
import math

import numpy as np
import pytest
import torch

from oracle import (evict_insert, run_sequence, scores_add, sdpa_cache, sdpa_chunk,
                    step_paper_order)
from paper_2608_19920_gb300 import workloads as wl


def _rand_seq(rng, B, Hq, Hkv, T, d):
    q = wl.round_bf16(rng.standard_normal((B, Hq, T, d), dtype=np.float32))
    k = wl.round_bf16(rng.standard_normal((B, Hkv, T, d), dtype=np.float32))
    v = wl.round_bf16(rng.standard_normal((B, Hkv, T, d), dtype=np.float32))
    return q, k, v


def _dense_causal(q, k, v):
    """Dense causal attention via torch's SDPA (float64, CPU) with GQA expansion."""
    qg = q.shape[1] // k.shape[1]
    qt = torch.from_numpy(np.asarray(q, np.float64))
    kt = torch.from_numpy(np.asarray(k, np.float64)).repeat_interleave(qg, dim=1)
    vt = torch.from_numpy(np.asarray(v, np.float64)).repeat_interleave(qg, dim=1)
    out = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)
    T = q.shape[2]
    causal = torch.ones(T, T, dtype=torch.bool).tril()
    logits = (qt @ kt.transpose(-1, -2)) / math.sqrt(q.shape[-1])
    weights = torch.softmax(logits.masked_fill(~causal, float("-inf")), dim=-1)
    return out.numpy(), weights.numpy()


@pytest.mark.parametrize("prefill,S", [(12, 8), (5, 7), (1, 1)])
def test_paper_order_without_eviction_equals_dense_causal(prefill, S):
    """M >= T: every chunk lands in empty slots, left to right (§3.1); the output
    is dense causal attention and each score the dense column sum from its
    token on (Eq. 3 with no eviction)."""
    rng = np.random.default_rng(3)
    B, Hq, Hkv, T, d = 2, 4, 2, 37, 16
    q, k, v = _rand_seq(rng, B, Hq, Hkv, T, d)
    out, st = run_sequence(q, k, v, M=48, S=S, W=0, prefill=prefill, order="paper")
    ref_out, weights = _dense_causal(q, k, v)
    np.testing.assert_allclose(out, ref_out, rtol=0, atol=1e-12)
    qg = Hq // Hkv
    for b in range(B):
        for h in range(Hkv):
            np.testing.assert_array_equal(st.slot_pos[b, h, :T], np.arange(T))
            assert (st.slot_pos[b, h, T:] == -1).all()
            for j in range(T):
                ref = weights[b, h * qg:(h + 1) * qg, :, j].sum()
                assert abs(st.scores[b, h, j] - ref) < 1e-12


def test_orders_agree_when_nothing_is_evicted():
    """Without evictions both orders compute the same attention and scores."""
    rng = np.random.default_rng(4)
    q, k, v = _rand_seq(rng, 1, 6, 3, 29, 8)
    o1, s1 = run_sequence(q, k, v, M=32, S=5, W=3, prefill=9, order="chunk")
    o2, s2 = run_sequence(q, k, v, M=32, S=5, W=3, prefill=9, order="paper")
    np.testing.assert_allclose(o1, o2, rtol=0, atol=1e-12)
    np.testing.assert_allclose(s1.scores, s2.scores, rtol=0, atol=1e-12)
    np.testing.assert_array_equal(s1.slot_pos, s2.slot_pos)


def test_rows_sum_to_one_and_hidden_slots_get_nothing():
    """Every query row's weights sum to 1 (§3.1.1), so a chunk adds B Hq S in
    total; slots whose token lies after a row's position, or that are empty,
    get exactly zero from that row."""
    rng = np.random.default_rng(5)
    B, Hq, Hkv, M, d, S, pos0 = 2, 6, 2, 40, 8, 6, 100
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=4)
    q, kn, vn = _rand_seq(rng, B, Hq, Hkv, S, d)
    res = evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                       pos0, 2, "fp64")
    out, inc, _ = sdpa_cache(q, res["k_cache"], res["v_cache"], res["slot_pos"], pos0)
    np.testing.assert_allclose(inc.sum(axis=-1), S, rtol=1e-12)
    qg = Hq // Hkv
    for b in range(B):
        for h in range(Hkv):
            for c in range(1, S):
                e = res["evict_idx"][b, h, c]
                # new token c is seen by rows c..S-1 only: rows < c give it nothing
                _, inc_rows, _ = sdpa_cache(q[b:b + 1, h * qg:(h + 1) * qg, :c],
                                            res["k_cache"][b:b + 1, h:h + 1],
                                            res["v_cache"][b:b + 1, h:h + 1],
                                            res["slot_pos"][b:b + 1, h:h + 1], pos0)
                assert (inc_rows[0, :, e] == 0).all()
            empty = res["slot_pos"][b, h] < 0
            assert (inc[b, h * qg:(h + 1) * qg][:, empty] == 0).all()


def test_evicted_tokens_do_not_influence_the_chunk():
    """The chunk attends after the eviction: the evicted slots' old K/V cannot
    change its output (unlike the default order, where they are visible)."""
    rng = np.random.default_rng(6)
    B, Hq, Hkv, M, d, S, pos0 = 1, 4, 2, 24, 8, 5, 80
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0)
    q, kn, vn = _rand_seq(rng, B, Hq, Hkv, S, d)
    o1, _, r1 = step_paper_order(st["scores"], st["slot_pos"], st["k_cache"], st["v_cache"], q,
                                 kn, vn, pos0, 0)
    k2, v2 = st["k_cache"].copy(), st["v_cache"].copy()
    for b in range(B):
        for h in range(Hkv):
            for e in r1["evict_idx"][b, h]:
                k2[b, h, e] = 7.0
                v2[b, h, e] = -5.0
    o2, _, _ = step_paper_order(st["scores"], st["slot_pos"], k2, v2, q, kn, vn, pos0, 0)
    np.testing.assert_array_equal(o1, o2)
    # the default order (attend, then evict) does see them
    a1, _, _ = sdpa_chunk(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], pos0)
    a2, _, _ = sdpa_chunk(q, k2, v2, kn, vn, st["slot_pos"], pos0)
    assert not np.allclose(a1, a2)


def test_zero_queries_closed_form():
    """q = 0: every visible slot gets weight 1 / (number visible).  After a full
    cache of M slots, row i of the chunk sees the M - S kept slots and new
    tokens 0..i, so an old slot collects sum_i 1/(M - S + i + 1) and new token
    c collects sum_{i >= c} 1/(M - S + i + 1)."""
    rng = np.random.default_rng(7)
    B, Hq, Hkv, M, d, S, pos0 = 1, 3, 1, 10, 4, 4, 50
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0)
    q = np.zeros((B, Hq, S, d), np.float32)
    _, kn, vn = _rand_seq(rng, B, Hq, Hkv, S, d)
    res = evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                       pos0, 0, "fp64")
    _, inc, _ = sdpa_cache(q, res["k_cache"], res["v_cache"], res["slot_pos"], pos0)
    old = sum(1.0 / (M - S + i + 1) for i in range(S))
    evicted = set(res["evict_idx"][0, 0].tolist())
    for j in range(M):
        if j in evicted:
            c = res["slot_pos"][0, 0, j] - pos0
            ref = sum(1.0 / (M - S + i + 1) for i in range(c, S))
        else:
            ref = old
        np.testing.assert_allclose(inc[0, :, j], ref, rtol=1e-13)


def _brute_force(scores, pos, pos0, S, W):
    cand = [j for j in range(len(pos)) if pos[j] < pos0 + S - W]
    key = {j: (-1 if pos[j] < 0 else scores[j]) for j in cand}
    best = None
    for sub in itertools.combinations(cand, S):
        s = sum(key[j] for j in sub)
        if best is None or (s, sub) < best:
            best = (s, sub)
    return list(best[1])


@pytest.mark.parametrize("seed", range(30))
def test_evict_insert_matches_brute_force(seed):
    """The S slots chosen on phi^P (integer scores: exact ties) are the
    minimal-sum subset, ties by the lexicographically smallest slot tuple;
    they take tokens pos0 + c in slot order with score 0."""
    rng = np.random.default_rng(200 + seed)
    M = int(rng.integers(2, 9))
    S = int(rng.integers(1, M + 1))
    W = int(rng.integers(0, S + 2)) if rng.random() < 0.7 else 0
    if M - max(0, W - S) < S:
        W = S
    d, pos0 = 4, 50
    n_empty = int(rng.integers(0, M + 1)) if rng.random() < 0.4 else 0
    st = wl.random_state(rng, 1, 1, M, d, pos0=pos0, n_empty=n_empty, int_scores=True)
    for r in range(max(0, W - S)):
        st["slot_pos"][0, 0, r] = pos0 - 1 - r
    _, kn, vn = _rand_seq(rng, 1, 1, 1, S, d)
    res = evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                       pos0, W, "fp32")
    expect = _brute_force(st["scores"][0, 0], st["slot_pos"][0, 0], pos0, S, W)
    assert list(res["evict_idx"][0, 0]) == expect
    for c, e in enumerate(expect):
        assert res["slot_pos"][0, 0, e] == pos0 + c
        assert res["scores"][0, 0, e] == 0
        np.testing.assert_array_equal(res["k_cache"][0, 0, e], kn[0, 0, c])
    kept = np.setdiff1d(np.arange(M), expect)
    np.testing.assert_array_equal(res["scores"][0, 0, kept], st["scores"][0, 0, kept])
    np.testing.assert_array_equal(res["k_cache"][0, 0, kept], st["k_cache"][0, 0, kept])


@pytest.mark.parametrize("seed", range(12))
def test_evict_insert_policies_match_brute_force(seed):
    """h2o_norm ranks by score / (P - t(j)) (exact rationals here), h2o_orig by
    the score summed over the batch, one choice for every b."""
    from fractions import Fraction
    rng = np.random.default_rng(300 + seed)
    B, M, S, W, d, pos0 = 3, 7, 2, 0, 4, 40
    st = wl.random_state(rng, B, 1, M, d, pos0=pos0, int_scores=True)
    st["slot_pos"][1:] = st["slot_pos"][0]
    _, kn, vn = _rand_seq(rng, B, 1, 1, S, d)
    norm = evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                        pos0, W, "fp64", "h2o_norm")
    orig = evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                        pos0, W, "fp64", "h2o_orig")
    for b in range(B):
        pos = st["slot_pos"][b, 0]
        key = [Fraction(int(st["scores"][b, 0, j])) / (pos0 - int(pos[j])) for j in range(M)]
        assert list(norm["evict_idx"][b, 0]) == _brute_force(key, pos, pos0, S, W)
    tot = st["scores"][:, 0].sum(axis=0)
    shared = _brute_force(tot, st["slot_pos"][0, 0], pos0, S, W)
    for b in range(B):
        assert list(orig["evict_idx"][b, 0]) == shared


def test_scores_add_is_the_group_sum():
    """Eq. 3 over the GQA group: integer-valued weights make the fp32 sum exact."""
    rng = np.random.default_rng(8)
    B, Hkv, qg, M = 2, 3, 4, 11
    scores = rng.integers(0, 50, size=(B, Hkv, M)).astype(np.float32)
    inc = rng.integers(0, 9, size=(B, Hkv * qg, M)).astype(np.float32)
    out = scores_add(scores, inc, "fp32")
    np.testing.assert_array_equal(out, scores + inc.reshape(B, Hkv, qg, M).sum(axis=2))


@pytest.mark.parametrize("policy", ["h2o", "h2o_norm", "h2o_orig"])
def test_paper_order_run_invariants(policy):
    """A long run with evictions: the last W tokens and the current chunk are
    resident, positions are unique, the cache holds exactly the K/V of the
    tokens its positions name, and each chunk's rows sum to 1."""
    rng = np.random.default_rng(9)
    B, Hq, Hkv, T, d, M, S, W = 2, 4, 2, 70, 8, 16, 4, 6
    q, k, v = _rand_seq(rng, B, Hq, Hkv, T, d)
    seen = []

    def on_step(i, bounds, before, res):
        p, e = bounds
        seen.append(res["score_inc"].sum())
        for b in range(B):
            for h in range(Hkv):
                pos = res["slot_pos"][b, h]
                occ = pos[pos >= 0]
                assert len(np.unique(occ)) == len(occ)
                assert set(range(max(0, e - W), e)) <= set(occ.tolist())
                for j, t in enumerate(pos):
                    if t >= 0:
                        np.testing.assert_array_equal(res["k_cache"][b, h, j], k[b, h, t])
                if policy == "h2o_orig":
                    np.testing.assert_array_equal(pos, res["slot_pos"][0, h])

    run_sequence(q, k, v, M=M, S=S, W=W, precision="fp32", on_step=on_step, policy=policy,
                 order="paper")
    sizes = [min(T, M)] + [min(S, T - p) for p in range(M, T, S)]
    np.testing.assert_allclose(seen, [B * Hq * s for s in sizes], rtol=1e-5)
