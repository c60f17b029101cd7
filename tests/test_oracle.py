"""Pins for the float64 oracle: checks against things other than the oracle itself.

* dense causal attention (a library routine) when the cache never evicts,
* the FlexAttention two-call identity for summed weights (§A.6.2),
* closed forms (all-zero queries, a single visible key),
* hand-derived worked examples (tests/golden/hand_example.json),
* brute-force enumeration of eviction sets on tiny inputs,
* invariants stated by the paper (rows of weights sum to 1, §3.1.1; only S
  slots change per chunk, §3.2; new tokens enter the cache, §3.3.1; S = M
  overwrites everything, §3.3).
"""
import itertools
from fractions import Fraction
import json
import math
import os

import numpy as np
import pytest
import torch
from scipy.special import logsumexp

from oracle import chunk_bounds, lse_merge, run_sequence, sdpa_chunk, update
from paper_2608_19920_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_example.json")


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
def test_no_eviction_equals_dense_causal(prefill, S):
    """Cache at least as long as the sequence: chunked H2O SDPA is exact causal attention."""
    rng = np.random.default_rng(1)
    B, Hq, Hkv, T, d = 2, 4, 2, 37, 16
    q, k, v = _rand_seq(rng, B, Hq, Hkv, T, d)
    out, st = run_sequence(q, k, v, M=48, S=S, W=0, prefill=prefill)
    ref_out, weights = _dense_causal(q, k, v)
    np.testing.assert_allclose(out, ref_out, rtol=0, atol=1e-12)
    # Eq. 3 with no eviction: score of the slot holding token t is the sum over
    # queries s >= t of the dense weights, summed over the q_g query heads.
    qg = Hq // Hkv
    for b in range(B):
        for h in range(Hkv):
            for j, t in enumerate(st.slot_pos[b, h]):
                if t < 0:
                    assert st.scores[b, h, j] == 0
                    continue
                ref = weights[b, h * qg:(h + 1) * qg, :, t].sum()
                assert abs(st.scores[b, h, j] - ref) < 1e-12
    # slots fill left to right (§3.1): slot j holds token j
    for b in range(B):
        for h in range(Hkv):
            np.testing.assert_array_equal(st.slot_pos[b, h, :T], np.arange(T))
            assert (st.slot_pos[b, h, T:] == -1).all()


def _state(rng, B, Hkv, M, d, pos0, n_empty=0, int_scores=False):
    return wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty, int_scores=int_scores)


def test_summed_weights_match_flex_two_call_identity():
    """§A.6.2: w = exp(lam~ - lam_bar) * SDPA_rev(K, Q, exp(-(lam - lam_bar))) with the mask flipped."""
    rng = np.random.default_rng(2)
    B, Hq, Hkv, M, S, d, pos0 = 1, 4, 2, 24, 6, 8, 40
    st = _state(rng, B, Hkv, M, d, pos0, n_empty=3)
    q, kn, vn = _rand_seq(rng, B, Hq, Hkv, S, d)
    st["slot_pos"][0, 0, 5] = pos0 + 2   # a slot that only some queries may see (§3.3.1 mask)
    _, inc, _ = sdpa_chunk(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], pos0)
    qg = Hq // Hkv
    scale = 1.0 / math.sqrt(d)
    for hq in range(Hq):
        h = hq // qg
        keys = torch.from_numpy(np.concatenate([st["k_cache"][0, h], kn[0, h]]).astype(np.float64))
        tpos = np.concatenate([st["slot_pos"][0, h], pos0 + np.arange(S)])
        vis = torch.from_numpy((tpos[None, :] >= 0) & (tpos[None, :] <= pos0 + np.arange(S)[:, None]))
        qq = torch.from_numpy(q[0, hq].astype(np.float64))
        a = (qq @ keys.T) * scale
        lam = torch.logsumexp(a.masked_fill(~vis, float("-inf")), dim=1)
        lam_bar = lam.mean()
        vals = torch.exp(-(lam - lam_bar))[:, None]                    # (S, 1)
        at = a.T.masked_fill(~vis.T, float("-inf"))                  # flipped roles
        lam_t = torch.logsumexp(at, dim=1)
        seen = vis.any(dim=0)
        y_rev = torch.nn.functional.scaled_dot_product_attention(
            keys[seen][None], qq[None], vals[None], attn_mask=vis.T[seen][None], scale=scale)[0, :, 0]
        w = torch.zeros(M + S, dtype=torch.float64)
        w[seen] = torch.exp(lam_t[seen] - lam_bar) * y_rev
        np.testing.assert_allclose(inc[0, hq], w.numpy(), rtol=1e-12, atol=1e-14)


def test_zero_queries_closed_form():
    """q = 0: every visible logit is 0, so m_ij = 1 / (visible keys of row i)."""
    rng = np.random.default_rng(3)
    B, Hq, Hkv, M, S, d, pos0 = 2, 2, 1, 10, 4, 4, 30
    st = _state(rng, B, Hkv, M, d, pos0, n_empty=4)
    q = np.zeros((B, Hq, S, d), np.float32)
    _, kn, vn = _rand_seq(rng, B, Hq, Hkv, S, d)
    out, inc, lse = sdpa_chunk(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], pos0)
    for b in range(B):
        occ = st["slot_pos"][b, 0] >= 0
        n_occ = occ.sum()
        vals = np.concatenate([st["v_cache"][b, 0], vn[b, 0]]).astype(np.float64)
        for hq in range(Hq):
            expect_inc = np.zeros(M + S)
            for i in range(S):
                n_i = n_occ + i + 1
                assert abs(lse[b, hq, i] - math.log(n_i)) < 1e-12
                vis = np.concatenate([occ, np.arange(S) <= i])
                expect_inc += vis / n_i
                np.testing.assert_allclose(out[b, hq, i], vals[vis].mean(axis=0), atol=1e-12)
            np.testing.assert_allclose(inc[b, hq], expect_inc, atol=1e-12)


def test_single_visible_key():
    """Empty cache, one token: the only visible value is returned with weight 1."""
    rng = np.random.default_rng(4)
    q, kn, vn = _rand_seq(rng, 1, 2, 1, 1, 8)
    M = 5
    out, inc, _ = sdpa_chunk(q, np.zeros((1, 1, M, 8)), np.zeros((1, 1, M, 8)), kn, vn,
                             -np.ones((1, 1, M), np.int32), 0)
    np.testing.assert_allclose(out[0, :, 0], np.repeat(vn[0, :, 0], 2, axis=0), atol=0)
    np.testing.assert_array_equal(inc[0], np.tile([0, 0, 0, 0, 0, 1.0], (2, 1)))


def _golden_array(x):
    def conv(e):
        if isinstance(e, list):
            return [conv(i) for i in e]
        if isinstance(e, str):
            return {"ln2": math.log(2.0), "ln3": math.log(3.0), "ln4": math.log(4.0)}[e]
        return e
    return np.array(conv(x), dtype=np.float64)


@pytest.mark.parametrize("case", json.load(open(GOLDEN))["cases"], ids=lambda c: c["name"])
@pytest.mark.parametrize("precision", ["fp64", "fp32"])
def test_hand_worked_examples(case, precision):
    g = _golden_array
    slot_pos = np.array(case["slot_pos"], np.int32)
    out, inc, _ = sdpa_chunk(g(case["q"]), g(case["k_cache"]), g(case["v_cache"]),
                             g(case["k_new"]), g(case["v_new"]), slot_pos, case["pos0"],
                             scale=case["scale"])
    np.testing.assert_allclose(out, g(case["expect_out"]), atol=1e-12)
    np.testing.assert_allclose(inc, g(case["expect_score_inc"]), atol=1e-12)
    ft = np.float32 if precision == "fp32" else np.float64
    res = update(g(case["scores"]).astype(ft), slot_pos, inc.astype(ft), g(case["k_new"]),
                 g(case["v_new"]), g(case["k_cache"]), g(case["v_cache"]), case["pos0"],
                 case["recent_window"], precision)
    np.testing.assert_array_equal(res["evict_idx"], np.array(case["expect_evict_idx"]))
    np.testing.assert_array_equal(res["slot_pos"], np.array(case["expect_slot_pos"]))
    np.testing.assert_allclose(res["scores"], g(case["expect_scores"]), rtol=1e-6)


def _brute_force_evict(acc, pos, pos0, S, W):
    """All S-subsets of candidates; minimal score sum (empty slot = -1), then lexicographic."""
    cand = [j for j in range(len(pos)) if pos[j] < pos0 + S - W]
    key = {j: (-1 if pos[j] < 0 else acc[j]) for j in cand}
    best = None
    for sub in itertools.combinations(cand, S):
        s = sum(key[j] for j in sub)
        if best is None or (s, sub) < best:
            best = (s, sub)
    return list(best[1])


@pytest.mark.parametrize("seed", range(40))
def test_eviction_matches_brute_force(seed):
    rng = np.random.default_rng(100 + seed)
    M = int(rng.integers(2, 9))
    S = int(rng.integers(1, M + 1))
    W = int(rng.integers(0, S + 2)) if rng.random() < 0.7 else 0
    if M - max(0, W - S) < S:
        W = S
    qg, d, pos0 = 2, 4, 50
    n_empty = int(rng.integers(0, M + 1)) if rng.random() < 0.4 else 0
    st = _state(rng, 1, 1, M, d, pos0, n_empty=n_empty, int_scores=True)
    # keep the recent window consistent with a real run: the W - S most recent
    # old tokens are resident when W > S
    for r in range(max(0, W - S)):
        st["slot_pos"][0, 0, r] = pos0 - 1 - r
    inc = rng.integers(0, 3, size=(1, qg, M + S)).astype(np.float32)
    inc[0, :, :M][:, st["slot_pos"][0, 0] < 0] = 0
    _, kn, vn = _rand_seq(rng, 1, qg, 1, S, d)
    res = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                 pos0, W, "fp32")
    acc = st["scores"][0, 0] + inc[0].sum(axis=0)[:M]
    expect = _brute_force_evict(acc, st["slot_pos"][0, 0], pos0, S, W)
    assert list(res["evict_idx"][0, 0]) == expect
    for c, e in enumerate(expect):
        assert res["slot_pos"][0, 0, e] == pos0 + c
        np.testing.assert_array_equal(res["k_cache"][0, 0, e], kn[0, 0, c])
        np.testing.assert_array_equal(res["v_cache"][0, 0, e], vn[0, 0, c])
        assert res["scores"][0, 0, e] == inc[0, :, M + c].sum()


def test_all_equal_scores_evict_lowest_candidates():
    rng = np.random.default_rng(5)
    M, S, W, pos0, d = 12, 3, 5, 100, 4
    st = _state(rng, 1, 1, M, d, pos0)
    st["slot_pos"][0, 0] = np.array([99, 10, 98, 11, 12, 13, 14, 15, 16, 17, 18, 19])
    st["scores"][:] = 1.0
    inc = np.zeros((1, 2, M + S), np.float32)
    _, kn, vn = _rand_seq(rng, 1, 2, 1, S, d)
    res = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                 pos0, W, "fp32")
    # positions 98, 99 are in the recent window [pos0 + S - W, ...) = [98, ...)
    assert list(res["evict_idx"][0, 0]) == [1, 3, 4]


def test_chunk_equal_to_cache_overwrites_everything():
    """S = M: the whole cache is overwritten and the policy plays no role (§3.3)."""
    rng = np.random.default_rng(6)
    M = S = 6
    st = _state(rng, 2, 2, M, 4, 20)
    inc = rng.random((2, 4, 2 * M)).astype(np.float32)
    _, kn, vn = _rand_seq(rng, 2, 4, 2, S, 4)
    res = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                 20, 0, "fp32")
    assert (res["evict_idx"] == np.arange(M)).all()
    assert (res["slot_pos"] == 20 + np.arange(M)).all()
    np.testing.assert_array_equal(res["k_cache"], kn)


def test_too_few_candidates_is_an_error():
    rng = np.random.default_rng(7)
    st = _state(rng, 1, 1, 4, 4, 10)
    st["slot_pos"][0, 0] = [9, 8, 7, 1]
    _, kn, vn = _rand_seq(rng, 1, 1, 1, 2, 4)
    with pytest.raises(ValueError):
        update(st["scores"], st["slot_pos"], np.zeros((1, 1, 6), np.float32), kn, vn,
               st["k_cache"], st["v_cache"], 10, 5, "fp32")


@pytest.mark.parametrize("S,W,prefill", [(32, 32, None), (16, 48, None), (24, 8, 100)])
def test_run_invariants(S, W, prefill):
    """A run with evictions keeps the invariants the paper states for the cache."""
    w = wl.WORKLOADS["tiny"].replace(T=420, S=S, W=W, M=128)
    q, k, v = wl.batch_tokens(w, 0, w.T)
    qg = w.q_g
    token_score = {}   # (b, h, token) -> accumulated score, tracked by token position

    def on_step(i, bounds, before, res):
        p, e = bounds
        s = e - p
        inc = res["score_inc"]
        # every query row's weights sum to 1 (§3.1.1): total = rows x query heads
        np.testing.assert_allclose(inc.sum(axis=-1), s, rtol=1e-12)
        _, pos_b, k_b, v_b = before
        for b in range(w.B):
            for h in range(w.Hkv):
                ev = set(res["evict_idx"][b, h].tolist())
                keep = np.array([j not in ev for j in range(w.M)])
                # only the S evicted slots change (§3.2 recurrence)
                np.testing.assert_array_equal(res["k_cache"][b, h][keep], k_b[b, h][keep])
                np.testing.assert_array_equal(res["v_cache"][b, h][keep], v_b[b, h][keep])
                np.testing.assert_array_equal(res["slot_pos"][b, h][keep], pos_b[b, h][keep])
                pos = res["slot_pos"][b, h]
                occ = pos[pos >= 0]
                assert len(np.unique(occ)) == len(occ)
                # the chunk's tokens and the recent window are resident (§3.3.1)
                assert set(range(max(0, e - max(W, s)), e)) <= set(occ.tolist())
                # cache consistency: slot j holds the K/V of token slot_pos[j]
                for j in np.nonzero(pos >= 0)[0]:
                    np.testing.assert_array_equal(res["k_cache"][b, h, j], k[b, h, pos[j]])
                    np.testing.assert_array_equal(res["v_cache"][b, h, j], v[b, h, pos[j]])
                # Eq. 3 bookkeeping by token: add this chunk's weights per token
                g = inc[b, h * qg:(h + 1) * qg].sum(axis=0)
                for j, t in enumerate(pos_b[b, h]):
                    if t >= 0:
                        token_score[(b, h, int(t))] = token_score.get((b, h, int(t)), 0.0) + g[j]
                for c in range(s):
                    token_score[(b, h, p + c)] = g[w.M + c]
                for j, t in enumerate(pos):
                    if t >= 0:
                        assert abs(res["scores"][b, h, j] - token_score[(b, h, int(t))]) < 1e-9

    run_sequence(q, k, v, w.M, w.S, w.W, prefill=prefill, on_step=on_step)


def test_lse_merge_matches_logsumexp():
    """§A.6.1 reduction: merging partial log-sum-exps equals the full one."""
    rng = np.random.default_rng(8)
    a = rng.standard_normal((5, 40)) * 6
    full = logsumexp(a, axis=1)
    for cut in (1, 13, 39):
        merged = lse_merge(logsumexp(a[:, :cut], axis=1), logsumexp(a[:, cut:], axis=1))
        np.testing.assert_allclose(merged, full, rtol=0, atol=1e-12)


def test_chunk_bounds():
    assert chunk_bounds(1024, 256, 32)[:2] == [(0, 256), (256, 288)]
    assert len(chunk_bounds(1024, 256, 32)) == 1 + 24
    assert chunk_bounds(10, 4, 4) == [(0, 4), (4, 8), (8, 10)]
    assert chunk_bounds(3, 8, 2) == [(0, 3)]


def test_row_subset_matches_full_chunk():
    rng = np.random.default_rng(9)
    B, Hq, Hkv, M, S, d, pos0 = 1, 4, 2, 20, 9, 8, 50
    st = _state(rng, B, Hkv, M, d, pos0, n_empty=2)
    q, kn, vn = _rand_seq(rng, B, Hq, Hkv, S, d)
    out, inc, lse = sdpa_chunk(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], pos0)
    rows = [0, 3, 8]
    o2, inc2, l2 = sdpa_chunk(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], pos0,
                              rows=rows)
    np.testing.assert_allclose(o2, out[:, :, rows], atol=1e-14)
    np.testing.assert_allclose(l2, lse[:, :, rows], atol=1e-14)
    np.testing.assert_allclose(inc2.sum(axis=-1), len(rows), rtol=1e-12)


# ------------------------------------------------- policy variants (§3.1.1) --
def _brute_force_evict_keyed(key_of, pos, pos0, S, W):
    """S-subset of candidates with the smallest key sum (empty slot = -1; keys are
    exact fractions), ties by the lexicographically smallest subset."""
    cand = [j for j in range(len(pos)) if pos[j] < pos0 + S - W]
    key = {j: (Fraction(-1) if pos[j] < 0 else key_of(j)) for j in cand}
    best = None
    for sub in itertools.combinations(cand, S):
        s = sum(key[j] for j in sub)
        if best is None or (s, sub) < best:
            best = (s, sub)
    return list(best[1])


def _policy_case(seed, B=1):
    rng = np.random.default_rng(500 + seed)
    M = int(rng.integers(2, 9))
    S = int(rng.integers(1, M + 1))
    W = int(rng.integers(0, S + 2)) if rng.random() < 0.7 else 0
    if M - max(0, W - S) < S:
        W = S
    qg, d, pos0 = 2, 4, 50
    n_empty = int(rng.integers(0, M + 1)) if rng.random() < 0.4 else 0
    st = _state(rng, B, 1, M, d, pos0, n_empty=n_empty, int_scores=True)
    for r in range(max(0, W - S)):
        st["slot_pos"][:, 0, r] = pos0 - 1 - r
    st["slot_pos"][1:] = st["slot_pos"][0]        # one set of positions for the batch
    st["scores"][st["slot_pos"] < 0] = 0
    inc = rng.integers(0, 3, size=(B, qg, M + S)).astype(np.float32)
    for b in range(B):
        inc[b, :, :M][:, st["slot_pos"][b, 0] < 0] = 0
    _, kn, vn = _rand_seq(rng, B, qg, 1, S, d)
    return st, inc, kn, vn, M, S, W, pos0


@pytest.mark.parametrize("precision", ["fp32", "fp64"])
@pytest.mark.parametrize("seed", range(30))
def test_norm_policy_matches_brute_force(seed, precision):
    """h2o_norm ranks occupied slots by score / (t - t(j)), t = P + S (§3.1.1)."""
    st, inc, kn, vn, M, S, W, pos0 = _policy_case(seed)
    res = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                 pos0, W, precision, "h2o_norm")
    acc = st["scores"][0, 0] + inc[0].sum(axis=0)[:M]
    pos = st["slot_pos"][0, 0]
    expect = _brute_force_evict_keyed(
        lambda j: Fraction(int(acc[j])) / (pos0 + S - int(pos[j])), pos, pos0, S, W)
    assert list(res["evict_idx"][0, 0]) == expect
    # stored scores stay unnormalized: Eq. 3 for kept slots, own column for new ones
    kept = np.setdiff1d(np.arange(M), expect)
    np.testing.assert_array_equal(res["scores"][0, 0, kept], acc[kept])
    for c, e in enumerate(expect):
        assert res["slot_pos"][0, 0, e] == pos0 + c
        assert res["scores"][0, 0, e] == inc[0, :, M + c].sum()


def test_norm_policy_evicts_the_older_of_two_equal_scores():
    rng = np.random.default_rng(9)
    M, S, W, pos0, d = 3, 1, 0, 100, 4
    st = _state(rng, 1, 1, M, d, pos0)
    st["slot_pos"][0, 0] = [90, 10, 95]        # ages 11, 91, 6 at t = 101
    st["scores"][0, 0] = [4.0, 4.0, 1.0]       # normalized: 0.364, 0.044, 0.167
    inc = np.zeros((1, 1, M + S), np.float32)
    _, kn, vn = _rand_seq(rng, 1, 1, 1, S, d)
    r_h2o = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                   pos0, W, "fp32", "h2o")
    r_norm = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                    pos0, W, "fp32", "h2o_norm")
    assert list(r_h2o["evict_idx"][0, 0]) == [2]       # smallest raw score
    assert list(r_norm["evict_idx"][0, 0]) == [1]      # long-resident, rarely used


@pytest.mark.parametrize("seed", range(20))
def test_orig_policy_for_one_batch_entry_is_h2o(seed):
    st, inc, kn, vn, M, S, W, pos0 = _policy_case(seed)
    a = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
               pos0, W, "fp32", "h2o")
    b = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
               pos0, W, "fp32", "h2o_orig")
    for key in a:
        np.testing.assert_array_equal(a[key], b[key])


@pytest.mark.parametrize("seed", range(30))
def test_orig_policy_matches_brute_force(seed):
    """h2o_orig: one selection per KV head from the scores summed over b."""
    B = 2 + seed % 2
    st, inc, kn, vn, M, S, W, pos0 = _policy_case(seed, B=B)
    res = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                 pos0, W, "fp32", "h2o_orig")
    acc = st["scores"][:, 0] + inc.sum(axis=1)[:, :M]          # (B, M), small integers
    tot = acc.sum(axis=0)
    expect = _brute_force_evict_keyed(lambda j: Fraction(int(tot[j])), st["slot_pos"][0, 0],
                                      pos0, S, W)
    for b in range(B):
        assert list(res["evict_idx"][b, 0]) == expect
        for c, e in enumerate(expect):
            assert res["slot_pos"][b, 0, e] == pos0 + c
            np.testing.assert_array_equal(res["k_cache"][b, 0, e], kn[b, 0, c])
            assert res["scores"][b, 0, e] == inc[b, :, M + c].sum()
    np.testing.assert_array_equal(res["slot_pos"][0], res["slot_pos"][-1])


@pytest.mark.parametrize("policy", ["h2o_norm", "h2o_orig"])
def test_run_invariants_for_policies(policy):
    """Whole runs with the variants keep the cache invariants (and h2o_orig keeps one
    set of positions across the batch)."""
    w = wl.WORKLOADS["tiny"].replace(T=360, S=24, W=16, M=96, B=2)
    q, k, v = wl.batch_tokens(w, 0, w.T)
    steps = []
    out, st = run_sequence(q, k, v, w.M, w.S, w.W, precision="fp32", policy=policy,
                           on_step=lambda i, pe, before, res: steps.append((pe, res)))
    for (p, e), res in steps[1:]:
        pos = res["slot_pos"]
        assert (pos < e).all() and (pos >= 0).all()
        for b in range(w.B):
            for h in range(w.Hkv):
                assert len(set(pos[b, h].tolist())) == w.M          # no token twice
                assert set(range(e - w.W, e)) <= set(pos[b, h].tolist())  # recent window
        if policy == "h2o_orig":
            assert (pos == pos[0:1]).all()
    assert np.isfinite(out).all()
