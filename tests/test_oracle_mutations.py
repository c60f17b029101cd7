"""Planted mistakes in the oracle must fail its pins.

Each case builds a copy of an oracle module from its source with one plausible
mistake planted (a mask off by one, a wrong GQA mapping, a dropped term, a
reversed tie-break, ...), runs compact versions of the pins against it, and
requires at least one of them to fail; the untouched oracle must pass all.
Everything runs on the CPU; the product path is not involved.
"""
import itertools
import math
import os
import types

import numpy as np
import pytest
import torch

from paper_2608_19920_gb300 import workloads as wl

ORACLE = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle")


def _load(fname, mutation=None):
    """The oracle module `fname` as source, with the n-th occurrence of `old`
    replaced by `new` when a mutation (old, new, n) is given."""
    with open(os.path.join(ORACLE, fname)) as f:
        src = f.read()
    if mutation is not None:
        old, new, n = mutation
        pos = -1
        for _ in range(n + 1):
            pos = src.index(old, pos + 1)
        src = src[:pos] + new + src[pos + len(old):]
    mod = types.ModuleType("oracle_variant_" + fname.replace(".", "_"))
    mod.__package__ = "oracle"  # relative imports resolve to the untouched oracle
    exec(compile(src, fname, "exec"), mod.__dict__)
    return mod


def _rand_seq(rng, B, Hq, Hkv, T, d):
    q = wl.round_bf16(rng.standard_normal((B, Hq, T, d), dtype=np.float32))
    k = wl.round_bf16(rng.standard_normal((B, Hkv, T, d), dtype=np.float32))
    v = wl.round_bf16(rng.standard_normal((B, Hkv, T, d), dtype=np.float32))
    return q, k, v


def _dense(q, k, v):
    qg = q.shape[1] // k.shape[1]
    qt = torch.from_numpy(np.asarray(q, np.float64))
    kt = torch.from_numpy(np.asarray(k, np.float64)).repeat_interleave(qg, dim=1)
    vt = torch.from_numpy(np.asarray(v, np.float64)).repeat_interleave(qg, dim=1)
    T = q.shape[2]
    causal = torch.ones(T, T, dtype=torch.bool).tril()
    w = torch.softmax(((qt @ kt.transpose(-1, -2)) / math.sqrt(q.shape[-1]))
                      .masked_fill(~causal, float("-inf")), dim=-1)
    return (w @ vt).numpy(), w.numpy()


# ------------------------------------------------------------- pin checks --
# Each returns True when the module passes that pin.

def pin_dense(mod, order="chunk"):
    """No eviction (M >= T): dense causal attention, and scores = dense column sums."""
    rng = np.random.default_rng(1)
    B, Hq, Hkv, T, d = 1, 4, 2, 23, 8
    q, k, v = _rand_seq(rng, B, Hq, Hkv, T, d)
    out, st = mod.run_sequence(q, k, v, M=32, S=5, W=0, prefill=7, order=order)
    ref, w = _dense(q, k, v)
    if not np.allclose(out, ref, rtol=0, atol=1e-10):
        return False
    qg = Hq // Hkv
    for h in range(Hkv):
        for j in range(T):
            if abs(st.scores[0, h, j] - w[0, h * qg:(h + 1) * qg, :, j].sum()) > 1e-10:
                return False
    return True


def pin_rowsum(mod):
    rng = np.random.default_rng(2)
    st = wl.random_state(rng, 2, 2, 40, 8, pos0=100, n_empty=3)
    q, kn, vn = _rand_seq(rng, 2, 4, 2, 6, 8)
    _, inc, _ = mod.sdpa_chunk(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], 100)
    return np.allclose(inc.sum(-1), 6, rtol=1e-12)


def _brute(key, pos, pos0, S, W):
    cand = [j for j in range(len(pos)) if pos[j] < pos0 + S - W]
    val = {j: (-1 if pos[j] < 0 else key[j]) for j in cand}
    best = None
    for sub in itertools.combinations(cand, S):
        s = sum(val[j] for j in sub)
        if best is None or (s, sub) < best:
            best = (s, sub)
    return list(best[1])


def pin_update_brute(mod):
    """Eviction = brute-force minimal subset; the new tokens' scores are their
    own columns' sums; slots take tokens in order."""
    for seed in range(12):
        rng = np.random.default_rng(50 + seed)
        M, S, W, pos0, qg = 7, int(rng.integers(1, 4)), 2, 40, 2
        st = wl.random_state(rng, 1, 1, M, 4, pos0=pos0, n_empty=int(seed % 3 == 0),
                             int_scores=True)
        st["slot_pos"][0, 0, 0] = pos0 - 1  # a recent token inside the window
        inc = rng.integers(0, 3, size=(1, qg, M + S)).astype(np.float32)
        _, kn, vn = _rand_seq(rng, 1, qg, 1, S, 4)
        res = mod.update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                         pos0, W, "fp32")
        acc = st["scores"][0, 0] + inc[0].sum(0)[:M]
        expect = _brute(acc, st["slot_pos"][0, 0], pos0, S, W)
        if list(res["evict_idx"][0, 0]) != expect:
            return False
        for c, e in enumerate(expect):
            if res["scores"][0, 0, e] != inc[0, :, M + c].sum() or res["slot_pos"][0, 0, e] != pos0 + c:
                return False
    return True


def pin_evict_insert(mod):
    for seed in range(8):
        rng = np.random.default_rng(80 + seed)
        M, S, pos0 = 7, 2, 40
        st = wl.random_state(rng, 1, 1, M, 4, pos0=pos0, int_scores=True)
        _, kn, vn = _rand_seq(rng, 1, 1, 1, S, 4)
        res = mod.evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                               pos0, 0, "fp32")
        expect = _brute(st["scores"][0, 0], st["slot_pos"][0, 0], pos0, S, 0)
        if list(res["evict_idx"][0, 0]) != expect or (res["scores"][0, 0, expect] != 0).any():
            return False
    return True


def pin_replay(mod):
    rng = np.random.default_rng(90)
    st = wl.random_state(rng, 1, 2, 12, 4, pos0=50)
    index = np.stack([rng.permutation(12)[:3] for _ in range(2)])[None].astype(np.int32)
    _, kn, vn = _rand_seq(rng, 1, 2, 2, 3, 4)
    res = mod.kv_replace(st["k_cache"], st["v_cache"], st["slot_pos"], index, kn, vn, 50)
    idx = torch.from_numpy(index.astype(np.int64))[..., None].expand(-1, -1, -1, 4)
    k = torch.from_numpy(st["k_cache"])
    ok = np.array_equal(res["delta_k"], torch.gather(k, 2, idx).numpy())
    ok &= np.array_equal(res["k_cache"], k.clone().scatter_(2, idx, torch.from_numpy(kn)).numpy())
    back = mod.kv_restore(res["k_cache"], res["v_cache"], res["slot_pos"], index, res["delta_k"],
                          res["delta_v"], res["delta_pos"])
    return ok and np.array_equal(back["v_cache"], st["v_cache"])


def pin_backward_fd(bmod, fmod):
    rng = np.random.default_rng(95)
    pos0 = 20
    st = wl.random_state(rng, 1, 1, 5, 4, pos0=pos0, n_empty=1)
    st["slot_pos"][0, 0, np.nonzero(st["slot_pos"][0, 0] >= 0)[0][0]] = pos0 + 1
    q, kn, vn, dout = (rng.standard_normal(s) for s in ((1, 2, 3, 4), (1, 1, 3, 4), (1, 1, 3, 4),
                                                        (1, 2, 3, 4)))
    args = [q, st["k_cache"].astype(np.float64), st["v_cache"].astype(np.float64), kn, vn]
    grads = bmod.sdpa_chunk_backward(*args, st["slot_pos"], pos0, dout)

    def loss(xs):
        out, _, _ = fmod.sdpa_chunk(*xs, st["slot_pos"], pos0)
        return float((out * dout).sum())

    for which in range(5):
        u = rng.standard_normal(args[which].shape)
        p = [a.copy() for a in args]
        m = [a.copy() for a in args]
        p[which] += 1e-6 * u
        m[which] -= 1e-6 * u
        fd = (loss(p) - loss(m)) / 2e-6
        if abs(fd - float((grads[which] * u).sum())) > 1e-5 * max(1.0, abs(fd)):
            return False
    return True


def pin_quant(q):
    """Hand rows with known codes (max 127 -> s = 1; max 254 -> s = 2), their
    read-back values, bf16 rounding against torch and by hand."""
    x = np.array([[127.0, -63.5, 1.0, 0.5, -0.5, 1.5, 2.5, 0.0]], np.float32)
    codes, s = q.quantize_rows(x)
    if s[0] != 1.0 or codes[0].tolist() != [127, -64, 1, 0, 0, 2, 2, 0]:
        return False
    codes, s = q.quantize_rows(np.array([[-254.0, 3.0, 5.0, -7.0]], np.float32))
    if s[0] != 2.0 or codes[0].tolist() != [-127, 2, 2, -4]:
        return False
    if q.dequantize_rows(codes, s)[0].tolist() != [-254.0, 4.0, 4.0, -8.0]:
        return False
    y = np.float32([1 + 2 ** -8, 1 + 3 * 2 ** -8, 3.14159, -2.71828e-3])
    return np.array_equal(q.round_to_bf16(y), torch.from_numpy(y).to(torch.bfloat16).float().numpy())


def pin_q8_write(q):
    """The slots evict_insert_q8 overwrites hold the chunk's own K (and V) rows,
    within half a step."""
    rng = np.random.default_rng(97)
    st = wl.random_state(rng, 1, 1, 8, 8, pos0=30)
    kc, ks = q.quantize_rows(st["k_cache"])
    vc, vs = q.quantize_rows(st["v_cache"])
    _, kn, vn = _rand_seq(rng, 1, 1, 1, 2, 8)
    res = q.evict_insert_q8(st["scores"], st["slot_pos"], kn, vn, kc, ks, vc, vs, 30, 0)
    for c, e in enumerate(res["evict_idx"][0, 0]):
        for codes, sc, new in ((res["k_codes"], res["k_scales"], kn), (res["v_codes"], res["v_scales"], vn)):
            if np.abs(codes[0, 0, e] * np.float64(sc[0, 0, e]) - new[0, 0, c]).max() > 0.51 * sc[0, 0, e]:
                return False
    return True


def _all_pins(mods):
    h, r, b = mods["h2o_oracle.py"], mods["replay.py"], mods["backward.py"]
    qm = mods["quant.py"]
    return {
        "dense": pin_dense(h),
        "dense_paper": pin_dense(h, "paper"),
        "rowsum": pin_rowsum(h),
        "update_brute": pin_update_brute(h),
        "evict_insert": pin_evict_insert(h),
        "replay": pin_replay(r),
        "backward_fd": pin_backward_fd(b, h),
        "quant": pin_quant(qm),
        "q8_write": pin_q8_write(qm),
    }


# (file, old text, planted text, occurrence): each a plausible mistake
MUTATIONS = {
    "mask_off_by_one": ("h2o_oracle.py", "(t[None, :] <= qpos)", "(t[None, :] < qpos)", 0),
    "gqa_mapping": ("h2o_oracle.py", "h = hq // qg", "h = hq % Hkv", 0),
    "missing_scale": ("h2o_oracle.py", "scale = 1.0 / math.sqrt(d)", "scale = 1.0", 0),
    "scaled_column_sums": ("h2o_oracle.py", "score_inc[b, hq] = m.sum(axis=0)",
                           "score_inc[b, hq] = 0.5 * m.sum(axis=0)", 0),
    "dropped_new_token_score": ("h2o_oracle.py", "out_scores[b, h, e] = new[b, h, c]",
                                "out_scores[b, h, e] = 0", 0),
    "reversed_tie_break": ("h2o_oracle.py", "order = np.lexsort((cand, rank1, rank0))",
                           "order = np.lexsort((-cand, rank1, rank0))", 0),
    "window_ignores_chunk": ("h2o_oracle.py", "cand = np.nonzero(pos < pos0 + S - W)[0]",
                             "cand = np.nonzero(pos < pos0 - W)[0]", 0),
    "unsorted_eviction_list": ("h2o_oracle.py", "return np.sort(cand[order[:S]])",
                               "return cand[order[:S]]", 0),
    "group_sum_drops_a_head": ("h2o_oracle.py", "for g in range(1, qg):", "for g in range(2, qg):",
                               0),
    "paper_mask_off_by_one": ("h2o_oracle.py", "(t[None, :] <= qpos)", "(t[None, :] < qpos)", 1),
    "paper_new_score_kept": ("h2o_oracle.py", "out_scores[b, h, e] = 0", "pass", 0),
    "paper_rank_reversed": ("h2o_oracle.py", "chosen = choose(out_scores[b, h], pos)",
                                   "chosen = choose(-out_scores[b, h], pos)", 0),
    "paper_scores_not_added": ("h2o_oracle.py", "out[b, h] = out[b, h] + t", "out[b, h] = t", 0),
    "delta_after_write": ("replay.py", "delta_k[b, h, c] = k_cache[b, h, e]",
                          "delta_k[b, h, c] = k_new[b, h, c]", 0),
    "restore_positions_only": ("replay.py", "out_v[b, h, e] = delta_v[b, h, c]", "pass", 0),
    "backward_without_mask": ("backward.py", 'a = a.masked_fill(~visible, float("-inf"))',
                              "a = a", 0),
    "backward_wrong_scale": ("backward.py", "scale = 1.0 / math.sqrt(d)", "scale = 1.0 / d", 0),
    "quant_scale_over_128": ("quant.py", "QMAX = 127", "QMAX = 128", 0),
    "quant_rounds_toward_zero": ("quant.py", "np.clip(np.rint(ratio)", "np.clip(np.trunc(ratio)", 0),
    "dequant_drops_scale": ("quant.py", " * np.asarray(scales, np.float32)[..., None]", "", 0),
    "bf16_truncates": ("quant.py", "r = ((u + 0x7FFF + lsb) >> 16) << 16", "r = (u >> 16) << 16", 0),
    "bf16_ties_away": ("quant.py", "u + 0x7FFF + lsb", "u + 0x8000", 0),
    "q8_write_swaps_k_and_v": ("quant.py", "kc[b, h, e], ks[b, h, e] = qk[b, h, c], sk[b, h, c]",
                               "kc[b, h, e], ks[b, h, e] = qv[b, h, c], sv[b, h, c]", 0),
}

FILES = ("h2o_oracle.py", "replay.py", "backward.py", "quant.py")


def test_untouched_oracle_passes_every_pin():
    mods = {f: _load(f) for f in FILES}
    assert all(_all_pins(mods).values()), _all_pins(mods)


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_fails_a_pin(name):
    fname, old, new, n = MUTATIONS[name]
    mods = {f: _load(f, (old, new, n) if f == fname else None) for f in FILES}
    try:
        results = _all_pins(mods)
    except Exception:  # the mistake breaks the oracle outright: caught as well
        return
    assert not all(results.values()), f"{name} passes every pin: {results}"
