"""Pins of the 8-bit K/V oracle (oracle/quant.py) against values fixed by its
definition and by arithmetic, not by re-running its own formulas: hand rows
with known codes, the nearest-code property checked by brute force, the
round-trip bound, sign symmetry, exact round trips when the scale is a power
of two, a library bf16 rounding, and the reductions of the q8 SDPA / update
steps to the pinned bf16 oracle."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_19920_gb300 import workloads as wl


def test_hand_row_codes():
    # max |x| = 127, so s = 1 and each code is x rounded half to even
    x = np.zeros(8, np.float32)
    x[:7] = [127.0, -63.5, 1.0, 0.5, -0.5, 1.5, 2.5]
    codes, s = oracle.quantize_rows(x[None])
    assert s[0] == np.float32(1.0)
    assert codes[0].tolist() == [127, -64, 1, 0, 0, 2, 2, 0]


def test_hand_row_scaled():
    # max |x| = 254 -> s = 2; 3.0 / 2 = 1.5 -> 2 (even), 5.0 / 2 = 2.5 -> 2, -7 / 2 = -3.5 -> -4
    x = np.array([[-254.0, 3.0, 5.0, -7.0]], np.float32)
    codes, s = oracle.quantize_rows(x)
    assert s[0] == np.float32(2.0)
    assert codes[0].tolist() == [-127, 2, 2, -4]
    assert oracle.dequantize_rows(codes, s)[0].tolist() == [-254.0, 4.0, 4.0, -8.0]


def test_zero_row():
    codes, s = oracle.quantize_rows(np.zeros((2, 16), np.float32))
    assert (s == 0).all() and (codes == 0).all()
    assert (oracle.dequantize_rows(codes, s) == 0).all()


def test_nearest_code_by_brute_force():
    rng = np.random.default_rng(3)
    x = wl.round_bf16(rng.standard_normal((6, 16), dtype=np.float32) * 3)
    codes, s = oracle.quantize_rows(x)
    grid = np.arange(-127, 128)
    for r in range(x.shape[0]):
        for e in range(x.shape[1]):
            t = np.float32(x[r, e]) / s[r]  # the float32 ratio both sides compute
            dist = np.abs(grid - np.float64(t))
            best = grid[dist == dist.min()]
            want = best[best % 2 == 0][0] if len(best) > 1 else best[0]
            assert codes[r, e] == want


def test_round_trip_bound_and_extremes():
    rng = np.random.default_rng(4)
    x = wl.round_bf16(rng.standard_normal((50, 128), dtype=np.float32))
    codes, s = oracle.quantize_rows(x)
    err = np.abs(x.astype(np.float64) - codes.astype(np.float64) * s[:, None].astype(np.float64))
    # |x/s - c| <= 1/2 plus the float32 rounding of the ratio x / s (|ratio| <= 127:
    # half an ulp is at most 2^-18), which may turn a near-tie into a tie
    assert (err <= s[:, None] * (0.5 + 2.0 ** -17)).all()
    amax_idx = np.abs(x).argmax(axis=1)
    assert (np.abs(codes[np.arange(50), amax_idx]) == 127).all()
    assert np.abs(codes).max() <= 127


def test_sign_symmetry():
    rng = np.random.default_rng(5)
    x = wl.round_bf16(rng.standard_normal((20, 64), dtype=np.float32))
    c1, s1 = oracle.quantize_rows(x)
    c2, s2 = oracle.quantize_rows(-x)
    assert np.array_equal(s1, s2) and np.array_equal(c1, -c2)


def test_round_to_bf16_matches_torch():
    rng = np.random.default_rng(6)
    x = (rng.standard_normal(10000) * np.exp(rng.uniform(-20, 20, 10000))).astype(np.float32)
    x = np.concatenate([x, np.float32([1 + 2 ** -8, 1 + 3 * 2 ** -8, -(1 + 2 ** -8), 0.0])])
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    assert np.array_equal(oracle.round_to_bf16(x), ref)
    # ties to even by hand: 1 + 2^-8 -> 1, 1 + 3 * 2^-8 -> 1 + 2^-6
    assert oracle.round_to_bf16(np.float32([1 + 2 ** -8]))[0] == 1.0
    assert oracle.round_to_bf16(np.float32([1 + 3 * 2 ** -8]))[0] == np.float32(1 + 2 ** -6)


def _exact_rows(rng, shape, k):
    """Rows c * 2^k with integer c in [-127, 127] and one |c| = 127 per row:
    their scale is exactly 2^k and they round-trip exactly."""
    c = rng.integers(-127, 128, size=shape)
    c[..., 0] = 127 * np.where(rng.random(shape[:-1]) < 0.5, 1, -1)
    return (c * 2.0 ** k).astype(np.float32), c.astype(np.int8)


def test_power_of_two_scales_round_trip_exactly():
    rng = np.random.default_rng(7)
    x, c = _exact_rows(rng, (30, 64), -9)
    codes, s = oracle.quantize_rows(x)
    assert (s == np.float32(2.0 ** -9)).all()
    assert np.array_equal(codes, c)
    assert np.array_equal(oracle.dequantize_rows(codes, s), x)


def test_sdpa_cache_q8_reduces_to_bf16_oracle_on_exact_rows():
    rng = np.random.default_rng(8)
    B, Hq, Hkv, S, M, d, pos0 = 1, 4, 2, 5, 24, 16, 40
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=2)
    k, _ = _exact_rows(rng, (B, Hkv, M, d), -6)
    v, _ = _exact_rows(rng, (B, Hkv, M, d), -7)
    sp = st["slot_pos"]
    sp[0, :, :S] = pos0 + np.arange(S)  # the chunk's tokens are in the cache
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kc, ks = oracle.quantize_rows(k)
    vc, vs = oracle.quantize_rows(v)
    out8, inc8, _ = oracle.sdpa_cache_q8(q, kc, ks, vc, vs, sp, pos0)
    out, inc, _ = oracle.sdpa_cache(q, k, v, sp, pos0)
    assert np.array_equal(out8, out) and np.array_equal(inc8, inc)


def test_sdpa_chunk_q8_reduces_to_bf16_oracle_on_exact_rows():
    rng = np.random.default_rng(9)
    B, Hq, Hkv, S, M, d, pos0 = 2, 2, 1, 4, 12, 16, 30
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=1)
    k, _ = _exact_rows(rng, (B, Hkv, M, d), -5)
    v, _ = _exact_rows(rng, (B, Hkv, M, d), -5)
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    kc, ks = oracle.quantize_rows(k)
    vc, vs = oracle.quantize_rows(v)
    out8, inc8, _ = oracle.sdpa_chunk_q8(q, kc, ks, vc, vs, kn, vn, st["slot_pos"], pos0)
    out, inc, _ = oracle.sdpa_chunk(q, k, v, kn, vn, st["slot_pos"], pos0)
    assert np.array_equal(out8, out) and np.array_equal(inc8, inc)


@pytest.mark.parametrize("policy", ["h2o", "h2o_norm", "h2o_orig"])
def test_evict_insert_q8_selects_like_bf16_and_quantises_the_written_rows(policy):
    rng = np.random.default_rng(10)
    B, Hkv, S, M, d, pos0, W = 2, 2, 3, 16, 16, 50, 4
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=1)
    if policy == "h2o_orig":
        st["slot_pos"][1] = st["slot_pos"][0]
    kc, ks = oracle.quantize_rows(st["k_cache"])
    vc, vs = oracle.quantize_rows(st["v_cache"])
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    r8 = oracle.evict_insert_q8(st["scores"], st["slot_pos"], kn, vn, kc, ks, vc, vs, pos0, W,
                                policy=policy)
    r = oracle.evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                            pos0, W, policy=policy)
    for key in ("scores", "slot_pos", "evict_idx"):
        assert np.array_equal(r8[key], r[key])
    written = np.zeros((B, Hkv, M), bool)
    for b in range(B):
        for h in range(Hkv):
            for c, e in enumerate(r["evict_idx"][b, h]):
                written[b, h, e] = True
                for nm, new in (("k", kn), ("v", vn)):
                    codes, s = r8[nm + "_codes"][b, h, e], r8[nm + "_scales"][b, h, e]
                    assert np.abs(codes.astype(np.float64) * s - new[b, h, c]).max() <= s * (0.5 + 2.0 ** -17)
                    assert s == np.abs(new[b, h, c]).max() / np.float32(127)
    assert np.array_equal(r8["k_codes"][~written], kc[~written])
    assert np.array_equal(r8["v_scales"][~written], vs[~written])


def test_update_q8_selects_like_bf16():
    rng = np.random.default_rng(11)
    B, Hq, Hkv, S, M, d, pos0, W = 1, 4, 2, 3, 16, 16, 50, 4
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0)
    inc = rng.random((B, Hq, M + S)).astype(np.float32)
    kc, ks = oracle.quantize_rows(st["k_cache"])
    vc, vs = oracle.quantize_rows(st["v_cache"])
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    r8 = oracle.update_q8(st["scores"], st["slot_pos"], inc, kn, vn, kc, ks, vc, vs, pos0, W)
    r = oracle.update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                      pos0, W)
    for key in ("scores", "slot_pos", "evict_idx"):
        assert np.array_equal(r8[key], r[key])
    qk, sk = oracle.quantize_rows(kn)
    for c, e in enumerate(r["evict_idx"][0, 1]):
        assert np.array_equal(r8["k_codes"][0, 1, e], qk[0, 1, c]) and r8["k_scales"][0, 1, e] == sk[0, 1, c]
