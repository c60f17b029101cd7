"""The seeded input generator: deterministic, block-independent, bf16-exact."""
import numpy as np
import torch

from paper_2608_19920_gb300 import workloads as wl


def test_round_bf16_matches_torch():
    x = np.random.default_rng(0).standard_normal(100000).astype(np.float32) * 37
    x[:4] = [0.0, -0.0, 1e-40, 3.3895314e38]
    ref = torch.from_numpy(x).to(torch.bfloat16).float().numpy()
    np.testing.assert_array_equal(wl.round_bf16(x), ref)
    np.testing.assert_array_equal(wl.bits_to_f32(wl.bf16_bits(ref)), ref)


def test_token_ranges_are_independent_of_how_they_are_cut():
    w = wl.WORKLOADS["tiny"]
    q, k, v = wl.tokens(w, 0, 0, 700)
    for a, b in [(0, 1), (255, 257), (300, 700), (511, 512)]:
        qa, ka, va = wl.tokens(w, 0, a, b)
        np.testing.assert_array_equal(qa, q[:, a:b])
        np.testing.assert_array_equal(ka, k[:, a:b])
        np.testing.assert_array_equal(va, v[:, a:b])


def test_values_are_bf16_and_heavy_keys_are_shifted():
    w = wl.WORKLOADS["batched_16k"]
    for b in range(w.B):
        heavy = wl.heavy_positions(w, b)
        lo, hi = w.n_sink
        assert lo <= len(heavy) <= hi and (heavy == np.arange(len(heavy))).all()
        assert 1.0 <= wl.key_shift(w, b) <= 3.0
    q, k, v = wl.tokens(w, 1, 0, 64)
    for x in (q, k, v):
        np.testing.assert_array_equal(wl.round_bf16(x), x)
    w2 = wl.WORKLOADS["llama8b_32k"]
    assert len(wl.heavy_positions(w2, 0)) >= 8 + int(0.01 * w2.T) - 8


def test_sequences_differ_per_batch_entry():
    w = wl.WORKLOADS["batched_16k"]
    qa, _, _ = wl.tokens(w, 0, 0, 8)
    qb, _, _ = wl.tokens(w, 1, 0, 8)
    assert not np.array_equal(qa, qb)
