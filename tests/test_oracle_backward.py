"""Pins of the chunk-SDPA gradient oracle (§3.1 Eq. 2, mask of §3.3.1).

The gradient oracle (float64 autograd) is checked against central finite
differences of the independently pinned NumPy forward ``sdpa_chunk``, against
torch's dense causal SDPA backward when the cache holds the whole prefix in
order, and against the zero gradient of every key no row can see.
"""
import math

import numpy as np
import pytest
import torch

from oracle import sdpa_chunk, sdpa_chunk_backward
from paper_2608_19920_gb300 import workloads as wl


def _case(seed, B=1, Hq=4, Hkv=2, S=3, M=6, d=5, pos0=20, n_empty=1, n_future=1):
    rng = np.random.default_rng(seed)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty)
    for b in range(B):
        for h in range(Hkv):
            occ = np.nonzero(st["slot_pos"][b, h] >= 0)[0]
            st["slot_pos"][b, h, occ[:n_future]] = pos0 + 1  # visible from row 1 on
    q = rng.standard_normal((B, Hq, S, d))
    kn = rng.standard_normal((B, Hkv, S, d))
    vn = rng.standard_normal((B, Hkv, S, d))
    dout = rng.standard_normal((B, Hq, S, d))
    return st, q, kn, vn, dout


@pytest.mark.parametrize("seed", range(4))
def test_gradient_matches_finite_differences(seed):
    st, q, kn, vn, dout = _case(seed)
    pos0 = 20
    args = [q, st["k_cache"].astype(np.float64), st["v_cache"].astype(np.float64), kn, vn]
    grads = sdpa_chunk_backward(*args, st["slot_pos"], pos0, dout)

    def loss(xs):
        out, _, _ = sdpa_chunk(xs[0], xs[1], xs[2], xs[3], xs[4], st["slot_pos"], pos0)
        return float((out * dout).sum())

    rng = np.random.default_rng(100 + seed)
    eps = 1e-6
    for which in range(5):
        u = rng.standard_normal(args[which].shape)
        plus = [a.copy() for a in args]
        minus = [a.copy() for a in args]
        plus[which] = plus[which] + eps * u
        minus[which] = minus[which] - eps * u
        fd = (loss(plus) - loss(minus)) / (2 * eps)
        an = float((grads[which] * u).sum())
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (which, fd, an)


def test_hidden_and_empty_slots_get_no_gradient():
    st, q, kn, vn, dout = _case(7, M=9, n_empty=2, n_future=0)
    pos0 = 20
    st["slot_pos"][0, 0, 3] = pos0 + 10   # after every row of the chunk
    _, dkc, dvc, _, _ = sdpa_chunk_backward(q, st["k_cache"], st["v_cache"], kn, vn,
                                            st["slot_pos"], pos0, dout)
    hidden = (st["slot_pos"] < 0) | (st["slot_pos"] > pos0 + q.shape[2] - 1)
    assert hidden.sum() >= 3
    assert (dkc[hidden] == 0).all() and (dvc[hidden] == 0).all()


def test_prefix_cache_equals_dense_causal_backward():
    """Cache slots hold tokens 0..P-1 in order: the chunk's gradient is the dense
    causal attention gradient with zero output gradient on the first P rows."""
    rng = np.random.default_rng(9)
    B, Hq, Hkv, T, d, P = 1, 4, 2, 11, 6, 7
    q = rng.standard_normal((B, Hq, T, d))
    k = rng.standard_normal((B, Hkv, T, d))
    v = rng.standard_normal((B, Hkv, T, d))
    dout = rng.standard_normal((B, Hq, T, d))
    dout[:, :, :P] = 0
    slot_pos = np.broadcast_to(np.arange(P, dtype=np.int32), (B, Hkv, P)).copy()
    dq, dkc, dvc, dkn, dvn = sdpa_chunk_backward(q[:, :, P:], k[:, :, :P], v[:, :, :P],
                                                 k[:, :, P:], v[:, :, P:], slot_pos, P,
                                                 dout[:, :, P:])
    qg = Hq // Hkv
    tq, tk, tv = (torch.tensor(x, requires_grad=True) for x in (q, k, v))
    out = torch.nn.functional.scaled_dot_product_attention(
        tq, tk.repeat_interleave(qg, 1), tv.repeat_interleave(qg, 1), is_causal=True)
    (out * torch.tensor(dout)).sum().backward()
    np.testing.assert_allclose(dq, tq.grad.numpy()[:, :, P:], rtol=0, atol=1e-12)
    np.testing.assert_allclose(dkc, tk.grad.numpy()[:, :, :P], rtol=0, atol=1e-12)
    np.testing.assert_allclose(dkn, tk.grad.numpy()[:, :, P:], rtol=0, atol=1e-12)
    np.testing.assert_allclose(dvc, tv.grad.numpy()[:, :, :P], rtol=0, atol=1e-12)
    np.testing.assert_allclose(dvn, tv.grad.numpy()[:, :, P:], rtol=0, atol=1e-12)
