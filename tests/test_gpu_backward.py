"""GPU parity of the chunk-SDPA gradient (h2o_sdpa_chunk_backward) against the
float64 oracle, through the C ABI.

Tolerance (derived from the arithmetic): the kernel rounds P and dS to bf16
(relative 2^-9 each) before the fp32-accumulated contractions, and uses the
bf16 forward output in D = dout . out; each gradient tensor must lie within
1e-2 of its own max-abs value elementwise.  Slots no row sees get exactly 0.

The cases cover both head sizes, 128-row tiles that hold the rows of two
query heads (q_g S not a multiple of 128), ragged key tiles, empty and
future slots, a one-token chunk, no cache, and the Llama-3-8B-shaped chunk."""
import numpy as np
import pytest
import torch

from oracle import sdpa_chunk_backward as ref_backward
from oracle import sdpa_chunk as ref_sdpa
from paper_2608_19920_gb300 import (build, h2o_device_errors, h2o_sdpa_chunk,
                                   h2o_sdpa_chunk_backward, h2o_sdpa_chunk_lse)
from paper_2608_19920_gb300 import workloads as wl

from test_gpu_parity import bf, f32

pytestmark = pytest.mark.gpu

GRAD_RTOL = 1e-2


@pytest.fixture(scope="module")
def dev():
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


CASES = [
    # B, Hq, Hkv, d, S, M, n_empty, n_future, pos0
    (1, 4, 2, 64, 32, 256, 0, 0, 256),       # the tiny workload's chunk shape
    (2, 8, 2, 128, 20, 300, 17, 5, 900),     # ragged S and M, empty and future slots
    (3, 6, 3, 64, 1, 130, 5, 0, 140),        # one token
    (1, 4, 2, 64, 6, 130, 3, 2, 150),        # N_k a multiple of 4, M not: the scalar passes
    (1, 2, 1, 64, 8, 4100, 20, 3, 4200),     # N_k > 4096: the softmax pass reads each row twice
    (1, 4, 4, 128, 200, 0, 0, 0, 0),         # no cache (a prefill)
    (1, 32, 8, 128, 512, 4096, 0, 0, 8192),  # the Llama-3-8B-shaped chunk
    (2, 8, 2, 128, 300, 700, 11, 20, 3000),  # row tiles across head boundaries, masked tiles
    (1, 4, 1, 64, 520, 130, 0, 40, 600),     # d = 64, several chunk tiles
    (1, 6, 2, 128, 45, 260, 9, 7, 400),      # q_g S = 135: a second row tile of 7 rows
]


# lse: log-sum-exp of fp32 logits of exact bf16 products (hardware exp2 / log2)
LSE_ATOL = 2e-3


@pytest.mark.parametrize("mode", ["recompute", "saved_lse"])
@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c)))
def test_backward_matches_oracle(dev, case, mode):
    B, Hq, Hkv, d, S, M, n_empty, n_future, pos0 = case
    rng = np.random.default_rng(hash(case) % 2**32)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty)
    for b in range(B):
        for h in range(Hkv):
            occ = np.nonzero(st["slot_pos"][b, h] >= 0)[0]
            for k in range(min(n_future, len(occ))):
                st["slot_pos"][b, h, occ[k]] = pos0 + (k % S)
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    dout = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    g = dict(q=bf(q, dev), kc=bf(st["k_cache"], dev), vc=bf(st["v_cache"], dev), kn=bf(kn, dev),
             vn=bf(vn, dev), sp=torch.from_numpy(st["slot_pos"]).to(dev))
    lse = None
    if mode == "recompute":
        out, _ = h2o_sdpa_chunk(g["q"], g["kc"], g["vc"], g["kn"], g["vn"], g["sp"], pos0)
    else:
        out, _, lse = h2o_sdpa_chunk_lse(g["q"], g["kc"], g["vc"], g["kn"], g["vn"], g["sp"], pos0)
    grads = h2o_sdpa_chunk_backward(g["q"], g["kc"], g["vc"], g["kn"], g["vn"], g["sp"], pos0, out,
                                    bf(dout, dev), lse=lse)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    refs = ref_backward(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], pos0, dout)
    for name, gpu, ref in zip(("dq", "dk_cache", "dv_cache", "dk_new", "dv_new"), grads, refs):
        if ref.size == 0:
            continue
        x = gpu.cpu().numpy().astype(np.float64)
        scale = np.abs(ref).max()
        err = np.abs(x - ref).max()
        assert err <= GRAD_RTOL * scale + 1e-6, f"{name}: max err {err:.3e} vs max {scale:.3e}"
    if M:
        hidden = (st["slot_pos"] < 0) | (st["slot_pos"] > pos0 + S - 1)
        assert (grads[1].cpu().numpy()[hidden] == 0).all()
        assert (grads[2].cpu().numpy()[hidden] == 0).all()


def test_backward_is_deterministic(dev):
    """No atomics: two calls on the same inputs give bit-identical gradients."""
    B, Hq, Hkv, d, S, M, pos0 = 1, 32, 8, 128, 512, 4096, 8192
    rng = np.random.default_rng(5)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=0)
    mk = lambda shape: bf(wl.round_bf16(rng.standard_normal(shape, dtype=np.float32)), dev)
    q, kn, vn, dout = mk((B, Hq, S, d)), mk((B, Hkv, S, d)), mk((B, Hkv, S, d)), mk((B, Hq, S, d))
    kc, vc = bf(st["k_cache"], dev), bf(st["v_cache"], dev)
    sp = torch.from_numpy(st["slot_pos"]).to(dev)
    out, _ = h2o_sdpa_chunk(q, kc, vc, kn, vn, sp, pos0)
    g1 = h2o_sdpa_chunk_backward(q, kc, vc, kn, vn, sp, pos0, out, dout)
    g2 = h2o_sdpa_chunk_backward(q, kc, vc, kn, vn, sp, pos0, out, dout)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    for a, b in zip(g1, g2):
        assert torch.equal(a, b)


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c)))
def test_forward_lse_matches_oracle(dev, case):
    """h2o_sdpa_chunk_lse: the same out and score_inc as h2o_sdpa_chunk (the
    same kernel when S > 1), and each row's log-sum-exp within LSE_ATOL of the
    oracle's (every row sees at least its own token, so lse is finite)."""
    B, Hq, Hkv, d, S, M, n_empty, n_future, pos0 = case
    rng = np.random.default_rng(hash(case) % 2**32 + 1)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty)
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    args = (bf(q, dev), bf(st["k_cache"], dev), bf(st["v_cache"], dev), bf(kn, dev), bf(vn, dev),
            torch.from_numpy(st["slot_pos"]).to(dev), pos0)
    out, inc, lse = h2o_sdpa_chunk_lse(*args)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    if S > 1:
        out0, inc0 = h2o_sdpa_chunk(*args)
        torch.cuda.synchronize()
        assert torch.equal(out, out0) and torch.equal(inc, inc0)
    _, _, lse_ref = ref_sdpa(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"], pos0)
    err = np.abs(lse.cpu().numpy().astype(np.float64) - lse_ref).max()
    assert err <= LSE_ATOL, f"lse max abs err {err:.3e}"
