"""GPU parity: the CUDA library (called through its C ABI) against the float64 oracle.

Tolerances (bf16 inputs, fp32 accumulation):
  * attention output: |gpu - ref| <= max(1e-2, ulp_bf16(gpu)/2 + (2^-9 + 2^-12) w)
    elementwise, with w = sum_j m_ij |v_j| (the oracle's output computed on
    |V|).  The flat 1e-2 is the stated bound and holds wherever the kernel's
    arithmetic allows it.  Two roundings can exceed it on rows dominated by a
    few large values: the weights m_ij are rounded to bf16 (relative error
    <= 2^-9) to feed the tensor-core P V product, which moves the output by up
    to 2^-9 w, and the fp32 result is rounded to bf16 once more for storage
    (<= half an ulp).  2^-12 w covers the fp32 accumulation, the hardware
    exp2 and the fp32 row normaliser.  An exact kernel would stay within
    ulp/2, below 1e-2 for |out| < 4;
  * summed weights score_inc: |gpu - ref| <= 1e-3 |ref| + 1e-7 elementwise;
  * eviction indices, slot positions, scores and cache bytes: bit-exact when the
    update is fed the same fp32 scores and score_inc as the oracle's fp32 mode.
"""
import numpy as np
import pytest
import torch

from oracle import sdpa_chunk as ref_sdpa
from oracle import update as ref_update
from paper_2608_19920_gb300 import (H2OLayer, build, h2o_device_errors, h2o_sdpa_chunk, h2o_update,
                                   h2o_update_policy)
from paper_2608_19920_gb300 import workloads as wl
from paper_2608_19920_gb300.runner import chunk_bounds

pytestmark = pytest.mark.gpu

OUT_ATOL = 1e-2
P_ROUND = 2.0 ** -9 + 2.0 ** -12  # bf16 rounding of the weights + fp32 / exp2 slack
INC_RTOL = 1e-3
INC_ATOL = 1e-7


@pytest.fixture(scope="module")
def dev():
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def bf(x, dev):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(dev)


def f32(t):
    return t.float().cpu().numpy()


def half_ulp_bf16(x):
    """Half the spacing of bf16 values around |x| (8 significant bits)."""
    ax = np.maximum(np.abs(x), 2.0 ** -126)
    return 0.5 * np.exp2(np.floor(np.log2(ax)) - 7)


def with_abs_values(fn, args, v_idx, **kw):
    """Runs an oracle SDPA function twice: as given, and with the value
    arguments at positions ``v_idx`` replaced by their absolute values.  The
    output is linear in V, so the second call's output is w = sum_j m_ij |v_j|.
    Returns (out, score_inc, w)."""
    out, inc, _ = fn(*args, **kw)
    a = list(args)
    for i in v_idx:
        a[i] = np.abs(np.asarray(a[i]))
    w, _, _ = fn(*a, **kw)
    return out, inc, w


def oracle_sdpa(q, kc, vc, kn, vn, sp, pos0, **kw):
    """The oracle's sdpa_chunk with the P-rounding weight w (see the module notes)."""
    return with_abs_values(ref_sdpa, (q, kc, vc, kn, vn, sp, pos0), (2, 4), **kw)


def check_out(out_gpu, out_ref, w_ref):
    o = f32(out_gpu) if torch.is_tensor(out_gpu) else out_gpu
    err = np.abs(o - out_ref)
    bound = np.maximum(OUT_ATOL, half_ulp_bf16(o) + P_ROUND * np.asarray(w_ref))
    bad = err > bound
    assert not bad.any(), (f"{bad.sum()} outputs out of tolerance: max abs err {err.max():.3e}, "
                           f"worst excess {(err - bound).max():.3e} at "
                           f"{np.argwhere(bad)[:3].tolist()}")
    return err.max()


def check_sdpa(out_gpu, inc_gpu, out_ref, inc_ref, w_ref):
    out_err = check_out(out_gpu, out_ref, w_ref)
    inc = inc_gpu.cpu().numpy().astype(np.float64)
    bad = np.abs(inc - inc_ref) > INC_RTOL * np.abs(inc_ref) + INC_ATOL
    big = np.abs(inc_ref) > 1e-4
    rel = (np.abs(inc - inc_ref)[big] / np.abs(inc_ref[big])).max() if big.any() else 0.0
    assert not bad.any(), (f"{bad.sum()} score_inc entries out of tolerance; max rel err on "
                           f"entries > 1e-4: {rel:.3e}; first at {np.argwhere(bad)[:3].tolist()}")
    return out_err, rel


SDPA_CASES = [
    # B, Hq, Hkv, d, S, M, n_empty, n_future, pos0
    (1, 4, 2, 64, 32, 256, 0, 0, 256),        # the tiny workload's chunk shape
    (2, 8, 2, 128, 20, 300, 17, 5, 900),      # ragged S < 32 (4 heads packed), ragged M, mask
    (1, 7, 1, 128, 200, 384, 0, 0, 1000),     # S > 128 with a ragged row tile, q_g = 7
    (1, 28, 4, 128, 96, 512, 3, 0, 5000),     # 96-row boxes, q_g = 7
    (3, 6, 3, 64, 1, 130, 5, 0, 140),         # decode step, S = 1
    (1, 4, 4, 128, 256, 0, 0, 0, 0),          # no cache: pure causal chunk
    (1, 8, 8, 64, 64, 128, 128, 0, 0),        # empty cache (prefill against empty slots)
    (2, 16, 4, 128, 130, 1000, 40, 30, 2000), # mixed: empties, future slots, ragged tiles
    (1, 32, 8, 128, 512, 4096, 0, 0, 8192),   # the Llama-3-8B-shaped chunk
    (2, 8, 2, 128, 300, 700, 11, 20, 3000),   # 3 row tiles per head (the last of 44 rows):
                                              # column sums through the workspace
    (1, 4, 1, 64, 520, 130, 0, 40, 600),      # d = 64, 5 row tiles per head, future slots
    (1, 4, 2, 128, 100, 0, 0, 0, 0),          # one key tile: the odd Q K^T issuer has none
    (1, 4, 2, 128, 48, 128, 0, 0, 300),       # two key tiles: one per Q K^T issuer
]


@pytest.mark.parametrize("case", SDPA_CASES, ids=lambda c: "x".join(map(str, c)))
def test_sdpa_chunk_matches_oracle(dev, case):
    B, Hq, Hkv, d, S, M, n_empty, n_future, pos0 = case
    rng = np.random.default_rng(hash(case) % 2**32)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty)
    for b in range(B):
        for h in range(Hkv):
            occ = np.nonzero(st["slot_pos"][b, h] >= 0)[0]
            for k in range(min(n_future, len(occ))):
                st["slot_pos"][b, h, occ[k]] = pos0 + (k % S)  # visible from row k % S on
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    out, inc = h2o_sdpa_chunk(bf(q, dev), bf(st["k_cache"], dev), bf(st["v_cache"], dev),
                              bf(kn, dev), bf(vn, dev),
                              torch.from_numpy(st["slot_pos"]).to(dev), pos0)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    ref_out, ref_inc, w = oracle_sdpa(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"],
                                      pos0)
    check_sdpa(out, inc, ref_out, ref_inc, w)
    # every query row's weights sum to 1 (§3.1.1)
    np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), S, rtol=1e-4)


DECODE_CASES = [
    # B, Hq, Hkv, d, M, n_empty, n_future, pos0, empty block [lo, hi)
    (1, 4, 1, 128, 1, 0, 0, 5, None),            # a single cache slot
    (2, 8, 2, 128, 63, 0, 0, 100, None),         # less than one 64-key tile
    (1, 5, 1, 128, 64, 0, 0, 70, None),          # q_g = 5 (the 8-head variant)
    (2, 16, 2, 128, 1000, 37, 20, 2000, None),   # q_g = 8, empty and future slots
    (2, 4, 4, 128, 5000, 600, 0, 6000, None),    # q_g = 1, 20 splits with a ragged last one
    (1, 8, 2, 64, 3000, 0, 0, 5000, (256, 768)), # d = 64; whole splits see no key
    (1, 32, 2, 64, 200, 0, 0, 300, None),        # q_g = 16: the chunk kernel takes S = 1
    (8, 32, 8, 128, 4096, 0, 0, 4200, None),     # the decode workload's shape, M = 4096
    (1, 8, 2, 128, 2500, 10, 5, 3000, (300, 700)),  # several splits, ragged last tile, empty block
    (1, 16, 2, 128, 1700, 0, 9, 1800, None),     # q_g = 8 over several splits
]


@pytest.mark.parametrize("case", DECODE_CASES, ids=lambda c: "x".join(map(str, c[:8])))
def test_decode_step_matches_oracle(dev, case):
    """S = 1: the split-K decode kernels (split + combine) against the oracle."""
    B, Hq, Hkv, d, M, n_empty, n_future, pos0, block = case
    rng = np.random.default_rng(hash(case) % 2**32)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty)
    for b in range(B):
        for h in range(Hkv):
            occ = np.nonzero(st["slot_pos"][b, h] >= 0)[0]
            st["slot_pos"][b, h, occ[:min(n_future, len(occ))]] = pos0 + 1 + np.arange(
                min(n_future, len(occ)))  # not visible to the token at pos0
    if block is not None:
        st["slot_pos"][:, :, block[0]:block[1]] = -1
    q = wl.round_bf16(rng.standard_normal((B, Hq, 1, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, 1, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, 1, d), dtype=np.float32))
    for rep in range(2):  # the same workspace twice in a row
        out, inc = h2o_sdpa_chunk(bf(q, dev), bf(st["k_cache"], dev), bf(st["v_cache"], dev),
                                  bf(kn, dev), bf(vn, dev),
                                  torch.from_numpy(st["slot_pos"]).to(dev), pos0)
        torch.cuda.synchronize()
        assert h2o_device_errors() == 0
        ref_out, ref_inc, w = oracle_sdpa(q, st["k_cache"], st["v_cache"], kn, vn,
                                          st["slot_pos"], pos0)
        check_sdpa(out, inc, ref_out, ref_inc, w)
        np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), 1.0, rtol=1e-4)
        # masked slots get exactly zero weight
        hidden = (st["slot_pos"] < 0) | (st["slot_pos"] > pos0)
        g_hidden = np.repeat(hidden, Hq // Hkv, axis=1)
        assert (inc[:, :, :M].cpu().numpy()[g_hidden] == 0).all()


def test_softmax_scale_argument(dev):
    rng = np.random.default_rng(11)
    B, Hq, Hkv, d, S, M, pos0 = 1, 4, 2, 64, 40, 200, 300
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0)
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    out, inc = h2o_sdpa_chunk(bf(q, dev), bf(st["k_cache"], dev), bf(st["v_cache"], dev),
                              bf(kn, dev), bf(vn, dev),
                              torch.from_numpy(st["slot_pos"]).to(dev), pos0, scale=0.3)
    ref_out, ref_inc, w = oracle_sdpa(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"],
                                      pos0, scale=0.3)
    check_sdpa(out, inc, ref_out, ref_inc, w)


UPDATE_CASES = [
    # B, Hq, Hkv, d, S, M, W, n_empty, int_scores
    (1, 4, 2, 64, 32, 256, 32, 0, False),
    (2, 8, 2, 128, 20, 300, 50, 17, True),
    (1, 4, 4, 128, 1, 4096, 64, 0, False),     # S = 1: argmin path
    (1, 4, 1, 128, 1, 70, 64, 0, True),        # S = 1 with ties
    (2, 4, 2, 64, 64, 64, 0, 0, False),        # S = M: everything is overwritten
    (1, 8, 2, 128, 512, 4096, 512, 0, False),  # the Llama-3-8B-shaped chunk
    (1, 2, 1, 64, 5, 2000, 100, 1500, True),   # many empty slots and ties
    (1, 2, 1, 64, 33, 1030, 0, 0, True),       # M not a multiple of the block size
    (4, 32, 8, 128, 256, 2048, 256, 0, False), # batched workload shape
    (2, 8, 2, 128, 1, 16384, 64, 0, False),    # S = 1, clusters of 2
    (1, 4, 2, 64, 1, 65536, 64, 3, True),      # S = 1, clusters of 8, ties and empties
    (2, 8, 2, 64, 1, 9000, 0, 0, True),        # S = 1, no recent window, ragged ranges
]


def _update_inputs(case, seed):
    B, Hq, Hkv, d, S, M, W, n_empty, int_scores = case
    rng = np.random.default_rng(seed)
    pos0 = M + 3 * S + 7
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty, int_scores=int_scores)
    if int_scores:
        inc = rng.integers(0, 3, size=(B, Hq, M + S)).astype(np.float32)
    else:
        inc = rng.gamma(0.3, 0.05, size=(B, Hq, M + S)).astype(np.float32)
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    return st, inc, kn, vn, pos0


@pytest.mark.parametrize("case", UPDATE_CASES, ids=lambda c: "x".join(map(str, c)))
def test_update_is_bit_exact(dev, case):
    B, Hq, Hkv, d, S, M, W, n_empty, int_scores = case
    st, inc, kn, vn, pos0 = _update_inputs(case, hash(case) % 2**32)
    g_scores = torch.from_numpy(st["scores"]).to(dev)
    g_pos = torch.from_numpy(st["slot_pos"]).to(dev)
    g_k = bf(st["k_cache"], dev)
    g_v = bf(st["v_cache"], dev)
    ev = torch.full((B, Hkv, S), -7, dtype=torch.int32, device=dev)
    h2o_update(g_scores, g_pos, torch.from_numpy(inc).to(dev), bf(kn, dev), bf(vn, dev), g_k, g_v,
               pos0, W, evict_idx=ev)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    ref = ref_update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                     pos0, W, "fp32")
    np.testing.assert_array_equal(ev.cpu().numpy(), ref["evict_idx"])
    np.testing.assert_array_equal(g_pos.cpu().numpy(), ref["slot_pos"])
    np.testing.assert_array_equal(g_scores.cpu().numpy().view(np.uint32),
                                  ref["scores"].astype(np.float32).view(np.uint32))
    np.testing.assert_array_equal(f32(g_k), ref["k_cache"])
    np.testing.assert_array_equal(f32(g_v), ref["v_cache"])


POLICY_CASES = [
    # B, Hq, Hkv, d, S, M, W, n_empty, int_scores
    (2, 8, 2, 128, 20, 300, 50, 17, True),      # cluster path, ties
    (1, 8, 2, 128, 512, 4096, 512, 0, False),   # the Llama-3-8B-shaped chunk
    (3, 4, 2, 64, 1, 500, 64, 0, False),        # S = 1: argmin path
    (2, 4, 1, 64, 40, 26000, 100, 0, False),    # keys beyond the cluster variant's shared memory
    (4, 32, 8, 128, 256, 2048, 256, 0, False),  # batched workload shape
    (3, 12, 3, 64, 1, 40000, 64, 0, False),     # S = 1, clusters of 4 (h2o_orig: 3 b each)
]


@pytest.mark.parametrize("case", POLICY_CASES, ids=lambda c: "x".join(map(str, c)))
@pytest.mark.parametrize("policy", ["h2o_norm", "h2o_orig"])
def test_update_policy_is_bit_exact(dev, policy, case):
    """h2o_update_policy against the oracle's policies of §3.1.1, bit for bit."""
    B, Hq, Hkv, d, S, M, W, n_empty, int_scores = case
    st, inc, kn, vn, pos0 = _update_inputs(case, hash((policy,) + case) % 2**32)
    if policy == "h2o_orig":     # one set of positions across the batch
        st["slot_pos"][1:] = st["slot_pos"][0]
    g_scores = torch.from_numpy(st["scores"]).to(dev)
    g_pos = torch.from_numpy(st["slot_pos"]).to(dev)
    g_k = bf(st["k_cache"], dev)
    g_v = bf(st["v_cache"], dev)
    ev = torch.full((B, Hkv, S), -7, dtype=torch.int32, device=dev)
    h2o_update_policy(g_scores, g_pos, torch.from_numpy(inc).to(dev), bf(kn, dev), bf(vn, dev),
                      g_k, g_v, pos0, W, policy, evict_idx=ev)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    ref = ref_update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                     pos0, W, "fp32", policy)
    np.testing.assert_array_equal(ev.cpu().numpy(), ref["evict_idx"])
    np.testing.assert_array_equal(g_pos.cpu().numpy(), ref["slot_pos"])
    np.testing.assert_array_equal(g_scores.cpu().numpy().view(np.uint32),
                                  ref["scores"].astype(np.float32).view(np.uint32))
    np.testing.assert_array_equal(f32(g_k), ref["k_cache"])
    np.testing.assert_array_equal(f32(g_v), ref["v_cache"])
    # the variant changes the victims on these inputs (not a silent h2o)
    plain = ref_update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"],
                       pos0, W, "fp32", "h2o")
    if S >= 20 and (B > 1 or policy == "h2o_norm"):
        assert not np.array_equal(plain["evict_idx"], ref["evict_idx"])


@pytest.mark.parametrize("policy", ["h2o_norm", "h2o_orig"])
def test_tiny_workload_policy_teacher_forced(dev, policy):
    """A whole tiny sequence (B = 2) with each variant: the GPU chunk step against
    the oracle's, from the GPU's own cache state, at every chunk."""
    w = wl.WORKLOADS["tiny"].replace(B=2)
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev, policy=policy)
    layer.reset()
    for i, (p, e) in enumerate(chunk_bounds(w.T, w.M, w.S)):
        q, k, v = wl.batch_tokens(w, p, e)
        before = dict(scores=layer.scores.cpu().numpy(), slot_pos=layer.slot_pos.cpu().numpy(),
                      k_cache=f32(layer.k_cache), v_cache=f32(layer.v_cache))
        out, inc, ev = layer.step(bf(q, dev), bf(k, dev), bf(v, dev), p)
        torch.cuda.synchronize()
        ref = ref_update(before["scores"], before["slot_pos"], inc.cpu().numpy(), k, v,
                         before["k_cache"], before["v_cache"], p, w.W, "fp32", policy)
        np.testing.assert_array_equal(layer.slot_pos.cpu().numpy(), ref["slot_pos"])
        np.testing.assert_array_equal(layer.scores.cpu().numpy().view(np.uint32),
                                      ref["scores"].astype(np.float32).view(np.uint32))
        np.testing.assert_array_equal(f32(layer.k_cache), ref["k_cache"])
    assert h2o_device_errors() == 0
    if policy == "h2o_orig":
        pos = layer.slot_pos.cpu().numpy()
        assert (pos == pos[0:1]).all()


def test_update_twice_in_a_row_without_evict_idx(dev):
    case = (2, 8, 2, 64, 16, 200, 16, 5, True)
    st, inc, kn, vn, pos0 = _update_inputs(case, 5)
    g_scores = torch.from_numpy(st["scores"]).to(dev)
    g_pos = torch.from_numpy(st["slot_pos"]).to(dev)
    g_k, g_v = bf(st["k_cache"], dev), bf(st["v_cache"], dev)
    ref = dict(scores=st["scores"], slot_pos=st["slot_pos"], k_cache=st["k_cache"],
               v_cache=st["v_cache"])
    for step in range(2):
        p = pos0 + step * 16
        h2o_update(g_scores, g_pos, torch.from_numpy(inc).to(dev), bf(kn, dev), bf(vn, dev),
                   g_k, g_v, p, 16)
        ref = ref_update(ref["scores"], ref["slot_pos"], inc, kn, vn, ref["k_cache"],
                         ref["v_cache"], p, 16, "fp32")
    torch.cuda.synchronize()
    np.testing.assert_array_equal(g_pos.cpu().numpy(), ref["slot_pos"])
    np.testing.assert_array_equal(g_scores.cpu().numpy(), ref["scores"])
    np.testing.assert_array_equal(f32(g_k), ref["k_cache"])


def test_update_reports_too_few_candidates_and_leaves_state(dev):
    """slot_pos not produced by the policy: every slot inside the window."""
    B, Hq, Hkv, d, S, M, W = 1, 2, 1, 64, 4, 16, 8
    pos0 = 100
    sp = np.full((B, Hkv, M), pos0 - 1, np.int32)  # all recent
    g_pos = torch.from_numpy(sp).to(dev)
    g_scores = torch.zeros((B, Hkv, M), device=dev)
    g_k = torch.zeros((B, Hkv, M, d), dtype=torch.bfloat16, device=dev)
    g_v = torch.zeros_like(g_k)
    kn = torch.ones((B, Hkv, S, d), dtype=torch.bfloat16, device=dev)
    h2o_update(g_scores, g_pos, torch.ones((B, Hq, M + S), device=dev), kn, kn, g_k, g_v, pos0, W)
    assert h2o_device_errors() == 2
    assert (g_pos.cpu().numpy() == sp).all() and g_k.abs().sum().item() == 0
    assert h2o_device_errors() == 0


@pytest.mark.parametrize("M", [16, 20000])
def test_decode_update_reports_too_few_candidates_and_leaves_state(dev, M):
    """S = 1 (cluster argmin kernel): every slot inside the window."""
    B, Hq, Hkv, d, W = 2, 4, 2, 64, 8
    pos0 = 100
    sp = np.full((B, Hkv, M), pos0 - 1, np.int32)
    g_pos = torch.from_numpy(sp).to(dev)
    sc = np.random.default_rng(3).random((B, Hkv, M), dtype=np.float32)
    g_scores = torch.from_numpy(sc).to(dev)
    g_k = torch.zeros((B, Hkv, M, d), dtype=torch.bfloat16, device=dev)
    kn = torch.ones((B, Hkv, 1, d), dtype=torch.bfloat16, device=dev)
    h2o_update(g_scores, g_pos, torch.ones((B, Hq, M + 1), device=dev), kn, kn, g_k,
               torch.zeros_like(g_k), pos0, W)
    assert h2o_device_errors() == 2
    assert (g_pos.cpu().numpy() == sp).all() and g_k.abs().sum().item() == 0
    np.testing.assert_array_equal(g_scores.cpu().numpy(), sc)
    assert h2o_device_errors() == 0


def _teacher_forced_step(layer, q, kn, vn, p, W):
    """Runs one GPU step and checks it against the oracle started from the GPU's state."""
    before = dict(k=f32(layer.k_cache), v=f32(layer.v_cache), pos=layer.slot_pos.cpu().numpy(),
                  scores=layer.scores.cpu().numpy())
    out, inc, ev = layer.step(q, kn, vn, p)
    torch.cuda.synchronize()
    qn, knn, vnn = f32(q), f32(kn), f32(vn)
    ref_out, ref_inc, w = oracle_sdpa(qn, before["k"], before["v"], knn, vnn, before["pos"], p)
    check_sdpa(out, inc, ref_out, ref_inc, w)
    ref = ref_update(before["scores"], before["pos"], inc.cpu().numpy(), knn, vnn, before["k"],
                     before["v"], p, W, "fp32")
    np.testing.assert_array_equal(ev.cpu().numpy(), ref["evict_idx"])
    np.testing.assert_array_equal(layer.slot_pos.cpu().numpy(), ref["slot_pos"])
    np.testing.assert_array_equal(layer.scores.cpu().numpy(), ref["scores"])
    np.testing.assert_array_equal(f32(layer.k_cache), ref["k_cache"])
    np.testing.assert_array_equal(f32(layer.v_cache), ref["v_cache"])


def test_tiny_workload_every_chunk_teacher_forced(dev):
    """The whole tiny workload (prefill + 24 chunks), every step checked."""
    w = wl.WORKLOADS["tiny"]
    q, k, v = wl.batch_tokens(w, 0, w.T)
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev)
    for p, e in chunk_bounds(w.T, w.M, w.S):
        _teacher_forced_step(layer, bf(q[:, :, p:e], dev), bf(k[:, :, p:e], dev),
                             bf(v[:, :, p:e], dev), p, w.W)
    assert h2o_device_errors() == 0


@pytest.mark.parametrize("name,check_chunks", [("llama8b_32k", (1, 2, 55)),
                                               ("batched_16k", (1, 30)),
                                               ("long_128k", (1, 3))])
def test_full_size_workload_sampled_chunks(dev, name, check_chunks):
    """Full-size workloads through the same launch path as the benchmark.

    The prefill's output is checked on sampled query rows and its summed
    weights (every slot's initial H2O score, Eq. 3) element by element for the
    whole first KV-head group (all q_g query heads, every key column); the
    listed chunks are checked completely (teacher-forced from the GPU's
    state)."""
    w = wl.WORKLOADS[name]
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev)
    bounds = chunk_bounds(w.T, w.M, w.S)
    last = max(check_chunks)
    for n, (p, e) in enumerate(bounds[:last + 1]):
        q, k, v = wl.batch_tokens(w, p, e)
        gq, gk, gv = bf(q, dev), bf(k, dev), bf(v, dev)
        if n == 0:
            out, inc, _ = layer.step(gq, gk, gv, p)
            rows = np.unique(np.concatenate([np.arange(8), np.linspace(0, e - 1, 24).astype(int)]))
            ref_out, _, wr = oracle_sdpa(q, np.zeros_like(f32(layer.k_cache)),
                                         np.zeros_like(f32(layer.v_cache)), k, v,
                                         -np.ones(layer.slot_pos.shape, np.int32), 0, rows=rows)
            check_out(f32(out)[:, :, rows], ref_out, wr)
            np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), e, rtol=1e-4)
            # group (b = 0, kv head 0): q_g heads x (M + S) columns, every row;
            # the oracle runs over row blocks (bounded memory) and the blocks'
            # summed weights add up
            g_out, g_w, g_inc = [], [], 0.0
            for r0 in range(0, e - p, 2048):
                o_, i_, w_ = oracle_sdpa(q[:1, :w.q_g], np.zeros((1, 1, w.M, w.d)),
                                         np.zeros((1, 1, w.M, w.d)), k[:1, :1], v[:1, :1],
                                         -np.ones((1, 1, w.M), np.int32), 0,
                                         rows=np.arange(r0, min(e - p, r0 + 2048)))
                g_out.append(o_)
                g_w.append(w_)
                g_inc = g_inc + i_
            check_sdpa(out[:1, :w.q_g], inc[:1, :w.q_g], np.concatenate(g_out, axis=2), g_inc,
                       np.concatenate(g_w, axis=2))
        elif n in check_chunks:
            _teacher_forced_step(layer, gq, gk, gv, p, w.W)
        else:
            layer.step(gq, gk, gv, p)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0


@pytest.mark.parametrize("name", ["decode_4k", "decode_16k", "decode_64k"])
def test_decode_workload_sampled_steps(dev, name):
    """Decode-style steps (S = 1) after the cache is filled; sampled steps teacher-forced.

    The cache is filled by prefill chunks of at most 4096 tokens: while empty
    slots remain they are taken lowest index first, so a chunked prefill leaves
    the same slots as one prefill call (§3.1 left-to-right fill)."""
    w = wl.WORKLOADS[name]
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev)
    pre = min(w.M, 4096)
    for p in range(0, w.M, pre):
        q, k, v = wl.batch_tokens(w, p, p + pre)
        out, inc, _ = layer.step(bf(q, dev), bf(k, dev), bf(v, dev), p)
        if p == 0:
            rows = np.array([0, 1, 7, pre // 2, pre - 1])
            # query heads 0..q_g-1 share KV head 0
            ref_out, _, wr = oracle_sdpa(q[:1, :w.q_g], np.zeros((1, 1, w.M, w.d)),
                                         np.zeros((1, 1, w.M, w.d)), k[:1, :1], v[:1, :1],
                                         -np.ones((1, 1, w.M), np.int32), 0, rows=rows)
            check_out(f32(out[:1, :w.q_g])[:, :, rows], ref_out, wr)
            np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), pre, rtol=1e-4)
    assert (layer.slot_pos.cpu().numpy() == np.arange(w.M)).all()
    check = {0, 1, 40} if w.M <= 16384 else {0, 40}
    for n in range(41):
        p = w.M + n
        q, k, v = wl.batch_tokens(w, p, p + 1)
        gq, gk, gv = bf(q, dev), bf(k, dev), bf(v, dev)
        if n in check:
            _teacher_forced_step(layer, gq, gk, gv, p, w.W)
        else:
            layer.step(gq, gk, gv, p)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
