"""GPU parity of the paper-order chunk step (§3.1, §3.3.1) against the oracle:
h2o_evict_insert and h2o_scores_add bit for bit, h2o_sdpa_cache within the
SDPA tolerances (out: 1e-2 above bf16 rounding; score_inc: 1e-3 relative +
1e-7), through the C ABI, on the same seeded inputs."""
import numpy as np
import pytest
import torch

from oracle import evict_insert as ref_evict_insert
from oracle import scores_add as ref_scores_add
from oracle import sdpa_cache as ref_sdpa_cache
from paper_2608_19920_gb300 import (H2OLayer, build, h2o_device_errors, h2o_evict_insert,
                                   h2o_scores_add, h2o_sdpa_cache)
from paper_2608_19920_gb300 import workloads as wl
from paper_2608_19920_gb300.runner import chunk_bounds

from test_gpu_parity import bf, check_out, check_sdpa, f32, with_abs_values

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


EVICT_CASES = [
    # B, Hkv, d, S, M, W, n_empty, int_scores, policy
    (2, 2, 128, 20, 300, 50, 17, True, "h2o"),        # cluster path, ties, empties
    (1, 8, 128, 512, 4096, 512, 0, False, "h2o"),     # the Llama-3-8B-shaped chunk
    (3, 2, 64, 1, 500, 64, 0, False, "h2o"),          # S = 1 (cluster argmin kernel)
    (2, 2, 64, 1, 20000, 64, 0, True, "h2o_norm"),    # S = 1, clusters of 2
    (2, 1, 64, 40, 26000, 100, 0, False, "h2o"),      # beyond the cluster kernel's smem
    (3, 2, 64, 16, 700, 32, 0, False, "h2o_orig"),    # one choice per kv head
    (2, 2, 128, 64, 64, 0, 64, False, "h2o_norm"),    # prefill: S = M into an empty cache
]


@pytest.mark.parametrize("case", EVICT_CASES, ids=lambda c: "x".join(map(str, c)))
def test_evict_insert_is_bit_exact(dev, case):
    B, Hkv, d, S, M, W, n_empty, int_scores, policy = case
    rng = np.random.default_rng(hash(case) % 2**32)
    pos0 = M + 3 * S + 7
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty, int_scores=int_scores)
    if policy == "h2o_orig":
        st["slot_pos"][1:] = st["slot_pos"][0]
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    g_scores = torch.from_numpy(st["scores"]).to(dev)
    g_pos = torch.from_numpy(st["slot_pos"]).to(dev)
    g_k, g_v = bf(st["k_cache"], dev), bf(st["v_cache"], dev)
    ev = torch.full((B, Hkv, S), -7, dtype=torch.int32, device=dev)
    h2o_evict_insert(g_scores, g_pos, bf(kn, dev), bf(vn, dev), g_k, g_v, pos0, W, policy=policy,
                     evict_idx=ev)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    ref = ref_evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                           pos0, W, "fp32", policy)
    np.testing.assert_array_equal(ev.cpu().numpy(), ref["evict_idx"])
    np.testing.assert_array_equal(g_pos.cpu().numpy(), ref["slot_pos"])
    np.testing.assert_array_equal(g_scores.cpu().numpy().view(np.uint32),
                                  ref["scores"].astype(np.float32).view(np.uint32))
    np.testing.assert_array_equal(f32(g_k), ref["k_cache"])
    np.testing.assert_array_equal(f32(g_v), ref["v_cache"])


CACHE_CASES = [
    # B, Hq, Hkv, d, S, M, pos0
    (1, 4, 2, 64, 32, 256, 256),       # the tiny workload's chunk shape
    (2, 8, 2, 128, 20, 300, 900),      # ragged S < 32, ragged M
    (1, 7, 1, 128, 200, 384, 1000),    # S > 128 with a ragged row tile, q_g = 7
    (1, 32, 8, 128, 512, 4096, 8192),  # the Llama-3-8B-shaped chunk
    (3, 12, 3, 128, 1, 5000, 6000),    # S = 1: the split-K decode kernels, no new-token column
    (2, 6, 3, 64, 1, 130, 140),        # S = 1, d = 64
    (1, 32, 2, 64, 1, 200, 300),       # S = 1, q_g = 16: the chunk kernel
]


@pytest.mark.parametrize("case", CACHE_CASES, ids=lambda c: "x".join(map(str, c)))
def test_sdpa_cache_matches_oracle(dev, case):
    """The cache as h2o_evict_insert leaves it: the chunk's tokens sit in
    scattered slots; row i sees the slots with positions <= pos0 + i."""
    B, Hq, Hkv, d, S, M, pos0 = case
    rng = np.random.default_rng(hash(case) % 2**32)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=min(5, M - S))
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    ins = ref_evict_insert(st["scores"], st["slot_pos"], kn, vn, st["k_cache"], st["v_cache"],
                           pos0, 0, "fp32")
    out, inc = h2o_sdpa_cache(bf(q, dev), bf(ins["k_cache"], dev), bf(ins["v_cache"], dev),
                              torch.from_numpy(ins["slot_pos"]).to(dev), pos0)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    ref_out, ref_inc, w = with_abs_values(ref_sdpa_cache, (q, ins["k_cache"], ins["v_cache"],
                                                           ins["slot_pos"], pos0), (2,))
    check_sdpa(out, inc, ref_out, ref_inc, w)
    np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), S, rtol=1e-4)


def test_scores_add_is_bit_exact(dev):
    rng = np.random.default_rng(12)
    B, Hkv, qg, M = 3, 4, 7, 3001
    scores = rng.gamma(0.5, 2.0, size=(B, Hkv, M)).astype(np.float32)
    inc = rng.gamma(0.3, 0.05, size=(B, Hkv * qg, M)).astype(np.float32)
    g = torch.from_numpy(scores).to(dev)
    h2o_scores_add(g, torch.from_numpy(inc).to(dev))
    torch.cuda.synchronize()
    ref = ref_scores_add(scores, inc, "fp32")
    np.testing.assert_array_equal(g.cpu().numpy().view(np.uint32), ref.view(np.uint32))


def _paper_step_teacher_forced(layer, q, kn, vn, p, W, policy="h2o"):
    before = dict(k=f32(layer.k_cache), v=f32(layer.v_cache), pos=layer.slot_pos.cpu().numpy(),
                  scores=layer.scores.cpu().numpy())
    out, inc, ev = layer.step(q, kn, vn, p)
    torch.cuda.synchronize()
    qn, knn, vnn = f32(q), f32(kn), f32(vn)
    ins = ref_evict_insert(before["scores"], before["pos"], knn, vnn, before["k"], before["v"],
                           p, W, "fp32", policy)
    np.testing.assert_array_equal(ev.cpu().numpy(), ins["evict_idx"])
    np.testing.assert_array_equal(layer.slot_pos.cpu().numpy(), ins["slot_pos"])
    np.testing.assert_array_equal(f32(layer.k_cache), ins["k_cache"])
    ref_out, ref_inc, w = with_abs_values(ref_sdpa_cache, (qn, ins["k_cache"], ins["v_cache"],
                                                           ins["slot_pos"], p), (2,))
    check_sdpa(out, inc, ref_out, ref_inc, w)
    ref_scores = ref_scores_add(ins["scores"], inc.cpu().numpy(), "fp32")
    np.testing.assert_array_equal(layer.scores.cpu().numpy().view(np.uint32),
                                  ref_scores.view(np.uint32))


@pytest.mark.parametrize("policy", ["h2o", "h2o_norm"])
def test_tiny_workload_paper_order_every_chunk(dev, policy):
    w = wl.WORKLOADS["tiny"]
    q, k, v = wl.batch_tokens(w, 0, w.T)
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev, policy=policy,
                     order="paper")
    layer.reset()
    for p, e in chunk_bounds(w.T, w.M, w.S):
        _paper_step_teacher_forced(layer, bf(q[:, :, p:e], dev), bf(k[:, :, p:e], dev),
                                   bf(v[:, :, p:e], dev), p, w.W, policy)
    assert h2o_device_errors() == 0


@pytest.mark.parametrize("name,check", [("llama8b_32k", (1, 2, 30)), ("decode_4k", (1, 2, 9))])
def test_full_size_paper_order_sampled(dev, name, check):
    """Full-size shapes through the same launch path as the benchmark; the listed
    steps are checked teacher-forced, the prefill on sampled rows."""
    w = wl.WORKLOADS[name]
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev, order="paper")
    layer.reset()
    bounds = chunk_bounds(w.T, w.M, w.S)[:max(check) + 1]
    for n, (p, e) in enumerate(bounds):
        q, k, v = wl.batch_tokens(w, p, e)
        gq, gk, gv = bf(q, dev), bf(k, dev), bf(v, dev)
        if n == 0:
            out, inc, _ = layer.step(gq, gk, gv, p)
            rows = np.unique(np.concatenate([np.arange(4), np.linspace(0, e - 1, 12).astype(int)]))
            ref_out, _, wr = with_abs_values(
                ref_sdpa_cache, (q[:1, :w.q_g], k[:1, :1], v[:1, :1],
                                 np.arange(e, dtype=np.int32)[None, None], 0), (2,), rows=rows)
            check_out(f32(out[:1, :w.q_g])[:, :, rows], ref_out, wr)
            np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), e, rtol=1e-4)
        elif n in check:
            _paper_step_teacher_forced(layer, gq, gk, gv, p, w.W)
        else:
            layer.step(gq, gk, gv, p)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
