"""GPU parity of the 8-bit K/V buffer calls against the oracle (oracle/quant.py),
through the C ABI, on the same seeded inputs: the quantiser, the read-back and
the q8 updates bit for bit (codes, scales, scores, positions, evict_idx); the
q8 SDPA calls within the SDPA tolerances of the bf16 calls (S = 1: the decode
kernels reading the codes; S > 1: the read-back, then the chunk kernel)."""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_19920_gb300 import (build, h2o_device_errors, h2o_evict_insert_q8,
                                   h2o_kv_dequantize, h2o_kv_quantize, h2o_sdpa_cache_q8,
                                   h2o_sdpa_chunk_q8, h2o_update_q8)
from paper_2608_19920_gb300._binding import H2O_DEVERR_CANDIDATES
from paper_2608_19920_gb300 import workloads as wl

from test_gpu_parity import bf, check_sdpa, with_abs_values

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def _rows(rng, n, d):
    """bf16 rows of mixed magnitudes, with zero rows and exact rounding ties."""
    x = rng.standard_normal((n, d), dtype=np.float32) * np.exp(rng.uniform(-6, 6, (n, 1)))
    x = wl.round_bf16(x.astype(np.float32))
    x[3] = 0.0                                    # s = 0
    x[5, :] = np.arange(d) % 9 - 4 + 0.5           # ties at s = 1
    x[5, 0] = 127.0
    x[7, :] = -x[7, :]
    return x


@pytest.mark.parametrize("d", [64, 128])
@pytest.mark.parametrize("n", [1, 37, 4133])
def test_quantize_is_bit_exact(dev, d, n):
    rng = np.random.default_rng(n * 1000 + d)
    x = _rows(rng, max(n, 8), d)[:n] if n >= 8 else wl.round_bf16(
        rng.standard_normal((n, d), dtype=np.float32))
    codes, scales = h2o_kv_quantize(bf(x, dev))
    torch.cuda.synchronize()
    rc, rs = oracle.quantize_rows(x)
    np.testing.assert_array_equal(scales.cpu().numpy().view(np.uint32), rs.view(np.uint32))
    np.testing.assert_array_equal(codes.cpu().numpy(), rc)


@pytest.mark.parametrize("d", [64, 128])
def test_dequantize_is_bit_exact(dev, d):
    rng = np.random.default_rng(d)
    n = 3001
    codes = rng.integers(-127, 128, size=(n, d)).astype(np.int8)
    scales = (rng.gamma(1.0, 1.0, n) * np.exp(rng.uniform(-10, 3, n))).astype(np.float32)
    scales[::97] = 0.0
    x = h2o_kv_dequantize(torch.from_numpy(codes).to(dev), torch.from_numpy(scales).to(dev))
    torch.cuda.synchronize()
    ref = oracle.dequantize_rows(codes, scales)
    np.testing.assert_array_equal(x.float().cpu().numpy().view(np.uint32), ref.view(np.uint32))


def _q8_state(rng, B, Hkv, M, d, pos0, n_empty=0, int_scores=False):
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=n_empty, int_scores=int_scores)
    kc, ks = oracle.quantize_rows(st["k_cache"])
    vc, vs = oracle.quantize_rows(st["v_cache"])
    return st, kc, ks, vc, vs


def _gpu_q8(kc, ks, vc, vs, dev):
    t = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    return t(kc), t(ks), t(vc), t(vs)


def _check_buffers(g, ref):
    np.testing.assert_array_equal(g[0].cpu().numpy(), ref["k_codes"])
    np.testing.assert_array_equal(g[1].cpu().numpy().view(np.uint32), ref["k_scales"].view(np.uint32))
    np.testing.assert_array_equal(g[2].cpu().numpy(), ref["v_codes"])
    np.testing.assert_array_equal(g[3].cpu().numpy().view(np.uint32), ref["v_scales"].view(np.uint32))


UPDATE_CASES = [
    # B, Hq, Hkv, d, S, M, W, n_empty, policy, insert
    (2, 8, 2, 128, 20, 300, 50, 17, "h2o", False),     # chunk order, ragged, empties
    (1, 32, 8, 128, 512, 4096, 512, 0, "h2o", False),  # the Llama-3-8B-shaped chunk
    (3, 8, 2, 64, 1, 500, 64, 0, "h2o", False),        # S = 1: the decode update kernel
    (3, 6, 2, 64, 16, 700, 32, 0, "h2o_orig", False),  # one choice per kv head
    (2, 8, 2, 128, 20, 300, 50, 17, "h2o", True),      # paper order (evict, then insert)
    (2, 4, 2, 64, 64, 64, 0, 64, "h2o_norm", True),    # prefill into an empty cache
    (1, 32, 8, 128, 512, 4096, 512, 0, "h2o", True),
]


@pytest.mark.parametrize("case", UPDATE_CASES, ids=lambda c: "x".join(map(str, c)))
def test_q8_update_is_bit_exact(dev, case):
    B, Hq, Hkv, d, S, M, W, n_empty, policy, insert = case
    rng = np.random.default_rng(hash(case) % 2**32)
    pos0 = M + 3 * S + 7
    st, kc, ks, vc, vs = _q8_state(rng, B, Hkv, M, d, pos0, n_empty, int_scores=True)
    if policy == "h2o_orig":
        st["slot_pos"][1:] = st["slot_pos"][0]
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    g_scores = torch.from_numpy(st["scores"]).to(dev)
    g_pos = torch.from_numpy(st["slot_pos"]).to(dev)
    g = _gpu_q8(kc, ks, vc, vs, dev)
    if insert:
        ev = h2o_evict_insert_q8(g_scores, g_pos, bf(kn, dev), bf(vn, dev), *g, pos0, W,
                                 policy=policy, Hq=Hq)
        ref = oracle.evict_insert_q8(st["scores"], st["slot_pos"], kn, vn, kc, ks, vc, vs, pos0,
                                     W, "fp32", policy)
    else:
        inc = rng.gamma(0.3, 0.05, size=(B, Hq, M + S)).astype(np.float32)
        ev = h2o_update_q8(g_scores, g_pos, torch.from_numpy(inc).to(dev), bf(kn, dev),
                           bf(vn, dev), *g, pos0, W, policy=policy)
        ref = oracle.update_q8(st["scores"], st["slot_pos"], inc, kn, vn, kc, ks, vc, vs, pos0, W,
                               "fp32", policy)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    np.testing.assert_array_equal(ev.cpu().numpy(), ref["evict_idx"])
    np.testing.assert_array_equal(g_pos.cpu().numpy(), ref["slot_pos"])
    np.testing.assert_array_equal(g_scores.cpu().numpy().view(np.uint32),
                                  ref["scores"].astype(np.float32).view(np.uint32))
    _check_buffers(g, ref)


def test_q8_update_without_candidates_leaves_the_buffers(dev):
    """Slot positions this policy never produces (all after the chunk): no
    candidates, each (b, h) is left as it is, evict_idx stays -1 and the error
    is recorded."""
    rng = np.random.default_rng(77)
    B, Hkv, d, S, M, pos0 = 1, 2, 64, 4, 32, 100
    st, kc, ks, vc, vs = _q8_state(rng, B, Hkv, M, d, pos0)
    st["slot_pos"][:] = pos0 + 100 + np.arange(M)
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    g = _gpu_q8(kc, ks, vc, vs, dev)
    ev = h2o_evict_insert_q8(torch.from_numpy(st["scores"]).to(dev),
                             torch.from_numpy(st["slot_pos"]).to(dev), bf(kn, dev), bf(kn, dev),
                             *g, pos0, 8)
    torch.cuda.synchronize()
    assert h2o_device_errors() & H2O_DEVERR_CANDIDATES
    assert (ev.cpu().numpy() == -1).all()
    _check_buffers(g, dict(k_codes=kc, k_scales=ks, v_codes=vc, v_scales=vs))


SDPA_CASES = [
    # B, Hq, Hkv, d, S, M, pos0, cache_only
    (1, 4, 2, 64, 32, 256, 256, False),       # the tiny workload's chunk shape
    (2, 8, 2, 128, 20, 300, 900, False),      # ragged S and M
    (1, 32, 8, 128, 512, 4096, 8192, False),  # the Llama-3-8B-shaped chunk
    (3, 12, 3, 128, 1, 5000, 6000, False),    # S = 1: the split-K decode kernels
    (2, 8, 2, 128, 20, 300, 900, True),       # paper order: the cache only
    (1, 32, 8, 128, 512, 4096, 8192, True),
    (2, 6, 3, 64, 1, 130, 140, True),         # S = 1, d = 64
    (1, 4, 1, 128, 1, 255, 300, False),       # S = 1: a ring slot of 127 code rows + the new bf16 row
    (2, 16, 2, 64, 1, 777, 900, False),       # S = 1, q_g = 8, d = 64
    (1, 8, 1, 128, 1, 1537, 1600, True),      # S = 1, q_g = 8, a last tile of one code row
    (1, 16, 2, 128, 1, 2052, 2100, False),    # S = 1, d = 128, M % 4 = 0: the tensor-core kernel
    (2, 8, 1, 128, 1, 1536, 1600, True),      # the same with q_g = 8, cache only
]


@pytest.mark.parametrize("case", SDPA_CASES, ids=lambda c: "x".join(map(str, c)))
def test_q8_sdpa_matches_oracle(dev, case):
    B, Hq, Hkv, d, S, M, pos0, cache_only = case
    rng = np.random.default_rng(hash(case) % 2**32)
    st, kc, ks, vc, vs = _q8_state(rng, B, Hkv, M, d, pos0, n_empty=min(5, M - S))
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32) / np.sqrt(d))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    g = _gpu_q8(kc, ks, vc, vs, dev)
    if cache_only:
        ins = oracle.evict_insert_q8(st["scores"], st["slot_pos"], kn, vn, kc, ks, vc, vs, pos0, 0)
        g = _gpu_q8(ins["k_codes"], ins["k_scales"], ins["v_codes"], ins["v_scales"], dev)
        sp = ins["slot_pos"]
        out, inc = h2o_sdpa_cache_q8(bf(q, dev), *g, torch.from_numpy(sp).to(dev), pos0)
        ref_out, ref_inc, w = with_abs_values(
            oracle.sdpa_cache_q8, (q, ins["k_codes"], ins["k_scales"], ins["v_codes"],
                                   ins["v_scales"], sp, pos0), (3,))
    else:
        sp = st["slot_pos"]
        out, inc = h2o_sdpa_chunk_q8(bf(q, dev), *g, bf(kn, dev), bf(vn, dev),
                                     torch.from_numpy(sp).to(dev), pos0)
        # |codes| give |bf16(c s)| (the rounding is symmetric, scales >= 0)
        ref_out, ref_inc, w = with_abs_values(oracle.sdpa_chunk_q8,
                                              (q, kc, ks, vc, vs, kn, vn, sp, pos0), (3, 6))
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    check_sdpa(out, inc, ref_out, ref_inc, w)
    np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), S, rtol=1e-4)
