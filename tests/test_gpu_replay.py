"""GPU parity of the replay-cache row kernels (h2o_kv_replace / h2o_kv_restore)
against the oracle of §3.2 / §A.1.1: bit-exact copies, through the C ABI."""
import numpy as np
import pytest
import torch

from oracle import kv_replace as ref_replace
from paper_2608_19920_gb300 import (build, h2o_device_errors, h2o_kv_replace, h2o_kv_restore,
                                   h2o_update)
from paper_2608_19920_gb300 import workloads as wl

from test_gpu_parity import bf, f32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def _case(seed, B, Hkv, M, S, d):
    rng = np.random.default_rng(seed)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=M + 50, n_empty=min(3, M - S))
    index = np.stack([np.stack([rng.permutation(M)[:S] for _ in range(Hkv)])
                      for _ in range(B)]).astype(np.int32)
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    return st, index, kn, vn


CASES = [(2, 3, 200, 17, 64), (1, 8, 4096, 512, 128), (8, 8, 4096, 1, 128), (1, 1, 5, 5, 128)]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "x".join(map(str, c)))
def test_replace_and_restore_are_bit_exact(dev, case):
    B, Hkv, M, S, d = case
    st, index, kn, vn = _case(hash(case) % 2**32, B, Hkv, M, S, d)
    pos0 = M + 50
    g_k, g_v = bf(st["k_cache"], dev), bf(st["v_cache"], dev)
    g_pos = torch.from_numpy(st["slot_pos"]).to(dev)
    g_idx = torch.from_numpy(index).to(dev)
    dk = torch.empty((B, Hkv, S, d), dtype=torch.bfloat16, device=dev)
    dv, dp = torch.empty_like(dk), torch.empty((B, Hkv, S), dtype=torch.int32, device=dev)
    h2o_kv_replace(g_idx, bf(kn, dev), bf(vn, dev), g_k, g_v, pos0, slot_pos=g_pos, delta_k=dk,
                   delta_v=dv, delta_pos=dp)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    ref = ref_replace(st["k_cache"], st["v_cache"], st["slot_pos"], index, kn, vn, pos0)
    np.testing.assert_array_equal(f32(g_k), ref["k_cache"])
    np.testing.assert_array_equal(f32(g_v), ref["v_cache"])
    np.testing.assert_array_equal(g_pos.cpu().numpy(), ref["slot_pos"])
    np.testing.assert_array_equal(f32(dk), ref["delta_k"])
    np.testing.assert_array_equal(f32(dv), ref["delta_v"])
    np.testing.assert_array_equal(dp.cpu().numpy(), ref["delta_pos"])
    # the reverse recurrence gives back the buffers bit for bit
    h2o_kv_restore(g_idx, dk, dv, g_k, g_v, slot_pos=g_pos, delta_pos=dp)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(f32(g_k), st["k_cache"])
    np.testing.assert_array_equal(f32(g_v), st["v_cache"])
    np.testing.assert_array_equal(g_pos.cpu().numpy(), st["slot_pos"])


def test_replaying_the_gpu_update_log(dev):
    """A replay cache fed the update's evict_idx writes the update's buffers;
    without delta buffers and positions, only K/V move."""
    rng = np.random.default_rng(31)
    B, Hq, Hkv, M, S, d, pos0 = 2, 8, 2, 1000, 40, 128, 3000
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0)
    inc = rng.gamma(0.3, 0.05, size=(B, Hq, M + S)).astype(np.float32)
    kn = bf(wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32)), dev)
    vn = bf(wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32)), dev)
    k0, v0 = bf(st["k_cache"], dev), bf(st["v_cache"], dev)
    k1, v1 = k0.clone(), v0.clone()
    ev = torch.empty((B, Hkv, S), dtype=torch.int32, device=dev)
    h2o_update(torch.from_numpy(st["scores"]).to(dev), torch.from_numpy(st["slot_pos"]).to(dev),
               torch.from_numpy(inc).to(dev), kn, vn, k1, v1, pos0, S, evict_idx=ev)
    h2o_kv_replace(ev, kn, vn, k0, v0, pos0)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    assert torch.equal(k0, k1) and torch.equal(v0, v1)


def test_out_of_range_index_is_reported_and_skipped(dev):
    """An index outside [0, M) sets H2O_DEVERR_INDEX and skips that row only."""
    B, Hkv, M, S, d = 1, 2, 64, 4, 64
    st, index, kn, vn = _case(5, B, Hkv, M, S, d)
    index[0, 1, 2] = M + 3   # the one bad entry
    g_k, g_v = bf(st["k_cache"], dev), bf(st["v_cache"], dev)
    h2o_kv_replace(torch.from_numpy(index).to(dev), bf(kn, dev), bf(vn, dev), g_k, g_v, 500)
    assert h2o_device_errors() == 4
    full = ref_replace(st["k_cache"], st["v_cache"], st["slot_pos"], index[:, :1], kn[:, :1],
                       vn[:, :1], 500)
    keep = [0, 1, 3]
    part = ref_replace(st["k_cache"][:, 1:], st["v_cache"][:, 1:], st["slot_pos"][:, 1:],
                       index[:, 1:, keep], kn[:, 1:, keep], vn[:, 1:, keep], 500)
    np.testing.assert_array_equal(f32(g_k)[:, :1], full["k_cache"][:, :1])
    np.testing.assert_array_equal(f32(g_k)[:, 1:], part["k_cache"])
    np.testing.assert_array_equal(f32(g_v)[:, 1:], part["v_cache"])
    assert h2o_device_errors() == 0
