"""Pins of the replay-cache row oracle (§3.2 recurrence, §A.1.1 scatter / gather).

The paper defines the buffer writes and reads as torch.scatter_ / torch.gather
along the slot axis with an index constant along the last axis (§A.1.1); the
oracle is checked against those definitions, against the inverse property of
the reverse recurrence, and against the (independently pinned) update oracle,
whose eviction writes are exactly such a scatter.
"""
import numpy as np
import pytest
import torch

from oracle import kv_replace, kv_restore, update
from paper_2608_19920_gb300 import workloads as wl


def _case(seed, B=2, Hkv=3, M=20, S=6, d=8):
    rng = np.random.default_rng(seed)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=100, n_empty=3)
    index = np.stack([np.stack([rng.permutation(M)[:S] for _ in range(Hkv)]) for _ in range(B)])
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    return st, index.astype(np.int32), kn, vn


@pytest.mark.parametrize("seed", range(5))
def test_replace_is_torch_scatter_and_delta_is_torch_gather(seed):
    st, index, kn, vn = _case(seed)
    res = kv_replace(st["k_cache"], st["v_cache"], st["slot_pos"], index, kn, vn, 100)
    d = kn.shape[-1]
    idx = torch.from_numpy(index.astype(np.int64))[..., None].expand(-1, -1, -1, d)
    k = torch.from_numpy(st["k_cache"])
    np.testing.assert_array_equal(res["delta_k"], torch.gather(k, 2, idx).numpy())
    np.testing.assert_array_equal(res["k_cache"],
                                  k.clone().scatter_(2, idx, torch.from_numpy(kn)).numpy())
    pos = torch.from_numpy(st["slot_pos"].astype(np.int64))
    i3 = torch.from_numpy(index.astype(np.int64))
    np.testing.assert_array_equal(res["delta_pos"], torch.gather(pos, 2, i3).numpy())
    newpos = torch.from_numpy(100 + np.broadcast_to(np.arange(index.shape[2]), index.shape).copy())
    np.testing.assert_array_equal(res["slot_pos"], pos.clone().scatter_(2, i3, newpos).numpy())


@pytest.mark.parametrize("seed", range(5))
def test_restore_inverts_replace(seed):
    """Eq. (recurrence-reverse): scatter(keys', index, gather(keys, index)) = keys."""
    st, index, kn, vn = _case(10 + seed)
    res = kv_replace(st["k_cache"], st["v_cache"], st["slot_pos"], index, kn, vn, 100)
    back = kv_restore(res["k_cache"], res["v_cache"], res["slot_pos"], index, res["delta_k"],
                      res["delta_v"], res["delta_pos"])
    np.testing.assert_array_equal(back["k_cache"], st["k_cache"])
    np.testing.assert_array_equal(back["v_cache"], st["v_cache"])
    np.testing.assert_array_equal(back["slot_pos"], st["slot_pos"])


def test_replaying_the_update_log_reproduces_its_cache():
    """A replay cache (§3.2) that is given the update's eviction indices writes
    the same buffers as the update itself; rows outside the index are untouched."""
    rng = np.random.default_rng(21)
    B, Hq, Hkv, M, S, d, pos0 = 2, 4, 2, 30, 5, 8, 200
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0)
    inc = rng.gamma(0.3, 0.05, size=(B, Hq, M + S)).astype(np.float32)
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    upd = update(st["scores"], st["slot_pos"], inc, kn, vn, st["k_cache"], st["v_cache"], pos0,
                 S, "fp32")
    res = kv_replace(st["k_cache"], st["v_cache"], st["slot_pos"], upd["evict_idx"], kn, vn, pos0)
    np.testing.assert_array_equal(res["k_cache"], upd["k_cache"])
    np.testing.assert_array_equal(res["v_cache"], upd["v_cache"])
    np.testing.assert_array_equal(res["slot_pos"], upd["slot_pos"])
    for b in range(B):
        for h in range(Hkv):
            kept = np.setdiff1d(np.arange(M), upd["evict_idx"][b, h])
            np.testing.assert_array_equal(res["k_cache"][b, h, kept], st["k_cache"][b, h, kept])
