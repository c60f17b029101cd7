"""Out-of-bounds writes, caught with canaries (compute-sanitizer is not
available): every output and in-place buffer of a call is carved out of a
larger allocation whose 1 KiB guard regions on both sides hold a sentinel, and
the guards must be untouched after the call.  Ragged shapes throughout."""
import numpy as np
import pytest
import torch

from paper_2608_19920_gb300 import (build, h2o_device_errors, h2o_evict_insert, h2o_kv_replace,
                                   h2o_sdpa_cache, h2o_sdpa_chunk, h2o_sdpa_chunk_backward,
                                   h2o_update)
from paper_2608_19920_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

GUARD_BYTES = 1024


class Guarded:
    """A tensor of `shape` inside a buffer with sentinel-filled guards."""

    def __init__(self, shape, dtype, dev, init=None):
        item = torch.empty((), dtype=dtype).element_size()
        self.g = GUARD_BYTES // item
        n = int(np.prod(shape))
        self.buf = torch.empty(n + 2 * self.g, dtype=dtype, device=dev)
        self.buf.view(torch.uint8).fill_(0xA5)
        self.t = self.buf[self.g:self.g + n].view(shape)
        if init is not None:
            self.t.copy_(init)

    def intact(self):
        raw = self.buf.view(torch.uint8)
        gb = self.g * self.buf.element_size()
        return bool((raw[:gb] == 0xA5).all()) and bool((raw[-gb:] == 0xA5).all())


@pytest.fixture(scope="module")
def dev():
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def _inputs(dev, B, Hq, Hkv, d, S, M, pos0, seed):
    rng = np.random.default_rng(seed)
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=min(3, M // 4))
    f = lambda x: torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(dev)
    q = f(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = f(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = f(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    return st, q, kn, vn, f


@pytest.mark.parametrize("case", [(2, 6, 3, 64, 20, 300, 900), (3, 8, 2, 128, 1, 777, 800),
                                  (1, 7, 1, 128, 130, 390, 1000)],
                         ids=lambda c: "x".join(map(str, c)))
def test_no_call_writes_outside_its_buffers(dev, case):
    B, Hq, Hkv, d, S, M, pos0 = case
    st, q, kn, vn, f = _inputs(dev, B, Hq, Hkv, d, S, M, pos0, hash(case) % 2**32)
    bf, f32, i32 = torch.bfloat16, torch.float32, torch.int32
    kc = Guarded((B, Hkv, M, d), bf, dev, f(st["k_cache"]))
    vc = Guarded((B, Hkv, M, d), bf, dev, f(st["v_cache"]))
    sp = Guarded((B, Hkv, M), i32, dev, torch.from_numpy(st["slot_pos"]))
    sc = Guarded((B, Hkv, M), f32, dev, torch.from_numpy(st["scores"]))
    out = Guarded((B, Hq, S, d), bf, dev)
    inc = Guarded((B, Hq, M + S), f32, dev)
    # chunk SDPA (decode kernels when S = 1, with a guarded workspace)
    from paper_2608_19920_gb300 import H2ODims, h2o_workspace_size
    n_ws = h2o_workspace_size(H2ODims(B, Hq, Hkv, d, S, M))
    ws = Guarded((max(n_ws, 16),), torch.uint8, dev)
    h2o_sdpa_chunk(q, kc.t, vc.t, kn, vn, sp.t, pos0, out=out.t, score_inc=inc.t,
                   workspace=ws.t if n_ws else None)
    # update
    ev = Guarded((B, Hkv, S), i32, dev)
    h2o_update(sc.t, sp.t, inc.t, kn, vn, kc.t, vc.t, pos0, S, evict_idx=ev.t)
    # backward of a chunk
    dout = f(np.random.default_rng(1).standard_normal((B, Hq, S, d), dtype=np.float32))
    o2, _ = h2o_sdpa_chunk(q, kc.t, vc.t, kn, vn, sp.t, pos0 + S)
    grads = h2o_sdpa_chunk_backward(q, kc.t, vc.t, kn, vn, sp.t, pos0 + S, o2, dout)
    # replay rows
    dk = Guarded((B, Hkv, S, d), bf, dev)
    dv = Guarded((B, Hkv, S, d), bf, dev)
    dp = Guarded((B, Hkv, S), i32, dev)
    h2o_kv_replace(ev.t, kn, vn, kc.t, vc.t, pos0 + 2 * S, slot_pos=sp.t, delta_k=dk.t,
                   delta_v=dv.t, delta_pos=dp.t)
    # paper order: evict-insert and cache-only SDPA
    ev2 = Guarded((B, Hkv, S), i32, dev)
    h2o_evict_insert(sc.t, sp.t, kn, vn, kc.t, vc.t, pos0 + 3 * S, S, evict_idx=ev2.t, Hq=Hq)
    inc_c = Guarded((B, Hq, M), f32, dev)
    out_c = Guarded((B, Hq, S, d), bf, dev)
    h2o_sdpa_cache(q, kc.t, vc.t, sp.t, pos0 + 3 * S, out=out_c.t, score_inc=inc_c.t)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    for name, g in dict(k_cache=kc, v_cache=vc, slot_pos=sp, scores=sc, out=out, score_inc=inc,
                        workspace=ws, evict_idx=ev, delta_k=dk, delta_v=dv, delta_pos=dp,
                        evict_idx2=ev2, score_inc_cache=inc_c, out_cache=out_c).items():
        assert g.intact(), f"{name}: a guard byte was overwritten"
    assert all(torch.isfinite(x).all() for x in grads if x.numel())
