"""h2o_sdpa_decode_static: the decode SDPA on the library's fixed device scratch.

Called through the C ABI and compared, bit for bit, with h2o_sdpa_chunk (the
same kernels with a caller-allocated workspace) on two calls in a row with
different inputs.  Kept in a file of its own that runs last, and written to
pass both alone in a fresh process and after the other tests.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2608_19920_gb300 import _binding as lib_mod
from paper_2608_19920_gb300 import build, h2o_device_errors, h2o_sdpa_chunk
from paper_2608_19920_gb300 import workloads as wl

pytestmark = pytest.mark.gpu

SCRATCH_LIMIT = 16 << 20  # bytes of the fixed scratch (include/h2o.h)


def _inputs(rng, B, Hq, Hkv, d, M, pos0, dev):
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0, n_empty=M // 10)
    f = lambda x: torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(torch.bfloat16).to(dev)
    q = f(rng.standard_normal((B, Hq, 1, d), dtype=np.float32))
    kn = f(rng.standard_normal((B, Hkv, 1, d), dtype=np.float32))
    vn = f(rng.standard_normal((B, Hkv, 1, d), dtype=np.float32))
    return (q, f(st["k_cache"]), f(st["v_cache"]), kn, vn,
            torch.from_numpy(st["slot_pos"]).to(dev))


def _call_static(lib, args, pos0, out, inc):
    q, kc, vc, kn, vn, sp = args
    B, Hq, S, d = q.shape
    dims = lib_mod.H2ODims(B, Hq, kn.shape[1], d, S, kc.shape[2])
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    return lib.h2o_sdpa_decode_static(ctypes.byref(dims), pos0, 0.0, p(q), p(kc), p(vc), p(kn),
                                      p(vn), p(sp), p(out), p(inc), None)


@pytest.mark.parametrize("shape", [(8, 32, 8, 128, 4096), (2, 12, 2, 64, 3001)],
                         ids=["decode_4k", "ragged_d64"])
def test_static_scratch_matches_workspace_path(shape):
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    dev = torch.device("cuda:0")
    lib = lib_mod.load()
    B, Hq, Hkv, d, M = shape
    rng = np.random.default_rng(M)
    for call in range(2):  # two calls in a row share the scratch
        pos0 = M + 5 + call
        args = _inputs(rng, B, Hq, Hkv, d, M, pos0, dev)
        out = torch.full((B, Hq, 1, d), 7.0, dtype=torch.bfloat16, device=dev)
        inc = torch.full((B, Hq, M + 1), -3.0, dtype=torch.float32, device=dev)
        assert _call_static(lib, args, pos0, out, inc) == 0
        ref_out, ref_inc = h2o_sdpa_chunk(*args, pos0)
        torch.cuda.synchronize()
        assert h2o_device_errors() == 0
        assert torch.equal(out, ref_out)
        assert torch.equal(inc, ref_inc)
        np.testing.assert_allclose(inc.sum(-1).cpu().numpy(), 1.0, rtol=1e-4)


def test_static_scratch_rejects_sizes_beyond_its_limit():
    build.build()
    lib = lib_mod.load()
    n = ctypes.c_size_t(0)
    big = lib_mod.H2ODims(16, 64, 8, 128, 1, 262144)
    assert lib.h2o_workspace_size(ctypes.byref(big), ctypes.byref(n)) == 0
    assert n.value > SCRATCH_LIMIT
    vp = ctypes.c_void_p(0x1000)
    assert lib.h2o_sdpa_decode_static(ctypes.byref(big), 262200, 0.0, *[vp] * 8, None) == -5
    chunk = lib_mod.H2ODims(1, 4, 2, 64, 32, 256)  # not a decode step
    assert lib.h2o_sdpa_decode_static(ctypes.byref(chunk), 256, 0.0, *[vp] * 8, None) == -4
