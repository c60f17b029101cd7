"""Device-side failure detection, exercised without a GPU fault: a bounded wait
on a barrier nothing completes runs out, the error word reports it, and the
context stays usable for the next calls."""
import numpy as np
import pytest
import torch

from paper_2608_19920_gb300 import build, h2o_device_errors, h2o_sdpa_chunk
from paper_2608_19920_gb300._binding import h2o_selftest_bounded_wait
from paper_2608_19920_gb300 import workloads as wl

from test_gpu_parity import bf, check_sdpa, oracle_sdpa

pytestmark = pytest.mark.gpu


def test_bounded_wait_runs_out_and_is_reported():
    build.build()
    dev = torch.device("cuda:0")
    assert h2o_device_errors() == 0
    h2o_selftest_bounded_wait(5_000_000)   # 5 ms on a barrier that never completes
    assert h2o_device_errors() == 1        # H2O_DEVERR_TIMEOUT, read and cleared
    assert h2o_device_errors() == 0
    # the context still runs the kernels correctly
    rng = np.random.default_rng(3)
    B, Hq, Hkv, d, S, M, pos0 = 1, 4, 2, 64, 32, 256, 256
    st = wl.random_state(rng, B, Hkv, M, d, pos0=pos0)
    q = wl.round_bf16(rng.standard_normal((B, Hq, S, d), dtype=np.float32))
    kn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    vn = wl.round_bf16(rng.standard_normal((B, Hkv, S, d), dtype=np.float32))
    out, inc = h2o_sdpa_chunk(bf(q, dev), bf(st["k_cache"], dev), bf(st["v_cache"], dev),
                              bf(kn, dev), bf(vn, dev), torch.from_numpy(st["slot_pos"]).to(dev),
                              pos0)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    ref_out, ref_inc, w = oracle_sdpa(q, st["k_cache"], st["v_cache"], kn, vn, st["slot_pos"],
                                      pos0)
    check_sdpa(out, inc, ref_out, ref_inc, w)
