"""Run-to-run reproducibility of a whole H2O sequence on the GPU.

§3.2 replays a forward pass from its log of evicted slots, so the decisions
must not change between two runs of the same sequence.  The eviction choice
depends on the summed attention weights, so score_inc itself has to come out
bit-identical run after run: with three or more 128-row tiles per query head
the chunk kernel stores each tile's column sums and a second kernel adds them
in a fixed order; with one or two tiles the additions onto zero commute.
"""
import numpy as np
import pytest
import torch

from paper_2608_19920_gb300 import H2OLayer, build, h2o_device_errors
from paper_2608_19920_gb300 import workloads as wl
from paper_2608_19920_gb300.runner import chunk_bounds

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dev():
    build.build()
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    return torch.device("cuda:0")


def _run(w, plan, inputs, dev, order="chunk"):
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev, order=order)
    layer.reset()
    record = []
    for (p, e), (q, k, v) in zip(plan, inputs):
        out, inc, ev = layer.step(q, k, v, p)
        record.append((out.clone(), inc.clone(), ev.clone()))
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    return record, layer.scores.clone(), layer.slot_pos.clone(), layer.k_cache.clone()


def _same_bits(a, b):
    return torch.equal(a.contiguous().view(torch.uint8), b.contiguous().view(torch.uint8))


@pytest.mark.parametrize("name,n_chunks,order", [("llama8b_32k", 12, "chunk"),
                                                 ("long_128k", 3, "chunk"),
                                                 ("llama8b_32k", 6, "paper")])
def test_sequence_is_bit_reproducible(dev, name, n_chunks, order):
    w = wl.WORKLOADS[name]
    plan = chunk_bounds(w.T, w.M, w.S)[:n_chunks + 1]
    inputs = [tuple(torch.from_numpy(np.ascontiguousarray(x)).to(torch.bfloat16).to(dev)
                    for x in wl.batch_tokens(w, p, e)) for p, e in plan]
    r1, sc1, sp1, kc1 = _run(w, plan, inputs, dev, order)
    r2, sc2, sp2, kc2 = _run(w, plan, inputs, dev, order)
    for n, ((o1, i1, e1), (o2, i2, e2)) in enumerate(zip(r1, r2)):
        assert _same_bits(i1, i2), f"score_inc differs between runs at step {n}"
        assert torch.equal(e1, e2), f"evicted slots differ between runs at step {n}"
        assert _same_bits(o1, o2), f"attention output differs between runs at step {n}"
    assert _same_bits(sc1, sc2) and torch.equal(sp1, sp2) and _same_bits(kc1, kc2)
