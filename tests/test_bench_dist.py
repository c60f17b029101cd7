"""The multi-process path of bench.py on CPU (gloo, world size 2): each rank runs its
own replica, timing is the max over ranks, only rank 0 reports."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    r, w, local = bench.dist_setup(world)
    assert (r, w, local) == (rank, world, rank)
    bench.barrier(w)
    t = bench.max_over_ranks(10.0 + rank, w)
    out[rank] = t
    import torch.distributed as dist
    dist.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
    assert dict(out) == {0: 11.0, 1: 11.0}


def test_reference_arm_nonzero_rank_exits_quietly(capsys, monkeypatch):
    import bench
    monkeypatch.setenv("WORLD_SIZE", "1")
    monkeypatch.setenv("RANK", "0")
    # rank 1 of 2 must print nothing and not run the oracle: simulate with a fake setup
    monkeypatch.setattr(bench, "dist_setup", lambda n: (1, 2, 1))

    class A:
        gpus, steps, warmup, ref_budget = 2, 1, 3, 1.0
    assert bench.run_reference(A, bench.wl.WORKLOADS["tiny"]) == 0
    assert capsys.readouterr().out == ""


def test_flop_accounting():
    import bench
    w = bench.wl.WORKLOADS["llama8b_32k"]
    pre, chunks = bench.step_flops(w)
    assert len(chunks) == 56
    assert abs(chunks[0] - 4 * 32 * 128 * 512 * (4096 + 256.5)) < 1
    assert abs(pre - 4 * 32 * 128 * 4096 * (4096 + 1) / 2) < 1


def test_launch_and_byte_accounting():
    """gpu_launches counts this library's kernels per chunk; decode bytes are
    the K and V rows read once (8-bit rows: d codes + a 4-byte scale)."""
    import bench
    lpc = bench.launches_per_chunk
    assert lpc(512, 4096) == 3                      # SDPA + column-sum reduction + update
    assert lpc(256, 2048) == 2                      # two row tiles per head: no reduction
    assert lpc(512, 4096, "paper") == 4             # evict-insert + SDPA + reduction + scores_add
    assert lpc(1, 4096) == 3                        # split + combine + update
    assert lpc(1, 4096, "paper") == 4
    assert lpc(1, 4096, "chunk", 16, 16) == 2       # q_g > 8: the chunk kernel
    assert lpc(512, 4096, "chunk", 8) == 5          # + read-back + quantising scatter
    assert lpc(4096, 4096, "chunk", 8) == 5         # the prefill
    assert lpc(512, 4096, "paper", 8) == 6
    assert lpc(1, 4096, "chunk", 8) == 4            # the decode kernels read the codes
    assert lpc(1, 4096, "paper", 8) == 5
    assert lpc(1, 4096, "chunk", 8, 16) == 4        # q_g > 8: read-back + chunk kernel
    w = bench.wl.WORKLOADS["decode_64k"]
    assert bench.decode_kv_bytes(w) == 2 * 8 * 8 * 65536 * 256
    assert bench.decode_kv_bytes(w, 8) == 2 * 8 * 8 * 65536 * 132
