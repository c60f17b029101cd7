"""Benchmark: H2O sparse attention over a whole long sequence on one GB300.

A step is one pass of the whole hot path over one sequence batch of the
workload: empty the cache, prefill M tokens, then every chunk of S tokens
(h2o_sdpa_chunk + h2o_update).  Default workload: one Llama-3-8B-shaped layer
(B=1, Hq=32, Hkv=8, d=128), T=32768 tokens, chunks of 512, cache of 4096 slots,
recent window 512.  Inputs are seeded synthetic bf16 tensors resident in HBM
(402 MB per step, more than the 129 MB L2, so each step streams them).  The
timed steps replay one CUDA graph of the whole step (``--no-graph``: eager).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                    [--workload NAME] [--no-e2e] [--no-cpu-baseline]

Prints one JSON line.  ``--impl reference`` times the float64 CPU oracle on a
bounded sample of the same workload instead (the reference arm).
Under torchrun every rank runs its own replica of the workload (the path has
no exchange step: batches and KV heads are independent), timing is the max
over ranks and rank 0 prints.
"""
from __future__ import annotations

import argparse
import datetime
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2608_19920_gb300 import workloads as wl  # noqa: E402

METRIC = "H2O SDPA prefill tokens/s and TFLOP/s (% of GB300 bf16 tensor peak), 1 GPU"


def chunk_flops(B, Hq, d, S, M_visible):
    """Algorithmic flops of one chunk: QK^T and PV over the visible keys only
    (M cache slots plus the causal half of the chunk's own S x S block)."""
    return 4.0 * B * Hq * d * S * (M_visible + (S + 1) / 2.0)


def step_plan(w: wl.Workload):
    """[(start, end)] of the prefill and the chunks of one sequence."""
    from paper_2608_19920_gb300.runner import chunk_bounds
    return chunk_bounds(w.T, w.M, w.S)


def visible_old(w: wl.Workload, S: int, order: str) -> int:
    """Cache slots every row of a steady-state chunk sees besides the chunk's
    own causal triangle: all M (attend, then evict), or M - S (the paper's
    order: S slots already hold the chunk)."""
    return w.M - S if order == "paper" else w.M


def step_flops(w: wl.Workload, order: str = "chunk"):
    plan = step_plan(w)
    prefill = chunk_flops(w.B, w.Hq, w.d, plan[0][1], 0)
    chunks = [chunk_flops(w.B, w.Hq, w.d, e - p, visible_old(w, e - p, order))
              for p, e in plan[1:]]
    return prefill, chunks


# dram__bytes_read.sum + dram__bytes_write.sum of one steady-state llama8b_32k
# chunk launch of the current SDPA kernel, from the ncu capture summarised in
# profiles/sdpa_chunk_kernel_llama8b_32k.md; None whenever the kernel has
# changed since that capture.
SDPA_DRAM_BYTES = 23.3321e6


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return dict(bf16=p.get("bf16_tflops", 1896.2), bf16_sus=p.get("bf16_tflops_sustained", 1698.6),
                    hbm=p.get("hbm_gbs", 6775.9), source="measured")
    return dict(bf16=1900.0, bf16_sus=1700.0, hbm=6800.0, source="fallback")


# ---------------------------------------------------------------- clocks --
class ClockSampler:
    """nvidia-smi clocks / throttle reasons, sampled every 10 ms; only samples
    whose timestamps fall inside [mark_start, mark_end] are summarised."""
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.file = None
        self.t_start = self.t_end = None

    def __enter__(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "10"],
                stdout=self.file, stderr=subprocess.DEVNULL)
            # sampling must be running before the timed region starts
            deadline = time.time() + 5.0
            while time.time() < deadline and os.path.getsize(self.file.name) == 0:
                time.sleep(0.02)
        except (OSError, FileNotFoundError):
            self.proc = None
        return self

    def mark_start(self):
        self.t_start = time.time()

    def mark_end(self):
        self.t_end = time.time()

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.05)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    @staticmethod
    def _stamp(x):
        try:
            return datetime.datetime.strptime(x, "%Y/%m/%d %H:%M:%S.%f").timestamp()
        except ValueError:
            return None

    def summary(self):
        if self.proc is None or self.file is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.file.flush()
        rows = []
        with open(self.file.name) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) >= 10:
                    rows.append(parts)
        os.unlink(self.file.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        inside = []
        if self.t_start is not None and self.t_end is not None:
            for r in rows:
                t = self._stamp(r[0])
                if t is not None and self.t_start <= t <= self.t_end:
                    inside.append(r)
        note = None
        if not inside:
            # timed region shorter than the sampling period: nearest sample
            mid = 0.5 * ((self.t_start or 0.0) + (self.t_end or 0.0))
            inside = [min(rows, key=lambda r: abs((self._stamp(r[0]) or 0.0) - mid))]
            note = "no sample inside the timed region; nearest sample used"

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(r[2]) for r in inside if num(r[2]) is not None]
        mx = [num(r[3]) for r in inside if num(r[3]) is not None]
        pw = [num(r[4]) for r in inside if num(r[4]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i in range(4) if r[6 + i].lower() == "active"})
        out = {"sm_mhz": statistics.median(sm) if sm else None,
               "sm_max_mhz": max(mx) if mx else None,
               "power_w": statistics.median(pw) if pw else None,
               "samples": len(inside) if note is None else 0, "reasons": reasons}
        if note:
            out["note"] = note
        return out


# ------------------------------------------------------------ distributed --
def dist_setup(n_gpus):
    """(rank, world, local_rank); initialises a gloo group for timing under torchrun."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
        dist.init_process_group("gloo", rank=rank, world_size=world)
    return rank, world, local


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


# ---------------------------------------------------------- CPU baseline --
def oracle_sample(w: wl.Workload, budget_s: float = 12.0, max_chunks: int = 8,
                  kv_bits: int = 16):
    """Times the float64 oracle on chunk steps of the workload (cache full).

    Sample: starting from a full cache (random state of the right shape), the
    oracle runs chunk steps (sparse SDPA + update; with ``kv_bits`` 8 their
    8-bit buffer forms) until ``budget_s`` seconds or ``max_chunks`` chunks;
    returns tokens/s and a description."""
    from oracle import quantize_rows, sdpa_chunk, sdpa_chunk_q8, update, update_q8
    rng = np.random.default_rng(0)
    p0 = w.M + w.S  # a position in the steady state
    st = wl.random_state(rng, w.B, w.Hkv, w.M, w.d, pos0=p0)
    if kv_bits == 8:
        st["k_codes"], st["k_scales"] = quantize_rows(st["k_cache"])
        st["v_codes"], st["v_scales"] = quantize_rows(st["v_cache"])
    n, t_total = 0, 0.0
    while n < max_chunks and t_total < budget_s:
        p = p0 + n * w.S
        if p + w.S > w.T:
            break
        q, k, v = wl.batch_tokens(w, p, p + w.S)
        t0 = time.perf_counter()
        if kv_bits == 8:
            buf = [st[x] for x in ("k_codes", "k_scales", "v_codes", "v_scales")]
            _, inc, _ = sdpa_chunk_q8(q, *buf, k, v, st["slot_pos"], p)
            r = update_q8(st["scores"], st["slot_pos"], inc, k, v, *buf, p, w.W, "fp64")
        else:
            _, inc, _ = sdpa_chunk(q, st["k_cache"], st["v_cache"], k, v, st["slot_pos"], p)
            r = update(st["scores"], st["slot_pos"], inc, k, v, st["k_cache"], st["v_cache"], p,
                       w.W, "fp64")
        t_total += time.perf_counter() - t0
        st = {x: r[x] for x in r if x != "evict_idx"}
        n += 1
    tokens = n * w.S * w.B
    return dict(value=tokens / t_total, unit="tokens/s", cores=os.cpu_count(), kind="oracle",
                seconds=t_total,
                sample=(f"{n} steady-state chunk steps ({w.S} tokens x B={w.B}, cache of {w.M} "
                        f"slots full{', 8-bit K/V buffers' if kv_bits == 8 else ''}) of the "
                        f"{w.name} workload, float64 NumPy oracle"))


def run_reference(args, w):
    rank, world, _ = dist_setup(args.gpus)
    if rank != 0:
        return 0
    times = []
    tokens = 0
    for i in range(args.warmup + args.steps):
        r = oracle_sample(w, budget_s=args.ref_budget, max_chunks=1, kv_bits=args.kv_bits)
        if i >= args.warmup:
            times.append(r["seconds"])
            tokens += w.S * w.B
    value = tokens / sum(times)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * sum(times) / len(times), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "Hq": w.Hq, "Hkv": w.Hkv, "d": w.d,
                       "T": w.T, "S": w.S, "M": w.M, "W": w.W,
                       "kv_buffers": ("int8 codes + fp32 row scales" if args.kv_bits == 8
                                      else "bf16"),
                       "step": "one steady-state chunk step per step (CPU sample)"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": os.cpu_count(),
                             "kind": "oracle",
                             "sample": f"one {w.S}-token chunk step per step, cache of {w.M} full"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return 0


# ------------------------------------------------------------------ ours --
def make_inputs(w, dev, pinned=False):
    """Chunk-major bf16 inputs of one sequence batch: a list of (q, k, v) per chunk."""
    import torch
    chunks = []
    for p, e in step_plan(w):
        q, k, v = wl.batch_tokens(w, p, e)
        ts = []
        for x in (q, k, v):
            t = torch.from_numpy(x).to(torch.bfloat16)
            ts.append(t.pin_memory() if pinned else t.to(dev))
        chunks.append(tuple(ts))
    return chunks


def run_ours(args, w):
    import torch
    from paper_2608_19920_gb300 import H2OLayer, h2o_device_errors
    from paper_2608_19920_gb300 import build as build_mod

    rank, world, local = dist_setup(args.gpus)
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    build_mod.build()
    plan = step_plan(w)
    pre_flops, chunk_fl = step_flops(w, args.order)
    total_flops = pre_flops + sum(chunk_fl)
    tokens_per_step = w.B * w.T

    inputs = make_inputs(w, dev)
    outs = [torch.empty((w.B, w.Hq, e - p, w.d), dtype=torch.bfloat16, device=dev)
            for p, e in plan]
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev, keep_evictions=True,
                     order=args.order, kv_bits=args.kv_bits)
    stream = torch.cuda.current_stream()
    n_chunks = len(plan) - 1
    # one pair of events per entry of the plan: [0] the prefill, then each chunk
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(len(plan))]

    def one_step(record=False):
        layer.reset()
        for i, ((p, e), (q, k, v)) in enumerate(zip(plan, inputs)):
            if record:
                ev[i][0].record(stream)
                layer.step(q, k, v, p, out=outs[i])
                ev[i][1].record(stream)
            else:
                layer.step(q, k, v, p, out=outs[i])

    for _ in range(args.warmup):
        one_step()
    torch.cuda.synchronize()
    if h2o_device_errors() != 0:
        raise SystemExit("device-side error during warm-up")
    # chunk-step durations (sdpa + update), eager launches, one step
    one_step(record=True)
    torch.cuda.synchronize()
    entry_ms = [a.elapsed_time(b) for a, b in ev]
    prefill_ms, chunk_step_ms = entry_ms[0], entry_ms[1:]
    # The whole step (cache reset, prefill, every chunk's two calls) is
    # captured once as a CUDA graph and replayed: every kernel of the step
    # runs on every replay, without the host's launch gaps between them.
    graph = None
    if args.graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            one_step()
        graph.replay()
        torch.cuda.synchronize()
        if h2o_device_errors() != 0:
            raise SystemExit("device-side error in the captured step")

    # ---- timed region: K steps, inputs resident in HBM
    barrier(world)
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clk:
        clk.mark_start()
        t0.record(stream)
        for s in range(args.steps):
            if graph is not None:
                graph.replay()
            else:
                one_step()
        t1.record(stream)
        torch.cuda.synchronize()
        clk.mark_end()
    elapsed_ms = t0.elapsed_time(t1)
    barrier(world)
    elapsed_ms = max_over_ranks(elapsed_ms, world)
    step_ms = elapsed_ms / args.steps
    clocks = clk.summary()
    if h2o_device_errors() != 0:
        raise SystemExit("device-side error during the timed region")

    # ---- dominant kernel: the chunk SDPA alone, timed on the same stream
    kern = time_sdpa_kernel(w, layer, inputs, plan, stream, reps=args.roofline_reps)

    value = tokens_per_step * world / (step_ms / 1e3)
    in_bytes = sum(x.numel() * x.element_size() for c in inputs for x in c)
    pk = peaks()
    alg_tflops = total_flops / (step_ms / 1e3) / 1e12
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": step_ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded Gaussian Q/K/V with planted heavy-hitter keys)",
        "config": {"workload": w.name, "B": w.B, "Hq": w.Hq, "Hkv": w.Hkv, "d": w.d, "T": w.T,
                   "S": w.S, "M": w.M, "W": w.W, "tokens_per_step": tokens_per_step,
                   "chunks_per_step": n_chunks,
                   "l2": f"inputs larger than L2 ({in_bytes / 1e6:.0f} MB per step)"
                         if in_bytes > 129e6 else f"{in_bytes / 1e6:.0f} MB of inputs per step",
                   "launch": "CUDA graph of the whole step" if args.graph else "eager",
                   "order": args.order,
                   "kv_buffers": "int8 codes + fp32 row scales" if args.kv_bits == 8 else "bf16",
                   "parallelism": f"replicas x{world}"},
        "tflops": alg_tflops,
        "tflops_frac_of_peak": alg_tflops / pk["bf16_sus"],
        "chunk_step_ms_median": statistics.median(chunk_step_ms) if chunk_step_ms else None,
        "prefill": {"tokens": w.B * (plan[0][1] - plan[0][0]), "ms": prefill_ms,
                    "tokens_per_s": w.B * (plan[0][1] - plan[0][0]) / (prefill_ms / 1e3),
                    "tflops": pre_flops / (prefill_ms / 1e3) / 1e12,
                    "timing": "eager SDPA + update of the prefill, one step, L2 warm"}
                   if w.M > 0 else None,
        "gpu_launches": args.steps * sum(launches_per_chunk(e - p, w.M, args.order,
                                                            args.kv_bits, w.Hq // w.Hkv)
                                         for p, e in plan),
        "clocks": clocks,
    }
    # the chunk SDPA is timed on its own (launch after launch, L2 flushed in
    # between): its denominator is the burst peak; the sustained one is given
    # alongside
    traffic = args.traffic if args.traffic is not None else (
        SDPA_DRAM_BYTES if w.name == "llama8b_32k" and args.order == "chunk" and
        args.kv_bits == 16 else None)
    if w.S == 1:
        # decode: K and V read once per step, HBM bound
        line["roofline"] = {
            "bound": "hbm",
            "kernel": "decode_split_kernel" + ("<8-bit rows>" if args.kv_bits == 8 else "") +
                      " + decode_combine_kernel (one step)",
            "achieved": kern["gbs"], "peak": pk["hbm"], "unit": "GB/s",
            "frac": kern["gbs"] / pk["hbm"], "traffic": traffic,
            "peak_source": f"{pk['source']} HBM copy bandwidth",
            "avg_launch_us": kern["avg_us"], "median_launch_us": kern["median_us"],
            "launches_timed": kern["launches"], "bytes_per_launch": kern["bytes"],
            "clocks": kern["clocks"],
        }
    else:
        line["roofline"] = {
            "bound": "tensor",
            "kernel": ("kv_dequantize_kernel + " if args.kv_bits == 8 else "") +
                      "sdpa_chunk_kernel<128,pair> (steady-state chunk" +
                      (", cache only)" if args.order == "paper" else ")"),
            "achieved": kern["alg_tflops"], "peak": pk["bf16"], "unit": "TFLOP/s",
            "frac": kern["alg_tflops"] / pk["bf16"], "traffic": traffic,
            "peak_source": f"{pk['source']} bf16 dense, burst",
            "frac_of_sustained": kern["alg_tflops"] / pk["bf16_sus"],
            "avg_launch_us": kern["avg_us"], "median_launch_us": kern["median_us"],
            "launches_timed": kern["launches"], "flops_per_launch": kern["flops"],
            "executed_tflops": kern["alg_tflops"] * kern["exec_ratio"],
            "clocks": kern["clocks"],
        }
    if args.e2e:
        line["e2e"] = run_e2e(w, layer, plan, outs, dev, args, world)
    if args.cpu_baseline and rank == 0 and world == 1:
        line["cpu_baseline"] = oracle_sample(w, kv_bits=args.kv_bits)
    if rank == 0:
        print(json.dumps(line))
    return 0


def time_sdpa_kernel(w, layer, inputs, plan, stream, reps, idx=None, prepare=True):
    """Average duration of the steady-state chunk SDPA launch (CUDA events)."""
    import torch
    from paper_2608_19920_gb300 import (h2o_evict_insert, h2o_evict_insert_q8, h2o_sdpa_cache,
                                       h2o_sdpa_cache_q8, h2o_sdpa_chunk, h2o_sdpa_chunk_q8)
    idx = len(plan) // 2 if idx is None else idx
    if prepare and idx > 0:
        # the cache as the sequence leaves it just before chunk idx
        layer.reset()
        for i in range(idx):
            layer.step(*inputs[i], plan[i][0])
    p, e = plan[idx]
    q, k, v = inputs[idx]
    out = torch.empty((w.B, w.Hq, e - p, w.d), dtype=torch.bfloat16, device=q.device)
    inc, _, ws = layer._buf(e - p)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=q.device)
    clean = torch.ones(256 * 1024 * 1024 // 4, dtype=torch.float32, device=q.device)

    q8 = layer.kv_bits == 8
    buf = (layer.k_codes, layer.k_scales, layer.v_codes, layer.v_scales) if q8 else None

    def call():
        if layer.order == "paper":  # the cache already holds the chunk (filled by the caller)
            if q8:
                h2o_sdpa_cache_q8(q, *buf, layer.slot_pos, p, out=out, score_inc=inc,
                                  workspace=ws)
            else:
                h2o_sdpa_cache(q, layer.k_cache, layer.v_cache, layer.slot_pos, p, out=out,
                               score_inc=inc, workspace=ws)
        elif q8:
            h2o_sdpa_chunk_q8(q, *buf, k, v, layer.slot_pos, p, out=out, score_inc=inc,
                              workspace=ws)
        else:
            h2o_sdpa_chunk(q, layer.k_cache, layer.v_cache, k, v, layer.slot_pos, p, out=out,
                           score_inc=inc, workspace=ws)

    if layer.order == "paper" and q8:
        h2o_evict_insert_q8(layer.scores, layer.slot_pos, k, v, *buf, p, layer.W,
                            policy=layer.policy, Hq=layer.Hq)
    elif layer.order == "paper":
        h2o_evict_insert(layer.scores, layer.slot_pos, k, v, layer.k_cache, layer.v_cache, p,
                         layer.W, policy=layer.policy, Hq=layer.Hq)
    # the call is replayed from a CUDA graph, as in the timed steps
    call()
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        call()
    evs = []
    with ClockSampler(torch.cuda.current_device()) as clk:
        clk.mark_start()
        for _ in range(reps + 2):
            # Evict the previous launch's data from L2 by writing a buffer
            # twice its size, then read another one so that the write-back of
            # those dirty lines happens here, not inside the timed launch.
            flush.zero_()
            clean.sum()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            graph.replay()
            b.record(stream)
            evs.append((a, b))
        torch.cuda.synchronize()
        clk.mark_end()
    times = [a.elapsed_time(b) for a, b in evs][2:]
    avg_ms = sum(times) / len(times)
    flops = chunk_flops(w.B, w.Hq, w.d, e - p, visible_old(w, e - p, layer.order))
    exec_flops = executed_mma_flops(w, e - p)
    kv_bytes = decode_kv_bytes(w, layer.kv_bits)
    return dict(avg_us=avg_ms * 1e3, median_us=statistics.median(times) * 1e3, launches=len(times),
                flops=flops, alg_tflops=flops / (avg_ms / 1e3) / 1e12,
                exec_ratio=exec_flops / flops, bytes=kv_bytes, gbs=kv_bytes / (avg_ms / 1e3) / 1e9,
                clocks=clk.summary())


def decode_kv_bytes(w, kv_bits: int = 16):
    """Algorithmic bytes of one decode step: every cache K and V row read once
    (8-bit buffers: d codes and a 4-byte scale per row)."""
    row = w.d * 2 if kv_bits == 16 else w.d + 4
    return 2.0 * w.B * w.Hkv * w.M * row


def launches_per_chunk(S, M, order="chunk", kv_bits=16, qg=4):
    """Kernels of this library one chunk launches: the SDPA (split + combine
    when S = 1 and a cache exists) and the update (the paper's order: the
    eviction-insert, the SDPA and the score addition); 8-bit buffers add the
    quantising scatter after the update and, where the chunk kernel runs, the
    read-back before it (the decode kernels read the codes themselves).  With
    three or more 128-row tiles per query head (S > 256) the chunk kernel is
    followed by the kernel that adds its per-tile column sums in order."""
    decode = S == 1 and M > 0 and qg <= 8
    sdpa = 2 if decode else (2 if (S + 127) // 128 >= 3 and S > 128 else 1)
    q8 = (1 + (0 if decode or M == 0 else 1)) if kv_bits == 8 else 0
    return sdpa + (2 if order == "paper" else 1) + q8


def executed_mma_flops(w, S):
    """Tensor-core flops the two-pass kernel issues for one chunk with a full
    cache: per visited 128x128 key tile, Q K^T twice and P V once."""
    tile = 2.0 * 128 * 128 * w.d
    n_cache = -(-w.M // 128)
    total = 0.0
    if S > 128:
        for i0 in range(0, S, 128):
            total += w.q_g * (n_cache + i0 // 128 + 1)
    else:
        per_tile = 128 // (-(-S // 32) * 32)
        total += -(-w.q_g // per_tile) * (n_cache + 1)
    return 3 * tile * total * w.B * w.Hkv


def run_e2e(w, layer, plan, outs, dev, args, world):
    """Same metric through the public API from pinned host buffers: every step
    copies the whole sequence's inputs host->device and every chunk's output
    back.  The copies overlap the compute, as a caller would arrange them: the
    next chunk's inputs go up on one copy stream while a chunk computes, each
    output comes back on a second one as soon as its chunk is done."""
    import torch
    host_in = make_inputs(w, dev, pinned=True)
    dev_in = [tuple(torch.empty_like(x, device=dev) for x in c) for c in host_in]
    host_out = [torch.empty(o.shape, dtype=o.dtype, pin_memory=True) for o in outs]
    h2d = sum(x.numel() * x.element_size() for c in host_in for x in c)
    d2h = sum(o.numel() * o.element_size() for o in outs)
    stream = torch.cuda.current_stream()
    s_in, s_out = torch.cuda.Stream(device=dev), torch.cuda.Stream(device=dev)
    n_c = len(plan)
    ev_in = [torch.cuda.Event() for _ in range(n_c)]
    ev_done = [torch.cuda.Event() for _ in range(n_c)]
    ev_out = torch.cuda.Event()

    def upload(i):
        with torch.cuda.stream(s_in):
            for a, b in zip(dev_in[i], host_in[i]):
                a.copy_(b, non_blocking=True)
            ev_in[i].record(s_in)

    ev_start = torch.cuda.Event()

    def step():
        # Fork the copy streams off the compute stream and join them back at
        # the end, so that a step is self-contained (and capturable): the
        # previous step's compute and read-backs are done with the buffers.
        ev_start.record(stream)
        s_in.wait_event(ev_start)
        s_out.wait_event(ev_start)
        layer.reset()
        upload(0)
        for i, ((p, e), dx, o, ho) in enumerate(zip(plan, dev_in, outs, host_out)):
            if i + 1 < n_c:
                upload(i + 1)
            stream.wait_event(ev_in[i])
            layer.step(dx[0], dx[1], dx[2], p, out=o)
            ev_done[i].record(stream)
            s_out.wait_event(ev_done[i])
            with torch.cuda.stream(s_out):
                ho.copy_(o, non_blocking=True)
        ev_out.record(s_out)
        stream.wait_event(ev_out)  # the read-backs are part of the step

    for _ in range(2):
        step()
    torch.cuda.synchronize()
    # As for the resident number, the whole step is replayed from a CUDA
    # graph: its copy nodes move every step's inputs from pinned host memory
    # and every chunk's output back on each replay.
    graph = None
    if args.graph:
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            step()
        graph.replay()
        torch.cuda.synchronize()
    barrier(world)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    n = max(2, args.steps // 2)
    t0.record(stream)
    for _ in range(n):
        if graph is not None:
            graph.replay()
        else:
            step()
    t1.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(t0.elapsed_time(t1) / n, world)
    return {"value": w.B * w.T * world / (ms / 1e3), "unit": "tokens/s",
            "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": ms,
            "copies": "overlapped with the compute (two copy streams)",
            "launch": "CUDA graph of the whole step, copies included" if args.graph else "eager"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama8b_32k", choices=sorted(wl.WORKLOADS))
    ap.add_argument("--no-e2e", dest="e2e", action="store_false")
    ap.add_argument("--order", default="chunk", choices=["chunk", "paper"],
                    help="chunk step order: attend then evict (default), or the paper's "
                         "evict-and-write first")
    ap.add_argument("--kv-bits", type=int, default=16, choices=[16, 8],
                    help="cache buffers: bf16 rows (default) or int8 codes with a float32 "
                         "scale per row")
    ap.add_argument("--no-graph", dest="graph", action="store_false",
                    help="launch the timed steps eagerly instead of replaying a CUDA graph")
    ap.add_argument("--no-cpu-baseline", dest="cpu_baseline", action="store_false")
    ap.add_argument("--traffic", type=float, default=None,
                    help="DRAM bytes per launch of the dominant kernel from an ncu capture")
    ap.add_argument("--ref-budget", type=float, default=20.0)
    ap.add_argument("--mode", default="step", choices=["step", "kernel", "backward"],
                    help="kernel: only repeat the steady-state chunk SDPA launch (for profiling); "
                         "backward: time the gradient of that chunk (h2o_sdpa_chunk_backward)")
    ap.add_argument("--reps", type=int, default=5)
    ap.add_argument("--roofline-reps", type=int, default=500,
                    help="launches of the dominant kernel timed for the roofline (after 2 "
                         "untimed ones), independent of --steps")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be at least 3")
    w = wl.WORKLOADS[args.workload]
    if args.impl == "reference":
        return run_reference(args, w)
    if args.mode == "kernel":
        return run_kernel_only(args, w)
    if args.mode == "backward":
        return run_backward(args, w)
    return run_ours(args, w)


def run_kernel_only(args, w, n_fill: int = 8):
    """Fills the cache with a prefill and ``n_fill`` chunks, then launches the
    chunk after them ``--reps`` times (a small, fixed launch list for ncu)."""
    import torch
    from paper_2608_19920_gb300 import H2OLayer, build as build_mod, h2o_device_errors
    build_mod.build()
    dev = torch.device("cuda", 0)
    plan = step_plan(w)[:n_fill + 2]
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev, order=args.order,
                     kv_bits=args.kv_bits)
    ins = []
    for p, e in plan:
        ins.append(tuple(torch.from_numpy(x).to(torch.bfloat16).to(dev)
                         for x in wl.batch_tokens(w, p, e)))
    layer.reset()
    for (p, e), (q, k, v) in zip(plan[:-1], ins[:-1]):
        layer.step(q, k, v, p)
    kern = time_sdpa_kernel(w, layer, ins, plan, torch.cuda.current_stream(), reps=args.reps,
                            idx=len(plan) - 1, prepare=False)
    torch.cuda.synchronize()
    assert h2o_device_errors() == 0
    print(json.dumps({"mode": "kernel", "workload": w.name, **kern}))
    return 0


def run_backward(args, w, n_fill: int = 8):
    """Times the chunk-SDPA gradient on the chunk after a prefill and ``n_fill``
    chunks (the forward's inputs and output, a random dout), L2 flushed before
    each launch, replayed from a CUDA graph: h2o_sdpa_chunk_backward (which
    recomputes each row's log-sum-exp) and h2o_sdpa_chunk_backward_lse (given
    the forward's, from h2o_sdpa_chunk_lse)."""
    import torch
    from paper_2608_19920_gb300 import (H2OLayer, build as build_mod, h2o_backward_workspace_size,
                                       h2o_device_errors, h2o_sdpa_chunk_backward,
                                       h2o_sdpa_chunk_lse)
    from paper_2608_19920_gb300._binding import H2ODims
    build_mod.build()
    dev = torch.device("cuda", 0)
    plan = step_plan(w)[:n_fill + 2]
    layer = H2OLayer(w.B, w.Hq, w.Hkv, w.d, w.M, w.S, w.W, device=dev)
    ins = [tuple(torch.from_numpy(x).to(torch.bfloat16).to(dev) for x in wl.batch_tokens(w, p, e))
           for p, e in plan]
    layer.reset()
    for (p, e), (q, k, v) in zip(plan[:-1], ins[:-1]):
        layer.step(q, k, v, p)
    p, e = plan[-1]
    q, k, v = ins[-1]
    S = e - p
    out, _, lse = h2o_sdpa_chunk_lse(q, layer.k_cache, layer.v_cache, k, v, layer.slot_pos, p)
    dout = torch.randn(out.shape, device=dev, generator=torch.Generator(dev).manual_seed(0))
    dout = dout.to(torch.bfloat16)
    ws = torch.empty(h2o_backward_workspace_size(H2ODims(w.B, w.Hq, w.Hkv, w.d, S, w.M)),
                     dtype=torch.uint8, device=dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    clean = torch.ones(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def timed(saved):
        def call():
            h2o_sdpa_chunk_backward(q, layer.k_cache, layer.v_cache, k, v, layer.slot_pos, p, out,
                                    dout, workspace=ws, lse=lse if saved else None)

        call()
        torch.cuda.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            call()
        times = []
        for _ in range(args.reps + 2):
            flush.zero_()
            clean.sum()
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            a.record(stream)
            graph.replay()
            b.record(stream)
            torch.cuda.synchronize()
            times.append(a.elapsed_time(b))
        assert h2o_device_errors() == 0
        return sum(times[2:]) / len(times[2:])

    avg_ms = timed(False)
    avg_ms_lse = timed(True)
    # five contractions over the visible keys (Q K^T again, dout V^T, dS K,
    # dS^T Q, P^T dout): 2.5 times the forward's algorithmic flops
    flops = 2.5 * chunk_flops(w.B, w.Hq, w.d, S, w.M)
    pk = peaks()
    tf = flops / (avg_ms / 1e3) / 1e12
    tf_lse = flops / (avg_ms_lse / 1e3) / 1e12
    print(json.dumps({"mode": "backward", "workload": w.name, "S": S, "flops": flops,
                      "avg_us": avg_ms * 1e3, "alg_tflops": tf, "frac_of_bf16_peak": tf / pk["bf16"],
                      "saved_lse_avg_us": avg_ms_lse * 1e3, "saved_lse_alg_tflops": tf_lse,
                      "saved_lse_frac_of_bf16_peak": tf_lse / pk["bf16"],
                      "workspace_bytes": ws.numel()}))
    return 0


if __name__ == "__main__":
    sys.exit(main())
