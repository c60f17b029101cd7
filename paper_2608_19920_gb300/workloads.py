"""Seeded synthetic inputs shaped like the paper's long-context workloads.

This module only draws random numbers and rounds them to bf16; it contains
none of the attention or eviction arithmetic, so that the CUDA path and the
float64 oracle can both consume its output without sharing any method code.

The paper evaluates on Helmet / LongBench V2 prompts run through Qwen3-4B
(§4), which are not available here.  Gaussian Q/K/V with planted heavy hitters
stand in for them: a fixed random unit vector ``u`` is added to every query,
and the keys of a few "sink" positions at the start of the sequence (plus a
small random fraction of all positions) are shifted along ``u``, so those keys
collect more attention mass than the rest, which is what H2O's score (§3.1.1,
Eq. 3) is designed to pick up.

Recipe (identical for every caller):

* Each sequence ``b`` has its own streams: ``SeedSequence([seed, b, tag])``
  with ``tag = 2**20`` for ``u``, ``2**20 + 1`` for the heavy set, and the
  block index ``kb`` for the tokens of positions ``[256 kb, 256 kb + 256)``.
  Token blocks are therefore independent: any range can be generated alone.
* Per block: Q ``(Hq, 256, d)``, then K ``(Hkv, 256, d)``, then V, i.i.d.
  N(0, 1) in float32, in that draw order.
* ``q_scale``: Q is multiplied by ``d**-0.5`` (workloads 2-5), then ``u`` is
  added to every query row.
* Heavy positions: the first ``n_sink`` positions plus ``round(frac * T)``
  positions drawn uniformly without replacement from ``[0, T)``; their keys get
  ``+ shift * u`` (every KV head).
* Every value is finally rounded to bf16 (round to nearest even), so both
  sides of a comparison start from identical bits.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

BLOCK = 256
_TAG_U = 1 << 20
_TAG_HEAVY = (1 << 20) + 1
_TAG_SHIFT = (1 << 20) + 2


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    B: int
    Hq: int
    Hkv: int
    d: int
    S: int          # chunk size
    M: int          # cache budget (slots per (b, kv-head))
    W: int          # recent window protected from eviction
    T: int          # tokens per sequence
    q_scale: bool   # multiply Q by d**-0.5 before adding u
    n_sink: tuple   # (lo, hi) inclusive range for the number of sink positions
    heavy_frac: float
    shift: tuple    # (lo, hi) range of the key shift along u
    per_seq_seed: bool = False
    seed: int = 0

    @property
    def q_g(self) -> int:
        return self.Hq // self.Hkv

    @property
    def n_chunks(self) -> int:
        """Chunks after the prefill of M tokens (ragged last chunk counted)."""
        return -(-(self.T - self.M) // self.S) if self.T > self.M else 0

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


# The five workload shapes.  Sizes are those of a Llama-3-8B / Qwen-like
# attention layer at long context; the paper's own runs use a cache of 32768
# slots and chunks of 1024 or 2048 tokens (§4).
WORKLOADS = {
    "tiny": Workload("tiny", B=1, Hq=4, Hkv=2, d=64, S=32, M=256, W=32, T=1024,
                     q_scale=False, n_sink=(3, 3), heavy_frac=0.0, shift=(2.0, 2.0)),
    "llama8b_32k": Workload("llama8b_32k", B=1, Hq=32, Hkv=8, d=128, S=512, M=4096, W=512,
                            T=32768, q_scale=True, n_sink=(8, 8), heavy_frac=0.01,
                            shift=(2.0, 2.0)),
    "long_128k": Workload("long_128k", B=1, Hq=28, Hkv=4, d=128, S=1024, M=8192, W=1024,
                          T=131072, q_scale=True, n_sink=(4, 4), heavy_frac=0.005,
                          shift=(2.0, 2.0)),
    "batched_16k": Workload("batched_16k", B=4, Hq=32, Hkv=8, d=128, S=256, M=2048, W=256,
                            T=16384, q_scale=True, n_sink=(4, 16), heavy_frac=0.0,
                            shift=(1.0, 3.0), per_seq_seed=True),
    "decode_4k": Workload("decode_4k", B=8, Hq=32, Hkv=8, d=128, S=1, M=4096, W=64,
                          T=4096 + 4096, q_scale=True, n_sink=(8, 8), heavy_frac=0.01,
                          shift=(2.0, 2.0)),
    "decode_16k": Workload("decode_16k", B=8, Hq=32, Hkv=8, d=128, S=1, M=16384, W=64,
                           T=16384 + 4096, q_scale=True, n_sink=(8, 8), heavy_frac=0.01,
                           shift=(2.0, 2.0)),
    "decode_64k": Workload("decode_64k", B=8, Hq=32, Hkv=8, d=128, S=1, M=65536, W=64,
                           T=65536 + 4096, q_scale=True, n_sink=(8, 8), heavy_frac=0.01,
                           shift=(2.0, 2.0)),
}


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns float32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = ((u >> 16) & 1) + np.uint32(0x7FFF)
    r = ((u + bias) & np.uint32(0xFFFF0000)).view(np.float32)
    return r


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of float32 values that are already bf16-representable."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    return (u >> 16).astype(np.uint16)


def bits_to_f32(b: np.ndarray) -> np.ndarray:
    """float32 values of bf16 bit patterns."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def _seq_seed(w: Workload, b: int) -> int:
    return w.seed + b if w.per_seq_seed else w.seed


def _u(w: Workload, b: int) -> np.ndarray:
    rng = np.random.default_rng(np.random.SeedSequence([_seq_seed(w, b), b, _TAG_U]))
    u = rng.standard_normal(w.d)
    return (u / np.linalg.norm(u)).astype(np.float32)


def heavy_positions(w: Workload, b: int) -> np.ndarray:
    """Sorted positions whose keys are shifted along u for sequence b."""
    rng = np.random.default_rng(np.random.SeedSequence([_seq_seed(w, b), b, _TAG_HEAVY]))
    lo, hi = w.n_sink
    n_sink = int(rng.integers(lo, hi + 1))
    n_rand = int(round(w.heavy_frac * w.T))
    rand = rng.choice(w.T, size=n_rand, replace=False) if n_rand else np.zeros(0, np.int64)
    return np.unique(np.concatenate([np.arange(min(n_sink, w.T)), rand]).astype(np.int64))


def key_shift(w: Workload, b: int) -> float:
    lo, hi = w.shift
    if lo == hi:
        return float(lo)
    rng = np.random.default_rng(np.random.SeedSequence([_seq_seed(w, b), b, _TAG_SHIFT]))
    return float(rng.uniform(lo, hi))


def tokens(w: Workload, b: int, t0: int, t1: int):
    """q (Hq, n, d), k (Hkv, n, d), v (Hkv, n, d) for positions [t0, t1) of sequence b.

    float32 arrays holding bf16-representable values.
    """
    assert 0 <= t0 <= t1 <= w.T
    n = t1 - t0
    q = np.empty((w.Hq, n, w.d), np.float32)
    k = np.empty((w.Hkv, n, w.d), np.float32)
    v = np.empty((w.Hkv, n, w.d), np.float32)
    if n == 0:
        return q, k, v
    seed = _seq_seed(w, b)
    for kb in range(t0 // BLOCK, (t1 - 1) // BLOCK + 1):
        rng = np.random.default_rng(np.random.SeedSequence([seed, b, kb]))
        bq = rng.standard_normal((w.Hq, BLOCK, w.d), dtype=np.float32)
        bk = rng.standard_normal((w.Hkv, BLOCK, w.d), dtype=np.float32)
        bv = rng.standard_normal((w.Hkv, BLOCK, w.d), dtype=np.float32)
        lo = max(t0, kb * BLOCK)
        hi = min(t1, (kb + 1) * BLOCK)
        q[:, lo - t0:hi - t0] = bq[:, lo - kb * BLOCK:hi - kb * BLOCK]
        k[:, lo - t0:hi - t0] = bk[:, lo - kb * BLOCK:hi - kb * BLOCK]
        v[:, lo - t0:hi - t0] = bv[:, lo - kb * BLOCK:hi - kb * BLOCK]
    u = _u(w, b)
    if w.q_scale:
        q *= np.float32(1.0 / math.sqrt(w.d))
    q += u
    heavy = heavy_positions(w, b)
    sel = heavy[(heavy >= t0) & (heavy < t1)] - t0
    if sel.size:
        k[:, sel, :] += np.float32(key_shift(w, b)) * u
    return round_bf16(q), round_bf16(k), round_bf16(v)


def batch_tokens(w: Workload, t0: int, t1: int):
    """q (B, Hq, n, d), k (B, Hkv, n, d), v (B, Hkv, n, d) for positions [t0, t1)."""
    qs, ks, vs = zip(*(tokens(w, b, t0, t1) for b in range(w.B)))
    return np.stack(qs), np.stack(ks), np.stack(vs)


def random_state(rng: np.random.Generator, B: int, Hkv: int, M: int, d: int, *,
                 pos0: int, n_empty: int = 0, int_scores: bool = False):
    """A plausible mid-sequence cache state for unit tests.

    Occupied slots hold distinct token positions below ``pos0`` in shuffled
    order (evictions make them non-monotonic, §3.1); ``n_empty`` randomly
    chosen slots per (b, kv-head) are empty (position -1).  Scores are
    non-negative (sums of attention weights); ``int_scores`` makes them small
    integers so that ties are exact.
    """
    assert pos0 >= M - n_empty
    slot_pos = np.empty((B, Hkv, M), np.int32)
    for b in range(B):
        for h in range(Hkv):
            pos = rng.choice(pos0, size=M - n_empty, replace=False) if pos0 else np.zeros(0)
            full = np.concatenate([pos, -np.ones(n_empty)]).astype(np.int32)
            slot_pos[b, h] = rng.permutation(full)
    if int_scores:
        scores = rng.integers(0, 6, size=(B, Hkv, M)).astype(np.float32)
    else:
        scores = (rng.gamma(0.5, 2.0, size=(B, Hkv, M))).astype(np.float32)
    scores[slot_pos < 0] = 0.0
    k_cache = round_bf16(rng.standard_normal((B, Hkv, M, d), dtype=np.float32))
    v_cache = round_bf16(rng.standard_normal((B, Hkv, M, d), dtype=np.float32))
    k_cache[slot_pos < 0] = 0.0
    v_cache[slot_pos < 0] = 0.0
    return dict(slot_pos=slot_pos, scores=scores, k_cache=k_cache, v_cache=v_cache)
