"""The C-ABI library builds, loads and exports every declared symbol; host-side
argument checking returns the documented codes without touching a GPU."""
import ctypes
import os
import re

import pytest

from paper_2608_19920_gb300 import _binding as b
from paper_2608_19920_gb300 import build as build_mod

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "h2o.h")

OK, NULL, SHAPE, ALIGN, UNSUP, WORKSPACE, ARG = 0, -1, -2, -3, -4, -5, -6


@pytest.fixture(scope="module")
def lib():
    build_mod.build()
    return b.load()


def declared_symbols():
    text = open(HEADER).read()
    return set(re.findall(r"H2O_API\s+[\w\s\*]*?\b(h2o_\w+)\s*\(", text))


def test_header_declares_the_binding_exports():
    assert declared_symbols() == set(b.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_symbols():
        assert hasattr(lib, name), name
    assert lib.h2o_version() >= 100
    for code in range(-10, 1):
        assert lib.h2o_status_string(code)


def _dims(B=1, Hq=4, Hkv=2, d=64, S=32, M=256):
    return b.H2ODims(B, Hq, Hkv, d, S, M)


def _sdpa(lib, dims, ptrs=None, pos0=256, scale=0.0):
    p = ptrs or [0x1000] * 8
    vp = ctypes.c_void_p
    return lib.h2o_sdpa_chunk(ctypes.byref(dims) if dims is not None else None, pos0, scale,
                              *[vp(x) for x in p], None, 0, None)


def test_sdpa_argument_checks(lib):
    assert _sdpa(lib, None) == NULL
    assert _sdpa(lib, _dims(Hq=5, Hkv=2)) == SHAPE
    assert _sdpa(lib, _dims(S=0)) == SHAPE
    assert _sdpa(lib, _dims(M=-1)) == SHAPE
    assert _sdpa(lib, _dims(d=96)) == UNSUP
    assert _sdpa(lib, _dims(), ptrs=[0x1000] * 7 + [0]) == NULL
    assert _sdpa(lib, _dims(), ptrs=[0x1000] * 6 + [0x1004, 0x1000]) == ALIGN
    assert _sdpa(lib, _dims(), pos0=-1) == ARG
    assert _sdpa(lib, _dims(), pos0=2 ** 31 - 8) == ARG
    assert _sdpa(lib, _dims(), scale=float("inf")) == ARG
    n = ctypes.c_size_t(7)
    assert lib.h2o_workspace_size(ctypes.byref(_dims()), ctypes.byref(n)) == OK and n.value == 0
    assert lib.h2o_workspace_size(ctypes.byref(_dims(d=32)), ctypes.byref(n)) == UNSUP


def test_decode_workspace(lib):
    """S = 1 with a cache takes the split-K decode kernels, whose per-split
    partials (max, sum, d outputs per query head) live in the caller's workspace."""
    n = ctypes.c_size_t(0)
    dims = _dims(B=8, Hq=32, Hkv=8, d=128, S=1, M=65536)
    assert lib.h2o_workspace_size(ctypes.byref(dims), ctypes.byref(n)) == OK
    # 64 (b, kv head) groups x 65536 slots: splits of 1024 slots (a multiple of
    # the 128-key tiles of the d = 128 kernel, at most 1024), 64 per group,
    # 4096 work items in 27 rounds over 152 CTAs
    assert n.value == 8 * 32 * 64 * (2 + 128) * 4
    assert n.value <= 16 << 20  # fits the fixed scratch of h2o_sdpa_decode_static
    small = _dims(B=1, Hq=4, Hkv=2, d=64, S=1, M=100)
    assert lib.h2o_workspace_size(ctypes.byref(small), ctypes.byref(n)) == OK
    assert n.value == 1 * 4 * 1 * (2 + 64) * 4
    # no cache, or a GQA group above 8: the chunk kernel, no workspace
    for d_ in (_dims(S=1, M=0), _dims(Hq=16, Hkv=1, S=1, M=100)):
        assert lib.h2o_workspace_size(ctypes.byref(d_), ctypes.byref(n)) == OK and n.value == 0
    # a missing or short workspace is refused before anything runs
    vp = ctypes.c_void_p
    ptrs = [vp(0x1000)] * 8
    assert lib.h2o_sdpa_chunk(ctypes.byref(small), 100, 0.0, *ptrs, None, 0, None) == WORKSPACE
    assert lib.h2o_sdpa_chunk(ctypes.byref(small), 100, 0.0, *ptrs, vp(0x2000), 4 * 66 * 4 - 1,
                              None) == WORKSPACE
    assert lib.h2o_sdpa_chunk(ctypes.byref(small), 100, 0.0, *ptrs, vp(0x2004), 4 * 66 * 4,
                              None) == ALIGN


def test_chunk_workspace(lib):
    """With three or more 128-row tiles per query head (S > 256) the chunk
    kernel stores per-row-tile column sums in the workspace, (B, Hq, tiles,
    M + S) fp32, and a second kernel adds them in row-tile order; one or two
    tiles per head add into score_inc directly and need no workspace."""
    n = ctypes.c_size_t(0)
    for S, tiles in ((32, 0), (128, 0), (256, 0), (257, 3), (512, 4), (4096, 32)):
        dims = _dims(B=2, Hq=8, Hkv=2, d=128, S=S, M=4096)
        assert lib.h2o_workspace_size(ctypes.byref(dims), ctypes.byref(n)) == OK
        assert n.value == 2 * 8 * tiles * (4096 + S) * 4, (S, n.value)
    vp = ctypes.c_void_p
    ptrs = [vp(0x1000)] * 8
    big = _dims(B=1, Hq=4, Hkv=2, d=128, S=512, M=1024)
    need = 1 * 4 * 4 * (1024 + 512) * 4
    assert lib.h2o_sdpa_chunk(ctypes.byref(big), 2048, 0.0, *ptrs, None, 0, None) == WORKSPACE
    assert lib.h2o_sdpa_chunk(ctypes.byref(big), 2048, 0.0, *ptrs, vp(0x2000), need - 1,
                              None) == WORKSPACE
    assert lib.h2o_sdpa_chunk(ctypes.byref(big), 2048, 0.0, *ptrs, vp(0x2008), need,
                              None) == ALIGN


def _upd(lib, dims, budget=256, W=32, pos0=256, ptrs=None, evict=None):
    p = ptrs or [0x1000] * 7
    vp = ctypes.c_void_p
    return lib.h2o_update(ctypes.byref(dims), pos0, *[vp(x) for x in p], budget, W,
                          vp(evict) if evict else None, None)


def test_update_argument_checks(lib):
    assert _upd(lib, _dims(), budget=255) == ARG
    assert _upd(lib, _dims(), W=-1) == ARG
    assert _upd(lib, _dims(), W=257) == ARG
    assert _upd(lib, _dims(S=300)) == SHAPE
    assert _upd(lib, _dims(), pos0=-3) == ARG
    assert _upd(lib, _dims(), ptrs=[0x1000] * 6 + [0]) == NULL
    assert _upd(lib, _dims(), evict=0x1002) == ALIGN
    assert _upd(lib, _dims(M=0, S=1), budget=0) == SHAPE


def _upd_policy(lib, dims, policy, budget=256, W=32, pos0=256):
    vp = ctypes.c_void_p
    return lib.h2o_update_policy(ctypes.byref(dims), pos0, *[vp(0x1000)] * 7, budget, W, policy,
                                 None, None)


def test_update_policy_argument_checks(lib):
    """Unknown policy codes are rejected on the host; the other checks are shared."""
    assert _upd_policy(lib, _dims(), 3) == ARG
    assert _upd_policy(lib, _dims(), -1) == ARG
    assert _upd_policy(lib, _dims(), 1, budget=255) == ARG
    assert _upd_policy(lib, _dims(S=300), 2) == SHAPE
    assert [b.POLICY[p] for p in ("h2o", "h2o_norm", "h2o_orig")] == [0, 1, 2]


def test_binding_refuses_to_run_without_the_library(tmp_path):
    saved = b._lib
    try:
        b._lib = None
        with pytest.raises(RuntimeError, match="not built"):
            b.load(str(tmp_path / "missing.so"))
    finally:
        b._lib = saved


def test_paper_order_argument_checks(lib):
    """h2o_evict_insert / h2o_sdpa_cache / h2o_scores_add refuse bad arguments
    on the host, before any device work."""
    vp = ctypes.c_void_p
    p = vp(0x1000)
    d = _dims()
    ev = lambda dims, budget=256, W=32, pos0=256, policy=0, ptrs=None: lib.h2o_evict_insert(
        ctypes.byref(dims), pos0, *(ptrs or [p] * 6), budget, W, policy, None, None)
    assert ev(d, budget=255) == ARG
    assert ev(d, policy=3) == ARG
    assert ev(d, W=257) == ARG
    assert ev(_dims(S=300)) == SHAPE
    assert ev(d, ptrs=[p] * 5 + [vp(0)]) == NULL
    assert ev(d, ptrs=[vp(0x1004)] + [p] * 5) == ALIGN
    sc = lambda dims, ptrs=None, ws=None, wsb=0: lib.h2o_sdpa_cache(
        ctypes.byref(dims), 256, 0.0, *(ptrs or [p] * 6), ws, wsb, None)
    assert sc(_dims(M=0)) == SHAPE
    assert sc(d, ptrs=[p] * 5 + [vp(0)]) == NULL
    assert sc(d, ptrs=[vp(0x1008)] + [p] * 5) == ALIGN
    assert sc(_dims(S=1, M=100)) == WORKSPACE  # the decode kernels need their workspace
    assert lib.h2o_scores_add(ctypes.byref(_dims(M=0)), p, p, None) == SHAPE
    assert lib.h2o_scores_add(ctypes.byref(d), vp(0), p, None) == NULL
    assert lib.h2o_scores_add(ctypes.byref(d), p, vp(0x1002), None) == ALIGN


def test_replay_rows_argument_checks(lib):
    """h2o_kv_replace / h2o_kv_restore refuse bad arguments on the host."""
    vp = ctypes.c_void_p
    p = vp(0x1000)
    d = _dims()
    rep = lambda dims, ptrs, pos0=256: lib.h2o_kv_replace(ctypes.byref(dims), pos0, *ptrs, None)
    ok = [p] * 5 + [None, None, None, None]
    assert rep(_dims(M=0, S=1), ok) == SHAPE
    assert rep(_dims(S=300), ok) == SHAPE
    assert rep(d, [vp(0)] + ok[1:]) == NULL
    assert rep(d, [p] * 5 + [None, p, None, None]) == NULL   # delta_k without delta_v
    assert rep(d, [p] * 4 + [vp(0x1008)] + [None] * 4) == ALIGN
    assert rep(d, ok, pos0=-1) == ARG
    res = lambda dims, ptrs: lib.h2o_kv_restore(ctypes.byref(dims), *ptrs, None)
    assert res(d, [p, p, vp(0), None, p, p, None]) == NULL
    assert res(d, [p, p, p, None, p, vp(0x100c), None]) == ALIGN


def test_backward_argument_checks(lib):
    """h2o_sdpa_chunk_backward refuses bad arguments on the host (through the
    binding's declared argument types)."""
    vp = ctypes.c_void_p
    p = vp(0x1000)
    d = _dims()
    n = ctypes.c_size_t(0)
    assert lib.h2o_backward_workspace_size(ctypes.byref(d), ctypes.byref(n)) == OK
    # lambda and D per stacked row: B Hkv = 2 groups of q_g S = 64 rows, each
    # padded to 128
    assert n.value == 2 * 2 * 128 * 4
    bwd = lambda dims, ptrs, ws=p, wsb=n.value, pos0=256: lib.h2o_sdpa_chunk_backward(
        ctypes.byref(dims), pos0, 0.0, *ptrs, ws, wsb, None)
    ok = [p] * 13
    assert bwd(d, ok, ws=None) == WORKSPACE
    assert bwd(d, ok, wsb=n.value - 1) == WORKSPACE
    assert bwd(d, [vp(0)] + ok[1:]) == NULL
    assert bwd(d, ok[:8] + [vp(0x1004)] + ok[9:]) == ALIGN
    assert bwd(d, ok, pos0=-1) == ARG
    assert bwd(_dims(d=96), ok) == UNSUP
    # q_g S = 600000 stacked rows: more than 4096 row tiles in a group
    assert bwd(_dims(S=300000), ok, pos0=0) == UNSUP
    # the saved-lse form: the lse pointer is checked like the others
    bwl = lambda lse: lib.h2o_sdpa_chunk_backward_lse(ctypes.byref(d), 256, 0.0, *ok[:8], lse,
                                                      *ok[8:], p, n.value, None)
    assert bwl(None) == NULL
    assert bwl(vp(0x1004)) == ALIGN
    fl = lambda lse: lib.h2o_sdpa_chunk_lse(ctypes.byref(d), 256, 0.0, *[p] * 8, lse, None, 0,
                                            None)
    assert fl(None) == NULL
    assert fl(vp(0x1008)) == ALIGN


def test_selftest_limit_is_checked_on_the_host(lib):
    assert lib.h2o_selftest_bounded_wait(10, None) == ARG          # below 1 us
    assert lib.h2o_selftest_bounded_wait(10 ** 9, None) == ARG     # above 100 ms


def test_q8_argument_checks(lib):
    """The 8-bit buffer calls refuse bad arguments on the host (through the
    binding's declared argument types), before any device work."""
    vp = ctypes.c_void_p
    p = vp(0x1000)
    d = _dims()
    qz = lambda n, dd, ptrs: lib.h2o_kv_quantize(n, dd, *ptrs, None)
    dq = lambda n, dd, ptrs: lib.h2o_kv_dequantize(n, dd, *ptrs, None)
    for f in (qz, dq):
        assert f(-1, 64, [p] * 3) == SHAPE
        assert f(4, 96, [p] * 3) == UNSUP
        assert f(0, 64, [None] * 3) == OK        # nothing to do
        assert f(4, 64, [p, None, p]) == NULL
        assert f(4, 128, [p, vp(0x1001), p]) == ALIGN
    n = ctypes.c_size_t(0)
    assert lib.h2o_q8_workspace_size(ctypes.byref(d), ctypes.byref(n)) == OK
    assert n.value == 2 * 2 * 256 * 64 * 2                  # K and V rows read back to bf16
    assert lib.h2o_q8_workspace_size(ctypes.byref(_dims(M=0)), ctypes.byref(n)) == OK
    assert n.value == 0
    base = ctypes.c_size_t(0)
    dd = _dims(S=1, M=100)
    assert lib.h2o_workspace_size(ctypes.byref(dd), ctypes.byref(base)) == OK
    assert lib.h2o_q8_workspace_size(ctypes.byref(dd), ctypes.byref(n)) == OK
    assert n.value == base.value       # S = 1: the decode kernels read the codes themselves

    up = lambda dims, ptrs, ev=p, budget=256, W=32, policy=0: lib.h2o_update_q8(
        ctypes.byref(dims), 256, *ptrs, budget, W, policy, ev, None)
    ok9 = [p] * 9
    assert up(d, ok9, ev=None) == NULL                       # evict_idx is required
    assert up(d, ok9[:5] + [None] + ok9[6:]) == NULL         # k_codes
    assert up(d, ok9[:6] + [vp(0x1004)] + ok9[7:]) == ALIGN  # k_scales
    assert up(d, ok9, budget=255) == ARG
    assert up(d, ok9, policy=7) == ARG
    assert up(_dims(d=96), ok9) == UNSUP
    ei = lambda dims, ptrs, ev=p, W=32: lib.h2o_evict_insert_q8(
        ctypes.byref(dims), 256, *ptrs, 256, W, 0, ev, None)
    ok8 = [p] * 8
    assert ei(d, ok8, ev=None) == NULL
    assert ei(d, ok8[:7] + [None]) == NULL                   # v_scales
    assert ei(d, ok8[:4] + [vp(0x1008)] + ok8[5:]) == ALIGN  # k_codes
    assert ei(d, ok8, W=257) == ARG
    assert ei(_dims(S=300), ok8) == SHAPE

    ws = ctypes.c_size_t(0)
    assert lib.h2o_q8_workspace_size(ctypes.byref(d), ctypes.byref(ws)) == OK
    ch = lambda dims, ptrs, w=p, wb=ws.value, pos0=256: lib.h2o_sdpa_chunk_q8(
        ctypes.byref(dims), pos0, 0.0, *ptrs, w, wb, None)
    ok10 = [p] * 10
    assert ch(d, ok10, w=None) == WORKSPACE
    assert ch(d, ok10, wb=ws.value - 1) == WORKSPACE
    assert ch(d, ok10, w=vp(0x1004)) == ALIGN
    assert ch(d, [p, None] + ok10[2:]) == NULL               # k_codes
    assert ch(d, ok10[:3] + [vp(0x100c)] + ok10[4:]) == ALIGN  # v_codes
    assert ch(d, [None] + ok10[1:]) == NULL                  # q, checked by the attention
    assert ch(d, ok10, pos0=-1) == ARG
    ca = lambda dims, ptrs, w=p, wb=ws.value: lib.h2o_sdpa_cache_q8(
        ctypes.byref(dims), 256, 0.0, *ptrs, w, wb, None)
    assert ca(_dims(M=0), [p] * 8, w=None, wb=0) == SHAPE
    assert ca(d, [p] * 8, w=None) == WORKSPACE
    assert ca(d, [p] * 4 + [None] + [p] * 3) == NULL         # v_scales


def test_q8_binding_marshals_to_the_host_checks(lib):
    """The Python q8 wrappers reject wrong tensors themselves and hand the rest
    to the C checks in the declared order (no GPU: a valid call ends at the
    device lookup)."""
    import types

    import torch
    bf16, i8, f32 = torch.bfloat16, torch.int8, torch.float32
    st = types.SimpleNamespace(cuda_stream=0)            # the legacy default stream
    with pytest.raises(ValueError):
        b.h2o_kv_quantize(torch.zeros((4, 64), dtype=f32), stream=st)
    with pytest.raises(b.H2OError) as e:
        b.h2o_kv_quantize(torch.zeros((4, 96), dtype=bf16), stream=st)
    assert e.value.status == UNSUP                       # d reached the C side as d
    with pytest.raises(b.H2OError) as e:
        b.h2o_kv_dequantize(torch.zeros((4, 64), dtype=i8), torch.zeros(4, dtype=f32), stream=st)
    assert e.value.status == -10                         # no device: past every argument check
    B, Hq, Hkv, d, S, M = 1, 4, 2, 64, 8, 32
    codes = torch.zeros((B, Hkv, M, d), dtype=i8)
    scales = torch.zeros((B, Hkv, M), dtype=f32)
    scores = torch.zeros((B, Hkv, M), dtype=f32)
    pos = torch.zeros((B, Hkv, M), dtype=torch.int32)
    kn = torch.zeros((B, Hkv, S, d), dtype=bf16)
    with pytest.raises(ValueError):                      # scales given as codes
        b.h2o_evict_insert_q8(scores, pos, kn, kn, codes, codes, codes, scales, 100, 8, stream=st)
    with pytest.raises(b.H2OError) as e:                 # budget != M, checked in C
        b.h2o_evict_insert_q8(scores, pos, kn, kn, codes, scales, codes, scales, 100, 8,
                              budget=M - 1, stream=st)
    assert e.value.status == ARG
    q = torch.zeros((B, Hq, S, d), dtype=bf16)
    with pytest.raises(ValueError):                      # v_scales of the wrong shape
        b.h2o_sdpa_chunk_q8(q, codes, scales, codes, scales[:, :, :-1], kn, kn, pos, 100, stream=st)
    with pytest.raises(b.H2OError) as e:
        b.h2o_sdpa_cache_q8(q, codes, scales, codes, scales, pos, -1,
                            workspace=torch.zeros(1 << 20, dtype=torch.uint8), stream=st)
    assert e.value.status == ARG                         # pos0 < 0
