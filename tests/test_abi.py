"""The C ABI on the host: exported symbols, argument checks, host helpers.

Nothing here launches a kernel: every call either is host-only or fails its
argument checks before any CUDA call, so these run without a GPU.
"""

import ctypes as C
import os
import re

import numpy as np
import pytest

import oracle as O

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def wz():
    import paper_2607_23265_gb300.build as build
    build.build()
    import paper_2607_23265_gb300.wavezip as m
    return m


def declared_symbols():
    text = open(os.path.join(ROOT, "include", "wavezip.h")).read()
    return sorted(set(re.findall(r"WZ_API[^;(]*?\b(wz_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    syms = declared_symbols()
    for name in ["wz_condense", "wz_condense_ex", "wz_condense_batch", "wz_relevance", "wz_dwt1d",
                 "wz_idwt1d", "wz_dwt2d", "wz_idwt2d", "wz_budget_size", "wz_dwt_len",
                 "wz_status_string"]:
        assert name in syms


def test_library_exports_every_declared_symbol(wz):
    lib = C.CDLL(wz.LIB_PATH)
    for name in declared_symbols():
        assert hasattr(lib, name), name


def test_struct_layout_matches_defaults(wz):
    a = wz.CondenseArgs()
    wz._lib.wz_condense_args_init(C.byref(a))
    assert (a.lam, a.tau, a.wta_wavelet, a.wsm_wavelet, a.mode, a.path, a.dtype) == (1.5, 0.0, 1, 4, 0, 0, 0)
    assert (a.temporal_mode, a.spatial_mode) == (wz.TEMPORAL_WTA, wz.SPATIAL_WSM)
    assert a.relevance_mode == wz.RELEVANCE_MEAN
    assert (a.wta_levels, a.wsm_levels) == (1, 1)
    b = wz.BatchArgs()
    wz._lib.wz_batch_args_init(C.byref(b))
    assert (b.lam, b.wta_wavelet, b.wsm_wavelet) == (1.5, 1, 4)


def test_budget_size_matches_oracle(wz):
    for T, H, W, r in [(64, 13, 13, 0.1), (256, 27, 27, 0.1), (16, 14, 14, 0.25), (1, 1, 3, 0.5),
                       (7, 9, 1, 1.0), (128, 16, 16, 0.05), (3, 5, 7, 0.123456)]:
        assert wz.wz_budget_size(T, H, W, r) == O.global_budget(r, T, H * W)
    assert wz.wz_budget_size(4, 4, 4, 0.0) == -1
    assert wz.wz_budget_size(4, 4, 4, 1.5) == -1
    assert wz.wz_budget_size(0, 4, 4, 0.5) == -1


def test_batch_rows(wz):
    rows, offs = wz.wz_batch_rows(3, 64, 13, 13, [0.05, 0.1, 0.25])
    Bs = [O.global_budget(r, 64, 169) for r in (0.05, 0.1, 0.25)]
    assert rows == sum(Bs) and offs == [0, Bs[0], Bs[0] + Bs[1], sum(Bs)]


def test_dwt_len(wz):
    for n in [1, 2, 13, 14, 16, 27, 64]:
        for p in [1, 2, 4, 10, 44]:
            assert wz.wz_dwt_len(n, p) == O.dwt_len(n, O.wavelet_filters(p)["F"])
    assert wz.wz_dwt_len(0, 4) == -1 and wz.wz_dwt_len(5, 11) == -1


@pytest.mark.parametrize("p", [1, 2, 3, 4, 6, 8, 10, 44])
def test_library_filters_match_oracle(wz, p):
    lib = wz.wz_wavelet_filters(p)
    ref = O.wavelet_filters(p)
    for k in ("dec_lo", "dec_hi", "rec_lo", "rec_hi"):
        assert np.allclose(lib[k], ref[k], atol=1e-11), k


def test_status_strings(wz):
    assert wz.status_string(0) == "ok"
    assert "invalid" in wz.status_string(-1)
    assert wz.status_string(12345) == "unknown status"


# Fake but aligned device addresses: argument checks reject the call before
# any pointer is used or any CUDA call is made.
P = 1 << 20


def _args(wz, **over):
    a = wz.CondenseArgs()
    wz._lib.wz_condense_args_init(C.byref(a))
    vals = dict(features=P, T=4, H=5, W=6, D=16, query=2 * P, Lq=3, ratio=0.5, out_tokens=3 * P,
                out_index=4 * P)
    vals.update(over)
    for k, v in vals.items():
        setattr(a, k, v)
    return a


@pytest.mark.parametrize("over,code", [
    (dict(features=None), -1), (dict(query=None), -1), (dict(out_tokens=None), -1),
    (dict(out_index=None), -1), (dict(T=0), -1), (dict(H=0), -1), (dict(D=12), -2),
    (dict(H=65), -2), (dict(T=5000), -2), (dict(Lq=0), -1), (dict(ratio=0.0), -1),
    (dict(ratio=1.01), -1), (dict(ratio=float("nan")), -1), (dict(lam=-1.0), -1),
    (dict(lam=float("inf")), -1), (dict(wta_wavelet=11), -1), (dict(wta_wavelet=0), -1),
    (dict(wsm_wavelet=11), -1), (dict(mode=3), -1), (dict(path=7), -1), (dict(dtype=5), -1),
    (dict(temporal_mode=3), -1), (dict(temporal_mode=-1), -1), (dict(spatial_mode=3), -1),
    (dict(relevance_mode=2), -1), (dict(relevance_mode=1), -2),                 # max-over-query: D % 64
    (dict(wta_levels=0), -1), (dict(wta_levels=5), -1), (dict(wsm_levels=5), -1),
    (dict(H=64, W=64, wsm_levels=4, wsm_wavelet=10), -2),                      # level tables exceed a CTA
    (dict(relevance_mode=1, D=64, dtype=1), -2), (dict(relevance_mode=1, D=64, Lq=129), -2),
    (dict(dtype=1, path=1), -2), (dict(features=P + 4), -1), (dict(out_tokens=3 * P + 8), -1),
    (dict(workspace=5 * P, workspace_bytes=16), -5), (dict(workspace=5 * P + 64, workspace_bytes=1 << 30), -1),
])
def test_condense_argument_errors(wz, over, code):
    a = _args(wz, **over)
    assert wz._lib.wz_condense_ex(C.byref(a)) == code


def test_simple_entry_point_errors(wz):
    lib = wz._lib
    assert lib.wz_condense(None, 4, 5, 6, 16, P, 3, 0.5, P, P, None) == -1
    assert lib.wz_condense(P, 4, 5, 6, 10, P, 3, 0.5, P, P, None) == -2
    assert lib.wz_relevance(P, 4, 5, 6, 16, 0, P, 0, P, P, None, None, 0, None, None) == -1
    assert lib.wz_relevance(P, 4, 5, 6, 12, 0, P, 2, P, P, None, None, 0, None, None) == -2
    assert lib.wz_relevance(P, 4, 5, 6, 16, 0, P, 2, P, P, None, None, 0, P + 2, None) == -1   # misaligned status
    assert lib.wz_dwt1d(None, 3, 8, 4, 0, P, P, None) == -1
    assert lib.wz_dwt1d(P, 3, 8, 4, 7, P, P, None) == -1
    assert lib.wz_idwt1d(P, P, 3, 0, 4, P, None) == -1
    assert lib.wz_dwt2d(P, 2, 70, 5, 8, 0, 4, 0, P, P, P, P, None) == -2
    assert lib.wz_idwt2d(P, P, None, P, 2, 5, 5, 8, 4, P, None) == -1


def test_batch_argument_errors(wz):
    b = wz.BatchArgs()
    wz._lib.wz_batch_args_init(C.byref(b))
    lq = (C.c_int32 * 2)(3, 4)
    rt = (C.c_float * 2)(0.5, 0.0)
    b.V, b.features, b.T, b.H, b.W, b.D = 2, P, 4, 5, 6, 16
    b.queries, b.Lq, b.ratio, b.out_tokens, b.out_index = 2 * P, lq, rt, 3 * P, 4 * P
    assert wz._lib.wz_condense_batch(C.byref(b)) == -1          # ratio 0
    rt[1] = 0.25
    b.V = 2000
    assert wz._lib.wz_condense_batch(C.byref(b)) == -2          # too many videos
    b.V = 2
    b.relevance_mode = wz.RELEVANCE_MAXSIM
    assert wz._lib.wz_condense_batch(C.byref(b)) == -2          # max-over-query wants D % 64 == 0
    b.D, lq[1] = 64, 200
    assert wz._lib.wz_condense_batch(C.byref(b)) == -2          # and at most 128 query rows
    b.D, lq[1], b.relevance_mode = 16, 4, wz.RELEVANCE_MEAN
    b.workspace, b.workspace_bytes = 5 * P, 8
    assert wz._lib.wz_condense_batch(C.byref(b)) == -5


def test_workspace_sizes_are_host_only(wz):
    n1 = wz.wz_condense_workspace_size(256, 27, 27, 3584, 0, 0.1)
    n2 = wz.wz_condense_workspace_size(256, 27, 27, 3584, 0, 0.25)
    assert 0 < n1 < n2 < 1 << 31
    assert wz.wz_condense_workspace_size(4, 4, 4, 12, 0, 0.5) == 0
    assert wz.wz_relevance_workspace_size(64, 13, 13, 3584) > 0
    assert wz.wz_batch_workspace_size(2, 64, 13, 13, 3584, 0, [0.1, 0.25]) > n1 / 100


def test_graph_cache_capacity_is_host_only(wz):
    """The replay cache's capacity and counters: set, query and restore
    without a GPU (an empty cache makes no CUDA call)."""
    st = wz.wz_graph_cache(-1)
    prev = st["previous_capacity"]
    assert prev >= 0 and st["kept"] == 0 and st["replays"] == 0 and st["captures"] == 0
    try:
        assert wz.wz_graph_cache(3)["previous_capacity"] == prev
        assert wz.wz_graph_cache(-5)["previous_capacity"] == 3     # negative: query only
        assert wz.wz_graph_cache(0)["previous_capacity"] == 3
        assert wz.wz_graph_cache(-1) == {"previous_capacity": 0, "kept": 0, "replays": 0, "captures": 0}
    finally:
        wz.wz_graph_cache(prev)
    assert wz.wz_graph_cache(-1)["previous_capacity"] == prev


def test_cached_path_checks_arguments_first(wz):
    """A call that would use the replay cache (caller workspace, no events)
    is rejected by the same argument checks, before any CUDA call."""
    for over, code in [(dict(D=12), -2), (dict(ratio=0.0), -1), (dict(workspace_bytes=16), -5)]:
        a = _args(wz, workspace=5 * P, workspace_bytes=1 << 30)
        for k, v in over.items():
            setattr(a, k, v)
        assert wz._lib.wz_condense_ex(C.byref(a)) == code
    assert wz.wz_graph_cache(-1)["kept"] == 0
