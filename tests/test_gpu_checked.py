"""The bounds-checked build (WZ_CHECKED: every guarded global write tests its
index) raises no status bit on a spread of calls, and its results equal the
normal build's bit for bit."""

import numpy as np
import pytest
import torch

import workload as wl

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wz():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_23265_gb300.wavezip as m
    assert torch.cuda.is_available()
    return m


CASES = [
    dict(shape=(12, 13, 13, 256, 6), ratio=0.2, kw={}),
    dict(shape=(9, 27, 27, 128, 4), ratio=0.1, kw=dict(wsm_levels=2, wta_levels=2)),
    dict(shape=(10, 11, 12, 192, 9), ratio=0.3, kw=dict(relevance="maxsim")),
    dict(shape=(8, 9, 7, 96, 3), ratio=0.25, kw=dict(path="simt", spatial_mode="saliency")),
    dict(shape=(20, 5, 6, 64, 2), ratio=0.5, kw=dict(tau=0.02, wsm_wavelet=44)),
    dict(shape=(3, 64, 64, 32, 2), ratio=0.05, kw=dict(wsm_wavelet=1)),
]


@pytest.mark.parametrize("case", CASES, ids=[str(i) for i in range(len(CASES))])
def test_checked_build_agrees(wz, case):
    T, H, W, D, Lq = case["shape"]
    X, Q = wl.random_video(T, H, W, D, Lq, seed=T + H)
    X, Q = X.cuda(), Q.cuda()
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ref = wz.wz_condense_ex(X, Q, case["ratio"], **case["kw"])
    with wz.checked_library():
        got = wz.wz_condense_ex(X, Q, case["ratio"], device_status=st, **case["kw"])
    torch.cuda.synchronize()
    assert int(st.item()) == 0
    for k in ("budgets", "index", "tokens", "count"):
        assert torch.equal(got[k], ref[k]), k


def test_checked_build_batch(wz):
    specs = [(16, 9, 9, 128, 4, 0.2), (16, 9, 9, 128, 30, 0.1)]
    vids = [wl.random_video(T, H, W, D, Lq, seed=7 + i) for i, (T, H, W, D, Lq, _) in enumerate(specs)]
    X = torch.stack([x for x, _ in vids]).cuda()
    Qs = torch.cat([q for _, q in vids]).cuda()
    Lqs, ratios = [s[4] for s in specs], [s[5] for s in specs]
    ref = wz.wz_condense_batch(X, Qs, Lqs, ratios)
    with wz.checked_library():
        got = wz.wz_condense_batch(X, Qs, Lqs, ratios)
    torch.cuda.synchronize()
    for k in ("budgets", "index", "tokens", "count"):
        assert torch.equal(got[k], ref[k]), k
