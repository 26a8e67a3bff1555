"""Max-over-query relevance (token x query-row cosines on the tensor cores) vs
the CPU oracle, through the C ABI.

Budgets and the index map are bit-exact (seeds are chosen so that every
integer decision is at least 1e-4 quota units from its boundary); r_t within
1e-5; tokens within the condensation tolerance.  The token cosines run on
bf16 features against the unit query rows split into bf16 hi + lo (relative
error of the row ~2^-17) with fp32 accumulation, so a_{t,n} is good to ~1e-5;
it reaches the tokens only through the gate of the WSM.
"""

import numpy as np
import pytest
import torch

import oracle as O
import workload as wl
from helpers import accepted_random, accepted_video, compare_condense, oracle_run

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wz():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_23265_gb300.wavezip as m
    assert torch.cuda.is_available()
    return m


def _run(wz, X, Q, ratio, **kw):
    out = wz.wz_condense_ex(X.cuda(), Q.cuda(), ratio, relevance="maxsim", **kw)
    torch.cuda.synchronize()
    return out


def _check_r(out, ref):
    rel = out["relevance"].cpu().double().numpy()
    assert np.allclose(rel[:, 0], ref["r"], atol=1e-5), np.abs(rel[:, 0] - ref["r"]).max()


@pytest.mark.parametrize("T,H,W,D,Lq,ratio", [
    (10, 13, 13, 128, 5, 0.2),     # the common case: two MMA K steps
    (7, 9, 11, 192, 37, 0.3),      # 693 tokens: ragged 128-row tile, Lq not a multiple of 16
    (4, 16, 16, 64, 128, 0.5),     # the largest query: N = 256 columns
    (3, 5, 5, 64, 1, 0.5),         # one row: the similarity branch itself
    (1, 27, 27, 256, 16, 0.1),     # one frame
    (40, 3, 4, 64, 3, 0.25),       # 12-token frames, 480 tokens: tiles span many frames
])
def test_maxsim_parity(wz, T, H, W, D, Lq, ratio):
    X, Q = accepted_random(T, H, W, D, Lq, ratio, seed=T * 13 + Lq, relevance="maxsim")
    ref = oracle_run(X, Q, ratio, relevance="maxsim")
    out = _run(wz, X, Q, ratio)
    compare_condense(out, ref, X.dtype)
    _check_r(out, ref)


def test_maxsim_one_row_equals_mean(wz):
    # with one query row both scorers compute the same a_{t,n} and r_t
    X, Q = accepted_random(12, 13, 13, 128, 1, 0.2, seed=5)
    a = _run(wz, X, Q, 0.2)
    b = wz.wz_condense_ex(X.cuda(), Q.cuda(), 0.2)
    torch.cuda.synchronize()
    assert torch.equal(a["budgets"], b["budgets"]) and torch.equal(a["index"], b["index"])
    assert np.allclose(a["relevance"][:, 0].cpu().numpy(), b["relevance"][:, 0].cpu().numpy(), atol=1e-6)
    d = (a["tokens"].float() - b["tokens"].float()).abs()
    assert float(d.max()) <= 1e-3 + 2e-2 * float(b["tokens"].float().abs().max())


def test_maxsim_structured_video(wz):
    spec = wl.VideoSpec(T=24, H=13, W=13, D=256, Lq=24, ratio=0.15, cuts=2, patches=2, seed=91)
    s, X, Q, _ = accepted_video(spec, relevance="maxsim")
    ref = oracle_run(X, Q, s.ratio, relevance="maxsim")
    out = _run(wz, X, Q, s.ratio)
    compare_condense(out, ref, X.dtype)
    _check_r(out, ref)


def test_maxsim_64_frame_workload(wz):
    spec, X, Q, _ = accepted_video(wl.CONFIGS["video64_13x13_bf16"], tries=4, relevance="maxsim")
    ref = oracle_run(X, Q, spec.ratio, relevance="maxsim")
    out = _run(wz, X, Q, spec.ratio)
    compare_condense(out, ref, X.dtype)
    _check_r(out, ref)


def test_maxsim_with_ablation_and_simt(wz):
    kw = dict(temporal_mode="raw", spatial_mode="saliency")
    X, Q = accepted_random(9, 11, 11, 128, 7, 0.25, seed=3, relevance="maxsim", **kw)
    ref = oracle_run(X, Q, 0.25, relevance="maxsim", **kw)
    out = _run(wz, X, Q, 0.25, path="simt", **kw)
    compare_condense(out, ref, X.dtype)


def test_maxsim_with_levels(wz):
    kw = dict(wta_levels=2, wsm_levels=2, wsm_wavelet=2)
    X, Q = accepted_random(8, 11, 12, 128, 9, 0.3, seed=17, relevance="maxsim", **kw)
    ref = oracle_run(X, Q, 0.3, relevance="maxsim", **kw)
    out = _run(wz, X, Q, 0.3, **kw)
    compare_condense(out, ref, X.dtype)
    _check_r(out, ref)


def test_maxsim_batch(wz):
    # videos of 1, 20 and 128 query rows share one buffer of query rows in turn
    T, H, W, D = 16, 9, 9, 128
    Lqs, ratios = [1, 20, 128], [0.3, 0.2, 0.25]
    vids = [accepted_random(T, H, W, D, lq, r, seed=300 + lq, relevance="maxsim") for lq, r in zip(Lqs, ratios)]
    X = torch.stack([v[0] for v in vids])
    Qc = torch.cat([v[1] for v in vids])
    out = wz.wz_condense_batch(X.cuda(), Qc.cuda(), Lqs, ratios, relevance="maxsim")
    torch.cuda.synchronize()
    offs = out["row_offsets"]
    for v, ((Xv, Qv), r) in enumerate(zip(vids, ratios)):
        ref = oracle_run(Xv, Qv, r, relevance="maxsim")
        one = {"budgets": out["budgets"][v], "count": out["count"][v:v + 1],
               "index": out["index"][offs[v]:offs[v + 1]], "tokens": out["tokens"][offs[v]:offs[v + 1]]}
        compare_condense(one, ref, Xv.dtype)
        assert np.allclose(out["relevance"][v, :, 0].cpu().double().numpy(), ref["r"], atol=1e-5)


def test_maxsim_unsupported_inputs(wz):
    X, Q = wl.random_video(4, 5, 5, 64, 3, dtype="f32", seed=1)
    with pytest.raises(wz.WaveZipError):
        _run(wz, X, Q, 0.5)                              # fp32 features
    X, Q = wl.random_video(4, 5, 5, 72, 3, seed=1)
    with pytest.raises(wz.WaveZipError):
        _run(wz, X, Q, 0.5)                              # D not a multiple of 64
    X, Q = wl.random_video(4, 5, 5, 64, 129, seed=1)
    with pytest.raises(wz.WaveZipError):
        _run(wz, X, Q, 0.5)                              # more than 128 query rows
