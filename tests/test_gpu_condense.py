"""CUDA condensation path vs the CPU oracle, through the C ABI.

Budgets, offsets and index maps must match bit-exactly; condensed tokens
within |g - o| <= 1e-3 + 2e-2 |o| of the oracle's values rounded to the
output dtype (bf16 inputs, fp32 accumulation, bf16 outputs).
"""

import numpy as np
import pytest
import torch

import oracle as O
import workload as wl
from helpers import (accepted_random, accepted_video, assert_tokens_close, compare_condense,
                     oracle_run, oracle_videos, to_np64)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wz():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_23265_gb300.wavezip as m
    assert torch.cuda.is_available()
    return m


def run(wz, X, Q, ratio, **kw):
    out = wz.wz_condense_ex(X.cuda(), Q.cuda(), ratio, **kw)
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("name", ["tiny_f32_16x14x14", "video64_13x13_bf16", "video128_16x16_objects"])
def test_config_parity_full(wz, name):
    spec, X, Q, _ = accepted_video(wl.CONFIGS[name])
    ref = oracle_run(X, Q, spec.ratio)
    out = run(wz, X, Q, spec.ratio)
    compare_condense(out, ref, X.dtype)


def test_config_256_frames_full(wz):
    """The 1.3 GB workload (256 frames of 27x27x3584 bf16, 18,662 condensed
    tokens): every budget, index row, condensed token and r~ against the
    oracle's full condensation."""
    spec, X, Q, _ = accepted_video(wl.CONFIGS["video256_27x27_bf16"], tries=4)
    ref = oracle_run(X, Q, spec.ratio)
    out = run(wz, X, Q, spec.ratio)
    assert int(out["count"].cpu()[0]) == ref["B"] == 18662
    compare_condense(out, ref, X.dtype)


def _random_case(wz, T, H, W, D, Lq, ratio, seed=0, dtype="bf16", **kw):
    okw = {k: v for k, v in kw.items()
           if k in ("lam", "tau", "wta_wavelet", "wsm_wavelet", "mode", "temporal_mode", "spatial_mode",
                    "relevance", "wta_levels", "wsm_levels")}
    X, Q = accepted_random(T, H, W, D, Lq, ratio, seed=seed, dtype=dtype, **okw)
    ref = oracle_run(X, Q, ratio, **okw)
    out = run(wz, X, Q, ratio, **kw)
    compare_condense(out, ref, X.dtype)
    return out, ref


@pytest.mark.parametrize("T,H,W,D,Lq,ratio", [
    (1, 5, 5, 64, 3, 0.5),        # one frame
    (5, 1, 1, 16, 2, 1.0),        # one token per frame
    (6, 2, 3, 8, 1, 0.5),         # tiny map, D = 8
    (7, 9, 11, 136, 4, 0.3),      # odd T, ragged channel tile and K chunk
    (9, 27, 27, 264, 8, 0.1),     # 27x27, several K chunks, ragged tail
    (4, 16, 16, 128, 4, 1.0),     # ratio 1: every frame keeps N tokens
    (12, 13, 13, 256, 16, 0.002),  # B = 4 tokens
    (3, 64, 64, 32, 2, 0.05),     # largest map
    (33, 14, 14, 96, 5, 0.25),
    (600, 3, 4, 16, 2, 0.3),      # more frames than temporal threads: 2 frames per thread
    (4096, 2, 2, 8, 1, 0.4),      # longest video: 8 frames per thread, 4096-way ranking
    (3, 4, 4, 32768, 2, 0.5),     # widest bf16 rows: 8 vectors per relevance thread, 256 channel tiles
    (2, 3, 5, 12288, 3, 0.4),     # 4 vectors per relevance thread
])
def test_shapes(wz, T, H, W, D, Lq, ratio):
    _random_case(wz, T, H, W, D, Lq, ratio, seed=T * 7 + H)


@pytest.mark.parametrize("kw", [dict(lam=0.0), dict(lam=2.0), dict(wsm_wavelet=1), dict(wsm_wavelet=2),
                                dict(mode="zero"), dict(mode="periodic"), dict(path="simt"),
                                dict(wta_wavelet=4), dict(wta_wavelet=2, wsm_wavelet=1),
                                dict(wta_wavelet=10, temporal_mode="wta"), dict(wsm_wavelet=44),
                                dict(wta_wavelet=44, wsm_wavelet=44), dict(wsm_wavelet=44, path="simt")])
def test_options(wz, kw):
    _random_case(wz, 10, 13, 13, 128, 6, 0.2, seed=5, **kw)


@pytest.mark.parametrize("T,H,W,D,ratio,kw", [
    (3, 27, 27, 256, 0.8, {}),                       # ~583 tokens a frame: blocks of 256, 256, 71
    (2, 40, 40, 64, 0.6, {}),                        # 960 tokens, a 40-row map: four blocks
    (3, 27, 27, 128, 0.7, dict(mode="zero")),
    (3, 27, 27, 128, 0.7, dict(mode="periodic")),    # supports wrap: every chunk
    (3, 27, 27, 128, 0.7, dict(wsm_wavelet=44)),     # 10-tap supports
    (3, 27, 27, 128, 0.7, dict(wsm_wavelet=1)),      # Haar: narrow supports
    (3, 27, 27, 128, 0.7, dict(wsm_levels=2)),       # multi-level: every chunk
    (2, 27, 27, 128, 0.8, dict(spatial_mode="saliency")),
])
def test_split_frames(wz, T, H, W, D, ratio, kw):
    # frames of more than 256 tokens are condensed in blocks of 256 output
    # tokens; a block's operator rows reach only part of the map, and the
    # tensor-core units skip the 32-token chunks outside it
    _random_case(wz, T, H, W, D, 4, ratio, seed=T * 31 + H, **kw)


@pytest.mark.parametrize("kw", [dict(wta_levels=2), dict(wta_levels=3, wta_wavelet=2), dict(wta_levels=4, wta_wavelet=4),
                                dict(wsm_levels=2), dict(wsm_levels=3, wsm_wavelet=1), dict(wsm_levels=2, wsm_wavelet=44),
                                dict(wsm_levels=2, path="simt"), dict(wsm_levels=2, mode="zero"),
                                dict(wsm_levels=3, mode="periodic", wsm_wavelet=2),
                                dict(wta_levels=4, wsm_levels=4, wsm_wavelet=1)])
def test_levels(wz, kw):
    _random_case(wz, 10, 13, 13, 128, 6, 0.2, seed=5, **kw)


@pytest.mark.parametrize("T,H,W,D,kw", [
    (24, 27, 27, 256, dict(wsm_levels=3)),                    # the 27x27 map, three db4 levels
    (9, 7, 9, 64, dict(wsm_levels=2, wta_levels=2)),          # non-square, subbands wider than the map
    (5, 64, 64, 32, dict(wsm_levels=2, wsm_wavelet=1)),       # the largest map
    (600, 3, 4, 16, dict(wta_levels=3)),                      # two frames per temporal thread
])
def test_levels_shapes(wz, T, H, W, D, kw):
    _random_case(wz, T, H, W, D, 4, 0.25, seed=T + H, **kw)


@pytest.mark.parametrize("kw", [dict(temporal_mode="raw"), dict(temporal_mode="uniform"),
                                dict(spatial_mode="saliency"), dict(spatial_mode="none"),
                                dict(spatial_mode="saliency", lam=0.7, temporal_mode="raw"),
                                dict(temporal_mode="uniform", spatial_mode="none", path="simt")])
def test_ablation_modes(wz, kw):
    _random_case(wz, 10, 13, 13, 128, 6, 0.2, seed=5, **kw)


@pytest.mark.parametrize("tm,sm", [("raw", "wsm"), ("uniform", "saliency"), ("raw", "none")])
def test_ablation_modes_structured_video(wz, tm, sm):
    kw = dict(temporal_mode=tm, spatial_mode=sm)
    spec = wl.VideoSpec(T=24, H=13, W=13, D=256, Lq=8, ratio=0.15, cuts=2, patches=2, seed=77)
    s, X, Q, _ = accepted_video(spec, **kw)
    ref = oracle_run(X, Q, s.ratio, **kw)
    out = run(wz, X, Q, s.ratio, **kw)
    compare_condense(out, ref, X.dtype)


def test_ablation_saliency_fp32(wz):
    _random_case(wz, 6, 9, 11, 64, 4, 0.3, seed=11, dtype="f32", spatial_mode="saliency")


@pytest.mark.parametrize("which", ["both", "tokens", "frames"])
def test_external_scores(wz, which):
    from helpers import MIN_MARGIN
    g = np.random.default_rng(21)
    T, H, W, D, Lq, ratio = 10, 13, 13, 128, 6, 0.2
    for attempt in range(20):
        a_ext = g.random((T, H * W)).astype(np.float32)
        r_ext = g.normal(0.1, 0.2, T).astype(np.float32)
        kw = {}
        if which in ("both", "tokens"):
            kw["token_scores"] = a_ext
        if which in ("both", "frames"):
            kw["frame_scores"] = r_ext
        X, Q = wl.random_video(T, H, W, D, Lq, seed=40 + attempt)
        ref = oracle_run(X, Q, ratio, **kw)
        if O.decision_margins(ref) >= MIN_MARGIN:
            break
    out = run(wz, X, Q, ratio, **{k: torch.from_numpy(v).cuda() for k, v in kw.items()})
    compare_condense(out, ref, X.dtype)
    if "frame_scores" in kw:
        assert np.allclose(out["relevance"][:, 0].cpu().numpy(), r_ext, atol=0)


def test_fp32_features(wz):
    _random_case(wz, 6, 14, 14, 96, 4, 0.25, seed=3, dtype="f32")


@pytest.mark.parametrize("D", [16384, 4104])
def test_fp32_wide_rows(wz, D):
    # f32 rows up to the f32 limit (half of the bf16 one): 8 and 2 vectors per relevance thread
    _random_case(wz, 3, 4, 4, D, 2, 0.5, seed=D, dtype="f32")


def test_zero_budget(wz):
    X, Q = wl.random_video(3, 4, 4, 16, 2, seed=1)
    ratio = 0.01                                  # 0.48 tokens -> B = 0
    assert wz.wz_budget_size(3, 4, 4, ratio) == 0
    out = run(wz, X, Q, ratio)
    assert out["tokens"].shape == (0, 16) and int(out["count"].cpu()[0]) == 0
    assert int(out["budgets"].sum()) == 0


def test_frame_filter_tail_rows(wz):
    """tau > 0 drops static frames; rows past the produced count are -1 / 0."""
    g = torch.Generator().manual_seed(3)
    base = torch.randn((1, 6, 6, 32), generator=g, dtype=torch.float64)
    frames = [base + 0.001 * torch.randn((1, 6, 6, 32), generator=g, dtype=torch.float64) for _ in range(8)]
    frames[4] = torch.randn((1, 6, 6, 32), generator=g, dtype=torch.float64)   # a scene cut
    X = torch.cat(frames).to(torch.bfloat16)
    Q = torch.randn((3, 32), generator=g, dtype=torch.float64).to(torch.bfloat16)
    ratio, tau = 0.9, 0.05
    ref = oracle_run(X, Q, ratio, tau=tau)
    assert len(ref["keep"]) < 8 and ref["count"] < ref["B"]
    assert O.decision_margins(ref) > 1e-4
    out = run(wz, X, Q, ratio, tau=tau)
    compare_condense(out, ref, X.dtype)


def test_all_negative_relevance_is_uniform(wz):
    g = torch.Generator().manual_seed(4)
    c = torch.randn((64,), generator=g, dtype=torch.float64)
    X = (c + 0.3 * torch.randn((10, 5, 5, 64), generator=g, dtype=torch.float64)).to(torch.bfloat16)
    Q = (-c).reshape(1, 64).repeat(2, 1).to(torch.bfloat16)
    ref = oracle_run(X, Q, 0.3)
    assert np.all(ref["r"] < 0) and ref["budgets"].max() - ref["budgets"].min() <= 1
    out = run(wz, X, Q, 0.3)
    compare_condense(out, ref, X.dtype)


@pytest.mark.parametrize("ratio", [0.5, 0.6])
def test_caps_bind(wz, ratio):
    """Two dominant frames capped at N; at 0.6 every positive frame ends up
    capped and the rest spreads uniformly over the zero-weight frames.  The
    quotas there are exact ties (computed identically on both sides), so no
    margin is asked for."""
    g = torch.Generator().manual_seed(6)
    c = torch.randn((64,), generator=g, dtype=torch.float64)
    noise = 0.5 * torch.randn((6, 4, 4, 64), generator=g, dtype=torch.float64)
    X = noise.clone()
    X[0] += 3 * c
    X[1] += 3 * c
    Q = c.reshape(1, 64).to(torch.bfloat16)
    X = X.to(torch.bfloat16)
    ref = oracle_run(X, Q, ratio)
    assert ref["budgets"][0] == 16 and ref["budgets"][1] == 16
    out = run(wz, X, Q, ratio)
    compare_condense(out, ref, X.dtype)


def test_workspace_and_status(wz):
    X, Q = accepted_random(8, 13, 13, 128, 4, 0.2, seed=9)
    Xc, Qc = X.cuda(), Q.cuda()
    a = run(wz, X, Q, 0.2)
    nbytes = wz.wz_condense_workspace_size(8, 13, 13, 128, 0, 0.2)
    ws = torch.empty((nbytes,), dtype=torch.uint8, device="cuda")
    st = torch.zeros((1,), dtype=torch.int32, device="cuda")
    b = wz.wz_condense_ex(Xc, Qc, 0.2, workspace=ws, device_status=st)
    c = wz.wz_condense_ex(Xc, Qc, 0.2, workspace=ws, device_status=st)
    torch.cuda.synchronize()
    assert int(st.cpu()[0]) == 0
    for k in ("tokens", "index", "budgets"):
        assert torch.equal(a[k], b[k]) and torch.equal(b[k], c[k]), k
    with pytest.raises(wz.WaveZipError):
        wz.wz_condense_ex(Xc, Qc, 0.2, workspace=ws[: nbytes // 2])


def test_plain_entry_point(wz):
    X, Q = accepted_random(6, 13, 13, 128, 4, 0.2, seed=2)
    tok, idx = wz.wz_condense(X.cuda(), Q.cuda(), 0.2)
    torch.cuda.synchronize()
    ref = oracle_run(X, Q, 0.2)
    assert np.array_equal(idx.cpu().numpy(), ref["out_index"])
    from helpers import round_like
    assert_tokens_close(to_np64(tok), round_like(ref["out_tokens"], torch.bfloat16))


def test_batch_parity(wz):
    specs = [wl.VideoSpec(T=16, H=13, W=13, D=256, Lq=lq, ratio=r, cuts=2, seed=s)
             for lq, r, s in [(8, 0.05, 21), (40, 0.1, 22), (17, 0.25, 23)]]
    vids = [accepted_video(s) for s in specs]
    X = torch.stack([v[1] for v in vids])
    Qs = torch.cat([v[2] for v in vids])
    out = wz.wz_condense_batch(X.cuda(), Qs.cuda(), [s.Lq for s, *_ in vids], [s.ratio for s, *_ in vids])
    torch.cuda.synchronize()
    offs = out["row_offsets"]
    for v, (s, Xv, Qv, _) in enumerate(vids):
        ref = oracle_run(Xv, Qv, s.ratio)
        sub = {"budgets": out["budgets"][v], "count": out["count"][v:v + 1],
               "index": out["index"][offs[v]:offs[v + 1]], "tokens": out["tokens"][offs[v]:offs[v + 1]]}
        compare_condense(sub, ref, Xv.dtype)


def test_batch_of_many_small_videos(wz):
    """130 videos in one call (several hundred frames, more videos than the
    prefix blocks of a warp): every video's budgets, index map and tokens."""
    g = np.random.default_rng(9)
    V, T, H, W, D = 130, 5, 5, 6, 64
    Lqs = [int(x) for x in g.integers(1, 9, size=V)]
    ratios = [float(x) for x in g.choice([0.1, 0.3, 0.7], size=V)]
    vids = [accepted_random(T, H, W, D, lq, r, seed=5000 + 13 * v) for v, (lq, r) in enumerate(zip(Lqs, ratios))]
    X = torch.stack([x for x, _ in vids])
    Qs = torch.cat([q for _, q in vids])
    out = wz.wz_condense_batch(X.cuda(), Qs.cuda(), Lqs, ratios)
    torch.cuda.synchronize()
    offs = out["row_offsets"]
    for v, ((Xv, Qv), r) in enumerate(zip(vids, ratios)):
        ref = oracle_run(Xv, Qv, r)
        sub = {"budgets": out["budgets"][v], "count": out["count"][v:v + 1],
               "index": out["index"][offs[v]:offs[v + 1]], "tokens": out["tokens"][offs[v]:offs[v + 1]]}
        compare_condense(sub, ref, Xv.dtype)


def test_config_serving_batch_full(wz):
    """The serving batch at full size (32 videos x 64 frames, 13x13x3584 bf16,
    Lq in [8, 128], ratios in {0.05, 0.1, 0.25}) in one call: every video's
    budgets, index map, condensed tokens and r~ against the oracle's full
    condensation of that video (computed on a pool of spawned processes)."""
    vids = oracle_videos(wl.batch_specs())
    X = torch.stack([v[1] for v in vids])
    Qs = torch.cat([v[2] for v in vids])
    out = wz.wz_condense_batch(X.cuda(), Qs.cuda(), [s.Lq for s, *_ in vids], [s.ratio for s, *_ in vids])
    torch.cuda.synchronize()
    offs = out["row_offsets"]
    assert offs[-1] == sum(ref["out_index"].shape[0] for *_, ref in vids)
    for v, (s, Xv, Qv, ref) in enumerate(vids):
        sub = {"budgets": out["budgets"][v], "count": out["count"][v:v + 1],
               "index": out["index"][offs[v]:offs[v + 1]], "tokens": out["tokens"][offs[v]:offs[v + 1]],
               "relevance": out["relevance"][v]}
        compare_condense(sub, ref, Xv.dtype)


def test_relevance_entry_point(wz):
    X, Q, _ = wl.make_video(wl.VideoSpec(T=12, H=13, W=13, D=512, Lq=7, seed=8))
    ts, fs, fm = wz.wz_relevance(X.cuda(), Q.cuda(), frame_mean=True)
    torch.cuda.synchronize()
    ref = oracle_run(X, Q, 0.1, token_frames=[])
    assert np.allclose(ts.cpu().double().numpy(), ref["a"], atol=2e-6)
    assert np.allclose(fs.cpu().double().numpy(), ref["r"], atol=2e-6)
    assert np.allclose(fm.cpu().double().numpy(), ref["vbar"], atol=1e-5)


@pytest.mark.parametrize("p,mode", [(1, "symmetric"), (4, "symmetric"), (4, "zero"), (4, "periodic"), (2, "symmetric"),
                                    (44, "symmetric"), (44, "periodic")])
def test_dwt_entry_points(wz, p, mode):
    g = torch.Generator().manual_seed(p)
    x = torch.randn((5, 27), generator=g)
    cA, cD = wz.wz_dwt1d(x.cuda(), p, mode)
    f = O.wavelet_filters(p)
    rA, rD = O.dwt1d(x.double().numpy(), f, mode, axis=1)
    assert np.allclose(cA.cpu().numpy(), rA, atol=1e-5) and np.allclose(cD.cpu().numpy(), rD, atol=1e-5)
    back = wz.wz_idwt1d(cA, cD, 27, p)
    assert np.allclose(back.cpu().numpy(), x.numpy(), atol=1e-5)
    X = torch.randn((3, 13, 10, 24), generator=g).to(torch.bfloat16)
    bands = wz.wz_dwt2d(X.cuda(), p, mode)
    ref = [O.dwt2d(X[t].double().numpy(), f, mode) for t in range(3)]
    for k in range(4):
        assert np.allclose(bands[k].cpu().numpy(), np.stack([r[k] for r in ref]), atol=1e-4)
    Y = wz.wz_idwt2d(*bands, 13, 10, p)
    torch.cuda.synchronize()
    assert np.allclose(Y.cpu().numpy(), X.float().numpy(), atol=1e-4)


def test_host_buffer_entry_point(wz):
    """wz_condense_host on pinned host buffers equals the device call."""
    X, Q = accepted_random(10, 13, 13, 128, 6, 0.2, seed=44)
    B = wz.wz_budget_size(10, 13, 13, 0.2)
    Xh, Qh = X.pin_memory(), Q.pin_memory()
    tok = torch.empty((B, 128), dtype=torch.bfloat16).pin_memory()
    idx = torch.empty((B, 3), dtype=torch.int32).pin_memory()
    wz.wz_condense_host(Xh, Qh, 0.2, tok, idx)
    torch.cuda.synchronize()
    ref = run(wz, X, Q, 0.2)
    assert torch.equal(tok, ref["tokens"].cpu()) and torch.equal(idx, ref["index"].cpu())
    with pytest.raises(ValueError):
        wz.wz_condense_host(X.cuda(), Qh, 0.2, tok, idx)
