"""The condensation pass captured in a CUDA graph replays to the same results
as direct launches, bit for bit, for new inputs written into the captured
buffers: captured by the caller (stream capture around the C ABI call) and
by the library's own replay cache."""

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


def test_condense_replays_in_a_cuda_graph(wz):
    T, H, W, D, Lq, ratio = 12, 13, 13, 256, 6, 0.2
    X0, Q0 = wl.random_video(T, H, W, D, Lq, seed=1)
    X1, Q1 = wl.random_video(T, H, W, D, Lq, seed=2)
    X, Q = X0.cuda(), Q0.cuda()
    B = wz.wz_budget_size(T, H, W, ratio)
    ws = torch.empty((wz.wz_condense_workspace_size(T, H, W, D, wz.DTYPE_BF16, ratio),), dtype=torch.uint8,
                     device="cuda")
    tokens = torch.empty((B, D), dtype=torch.bfloat16, device="cuda")
    index = torch.empty((B, 3), dtype=torch.int32, device="cuda")
    status = torch.zeros((1,), dtype=torch.int32, device="cuda")
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):   # warm-up outside the capture (attributes, tensor-map driver entry)
        wz.wz_condense_ex(X, Q, ratio, workspace=ws, out_tokens=tokens, out_index=index, device_status=status,
                          stream=s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        res = wz.wz_condense_ex(X, Q, ratio, workspace=ws, out_tokens=tokens, out_index=index,
                                device_status=status, stream=s)
    for Xn, Qn in ((X1, Q1), (X0, Q0)):
        X.copy_(Xn.cuda())
        Q.copy_(Qn.cuda())
        g.replay()
        torch.cuda.synchronize()
        got_t, got_i, got_b = tokens.clone(), index.clone(), res["budgets"].clone()
        ref = wz.wz_condense_ex(Xn.cuda(), Qn.cuda(), ratio)
        torch.cuda.synchronize()
        assert torch.equal(got_b, ref["budgets"])
        assert torch.equal(got_i, ref["index"])
        assert torch.equal(got_t, ref["tokens"])
    assert int(status.item()) == 0


def _buffers(wz, T, H, W, D, ratio, V=None):
    """Caller-owned workspace, outputs and status word (the same pointers on
    every call, which is what lets the library replay its captured graph)."""
    dev = "cuda"
    if V is None:
        B = wz.wz_budget_size(T, H, W, ratio)
        wsb = wz.wz_condense_workspace_size(T, H, W, D, wz.DTYPE_BF16, ratio)
        lead = ()
    else:
        B, _ = wz.wz_batch_rows(V, T, H, W, ratio)
        wsb = wz.wz_batch_workspace_size(V, T, H, W, D, wz.DTYPE_BF16, ratio)
        lead = (V,)
    return {"workspace": torch.empty((wsb,), dtype=torch.uint8, device=dev),
            "out_tokens": torch.empty((B, D), dtype=torch.bfloat16, device=dev),
            "out_index": torch.empty((B, 3), dtype=torch.int32, device=dev),
            "out_budgets": torch.empty(lead + (T,), dtype=torch.int32, device=dev),
            "out_count": torch.empty(lead or (1,), dtype=torch.int32, device=dev),
            "out_relevance": torch.empty(lead + (T, 4), dtype=torch.float32, device=dev),
            "device_status": torch.zeros((1,), dtype=torch.int32, device=dev)}


def _assert_same(got, ref):
    for k in ("budgets", "count", "index", "tokens"):
        assert torch.equal(got[k], ref[k]), k
    # r~ is NaN on filtered frames: compare with the NaNs mapped to one value
    assert torch.equal(got["relevance"].nan_to_num(-7.0), ref["relevance"].nan_to_num(-7.0))


def _snapshot(out):
    return {k: v.clone() for k, v in out.items() if isinstance(v, torch.Tensor)}


def test_replay_cache_matches_direct_launches(wz):
    """wz_condense_ex with a caller workspace: the first call launches
    directly, the second captures the launch sequence, later ones replay it;
    every call, including replays over new contents of the same buffers,
    equals the direct launches bit for bit."""
    prev = wz.wz_graph_cache(8)["previous_capacity"]
    try:
        T, H, W, D, Lq, ratio = 16, 13, 13, 256, 8, 0.15
        vids = [wl.random_video(T, H, W, D, Lq, seed=s) for s in (11, 12, 13)]
        X = torch.empty_like(vids[0][0], device="cuda")
        Q = torch.empty_like(vids[0][1], device="cuda")
        bufs = _buffers(wz, T, H, W, D, ratio)
        before = wz.wz_graph_cache(-1)
        for rep, (Xn, Qn) in enumerate(vids + vids[:1]):
            X.copy_(Xn.cuda())
            Q.copy_(Qn.cuda())
            got = _snapshot(wz.wz_condense_ex(X, Q, ratio, **bufs))
            ref = wz.wz_condense_ex(Xn.cuda(), Qn.cuda(), ratio)   # no workspace: direct launches
            torch.cuda.synchronize()
            _assert_same(got, ref)
        after = wz.wz_graph_cache(-1)
        assert after["captures"] - before["captures"] == 1
        assert after["replays"] - before["replays"] == 2      # calls 3 and 4 (call 2 captured)
        assert int(bufs["device_status"].item()) == 0
    finally:
        wz.wz_graph_cache(prev)


def test_replay_cache_keys_every_argument(wz):
    """Arguments that differ in one option, one ratio or one buffer get a
    graph of their own; with room for one graph, alternating argument sets
    recapture and stay exact; capacity 0 launches directly."""
    prev = wz.wz_graph_cache(8)["previous_capacity"]
    try:
        T, H, W, D, Lq = 12, 16, 16, 128, 5
        Xh, Qh = wl.random_video(T, H, W, D, Lq, seed=31)
        X, Q = Xh.cuda(), Qh.cuda()
        big = _buffers(wz, T, H, W, D, 0.3)     # the largest budget of the cases below
        cases = [dict(ratio=0.2), dict(ratio=0.3), dict(ratio=0.2, lam=0.0), dict(ratio=0.2, tau=0.05),
                 dict(ratio=0.2, wsm_wavelet=2), dict(ratio=0.2, spatial_mode="saliency")]
        wz.wz_graph_cache(0)      # drop the graphs of earlier calls
        for cap in (8, 1, 0):
            wz.wz_graph_cache(cap)
            for _ in range(3):
                for kw in cases:
                    kw = dict(kw)
                    ratio = kw.pop("ratio")
                    B = wz.wz_budget_size(T, H, W, ratio)
                    bufs = dict(big, out_tokens=big["out_tokens"][:B], out_index=big["out_index"][:B])
                    got = _snapshot(wz.wz_condense_ex(X, Q, ratio, **kw, **bufs))
                    ref = wz.wz_condense_ex(X, Q, ratio, **kw)
                    torch.cuda.synchronize()
                    _assert_same(got, ref)
            st = wz.wz_graph_cache(-1)
            assert st["kept"] == min(cap, len(cases))
        assert int(big["device_status"].item()) == 0
    finally:
        wz.wz_graph_cache(prev)


def test_replay_cache_serving_batch(wz):
    """wz_condense_batch through the replay cache equals direct launches."""
    prev = wz.wz_graph_cache(8)["previous_capacity"]
    try:
        V, T, H, W, D = 4, 8, 13, 13, 256
        Lqs, ratios = [3, 9, 5, 16], [0.1, 0.2, 0.05, 0.3]
        vids = [wl.random_video(T, H, W, D, lq, seed=40 + v) for v, lq in enumerate(Lqs)]
        X = torch.stack([x for x, _ in vids]).cuda()
        Qs = torch.cat([q for _, q in vids]).cuda()
        bufs = _buffers(wz, T, H, W, D, ratios, V=V)
        before = wz.wz_graph_cache(-1)
        for _ in range(3):
            got = _snapshot(wz.wz_condense_batch(X, Qs, Lqs, ratios, **bufs))
            ref = wz.wz_condense_batch(X, Qs, Lqs, ratios)
            torch.cuda.synchronize()
            _assert_same(got, ref)
        after = wz.wz_graph_cache(-1)
        assert after["captures"] - before["captures"] == 1 and after["replays"] - before["replays"] == 1
    finally:
        wz.wz_graph_cache(prev)
