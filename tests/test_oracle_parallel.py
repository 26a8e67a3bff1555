"""The frame-parallel driver of the oracle (the second CPU baseline) gives the
oracle's own result: same budgets and index map, tokens to 1e-12."""

import numpy as np
import torch

import oracle as O
import workload as wl
from oracle.parallel import condense_parallel, condense_videos_parallel, spawn_pool


def test_parallel_driver_matches_the_oracle():
    spec = wl.VideoSpec(T=12, H=9, W=11, D=64, Lq=5, ratio=0.2, ar=0.9, cuts=2, seed=5)
    X, Q, _ = wl.make_video(spec)
    bits = X.view(torch.int16).numpy().view(np.uint16)
    ref = O.condense(X.double().numpy(), Q.double().numpy(), spec.ratio)
    got = condense_parallel(bits, Q.double().numpy(), spec.ratio, workers=2, frames_per_job=3)
    assert np.array_equal(got["budgets"], ref["budgets"])
    assert np.array_equal(got["out_index"], ref["out_index"])
    assert np.allclose(got["out_tokens"], ref["out_tokens"], rtol=0, atol=1e-12)
    assert np.allclose(got["r"], ref["r"], rtol=0, atol=1e-14)


def test_video_pool_driver_matches_the_oracle(tmp_path):
    specs = [wl.VideoSpec(T=6, H=5, W=7, D=32, Lq=lq, ratio=r, ar=0.9, cuts=1, seed=40 + v)
             for v, (lq, r) in enumerate([(3, 0.2), (5, 0.5)])]
    vids = [wl.make_video(s)[:2] for s in specs]
    path = str(tmp_path / "x.npy")
    np.save(path, np.stack([X.view(torch.int16).numpy().view(np.uint16) for X, _ in vids]))
    pool = spawn_pool(2)
    try:
        got = condense_videos_parallel(path, [Q.double().numpy() for _, Q in vids], [s.ratio for s in specs], pool)
    finally:
        pool.terminate()
    for (X, Q), s, g in zip(vids, specs, got):
        ref = O.condense(X.double().numpy(), Q.double().numpy(), s.ratio)
        assert np.array_equal(g["budgets"], ref["budgets"])
        assert np.array_equal(g["out_index"], ref["out_index"])
        assert np.allclose(g["out_tokens"], ref["out_tokens"], rtol=0, atol=1e-12)
