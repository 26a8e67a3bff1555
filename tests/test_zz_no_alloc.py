"""wz_relevance_static, the relevance entry point that allocates nothing.

It serves callers that may not allocate device memory at call time (graph
capture without allocation nodes, fixed-budget serving loops, hosts whose
memory belongs to another allocator).  Its scores must equal those of
wz_relevance; two calls in a row check that the shared fixed array carries
nothing over from one call to the next.  This file is collected last.
"""

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


def _same(got, ref):
    for g, r in zip(got, ref):
        if r is None:
            assert g is None
        else:
            assert np.allclose(g.cpu().double().numpy(), r.cpu().double().numpy(), atol=2e-6, rtol=0)


@pytest.mark.parametrize("dtype,frame_mean", [("bf16", True), ("bf16", False), ("f32", True)])
def test_static_scores_match_the_workspace_entry_point_twice(wz, dtype, frame_mean):
    cases = [wl.VideoSpec(T=24, H=13, W=13, D=512, Lq=9, dtype=dtype, seed=31),
             wl.VideoSpec(T=40, H=16, W=16, D=896, Lq=3, dtype=dtype, seed=32)]
    for spec in cases:                      # two calls in a row, different sizes
        X, Q, _ = wl.make_video(spec)
        Xc, Qc = X.cuda(), Q.cuda()
        got = wz.wz_relevance_static(Xc, Qc, frame_mean=frame_mean)
        ref = wz.wz_relevance(Xc, Qc, frame_mean=frame_mean)
        torch.cuda.synchronize()
        _same(got, ref)


def test_static_call_allocates_no_device_memory(wz):
    X, Q, _ = wl.make_video(wl.VideoSpec(T=16, H=13, W=13, D=512, Lq=5, seed=33))
    Xc, Qc = X.cuda(), Q.cuda()
    out = (torch.empty((16, 169), device="cuda"), torch.empty((16,), device="cuda"),
           torch.empty((16, 512), device="cuda"))
    status = torch.zeros((1,), dtype=torch.int32, device="cuda")
    wz.wz_relevance_static(Xc, Qc, out=out, device_status=status)   # loads the kernels, looks the array up
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    for _ in range(3):
        wz.wz_relevance_static(Xc, Qc, out=out, device_status=status)
        wz.wz_relevance_static(Xc, Qc, out=out)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert int(status.item()) == 0
    _same(out, wz.wz_relevance(Xc, Qc, frame_mean=True))


def test_static_status_word_and_checked_build(wz):
    """Two calls report no failure in the caller's status word; the
    bounds-checked build (index tests on every global write, its own fixed
    array) sets no bit and gives the same scores, with or without a caller
    status word."""
    X, Q, _ = wl.make_video(wl.VideoSpec(T=20, H=13, W=13, D=512, Lq=4, seed=34))
    Xc, Qc = X.cuda(), Q.cuda()
    status = torch.zeros((1,), dtype=torch.int32, device="cuda")
    first = wz.wz_relevance_static(Xc, Qc, frame_mean=True, device_status=status)
    second = wz.wz_relevance_static(Xc, Qc, frame_mean=True, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    for x, y in zip(first, second):
        assert torch.equal(x, y)
    with wz.checked_library():
        cst = torch.zeros((1,), dtype=torch.int32, device="cuda")
        a = wz.wz_relevance_static(Xc, Qc, frame_mean=True, device_status=cst)
        b = wz.wz_relevance_static(Xc, Qc, frame_mean=True)
        torch.cuda.synchronize()
    assert int(cst.item()) == 0
    _same(a, first)
    _same(b, first)


def test_static_rejects_sizes_beyond_its_array(wz):
    X = torch.zeros((2048, 4, 4, 4096), dtype=torch.bfloat16, device="cuda")
    Q = torch.zeros((1, 4096), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(wz.WaveZipError) as e:
        wz.wz_relevance_static(X, Q)
    assert e.value.status == wz.ERR_WORKSPACE
