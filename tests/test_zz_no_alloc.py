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


def test_static_scores_match_the_workspace_entry_point_twice(wz):
    cases = [wl.VideoSpec(T=24, H=13, W=13, D=512, Lq=9, seed=31),
             wl.VideoSpec(T=40, H=16, W=16, D=896, Lq=3, seed=32)]
    for spec in cases:                      # two calls in a row, different sizes
        X, Q, _ = wl.make_video(spec)
        Xc, Qc = X.cuda(), Q.cuda()
        got = wz.wz_relevance_static(Xc, Qc, frame_mean=True)
        ref = wz.wz_relevance(Xc, Qc, frame_mean=True)
        torch.cuda.synchronize()
        for g, r in zip(got, ref):
            assert np.allclose(g.cpu().double().numpy(), r.cpu().double().numpy(), atol=2e-6, rtol=0)


def test_static_rejects_sizes_beyond_its_array(wz):
    X = torch.zeros((2048, 4, 4, 4096), dtype=torch.bfloat16, device="cuda")
    Q = torch.zeros((1, 4096), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(wz.WaveZipError) as e:
        wz.wz_relevance_static(X, Q)
    assert e.value.status == wz.ERR_WORKSPACE
