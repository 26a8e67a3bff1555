"""The condensation pass captured in a CUDA graph (stream capture of the C ABI
call with a caller workspace) replays to the same results as direct calls,
bit for bit, for new inputs written into the captured buffers."""

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
