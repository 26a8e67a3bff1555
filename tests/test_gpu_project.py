"""Projector P (Eq. 17) on the tensor cores vs the CPU oracle, through the C ABI.

Tolerance, from the arithmetic: bf16 operands are exact in both; the GPU
accumulates in fp32 (relative error ~ sqrt(K) 2^-24, far below bf16), the
hidden layer is rounded to bf16 on both sides (a rounding decision can flip
only where fp32 and fp64 straddle a bf16 midpoint, which moves one hidden
value by one bf16 ulp), and the output is rounded to bf16 (2^-8 relative).
So |g - o| <= 1e-2 |o| + 1e-3 max|o| with the oracle rounded to bf16.
"""

import numpy as np
import pytest
import torch

import oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def wz():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2607_23265_gb300.wavezip as m
    assert torch.cuda.is_available()
    return m


def _case(B, D, C, E, seed, bias=True):
    g = torch.Generator().manual_seed(seed)
    Z = torch.randn((B, D), generator=g).to(torch.bfloat16)
    W1 = (torch.randn((C, D), generator=g) / D ** 0.5).to(torch.bfloat16)
    W2 = (torch.randn((E, C), generator=g) / C ** 0.5).to(torch.bfloat16)
    b1 = (0.1 * torch.randn((C,), generator=g)).float() if bias else None
    b2 = (0.1 * torch.randn((E,), generator=g)).float() if bias else None
    return Z, W1, b1, W2, b2


def _check(got, ref):
    ref = O.round_bf16(ref)
    got = got.double().numpy()
    err = np.abs(got - ref)
    bound = 1e-2 * np.abs(ref) + 1e-3 * np.abs(ref).max()
    assert np.all(err <= bound), f"max |d| {err.max():.3e} at {np.unravel_index(err.argmax(), err.shape)}"


def _np(t):
    return None if t is None else t.double().numpy()


@pytest.mark.parametrize("B,D,C,E,bias", [
    (200, 128, 256, 192, True),    # ragged M tile, partial N tile
    (129, 256, 512, 256, False),   # one row past a tile, no biases
    (1, 64, 64, 64, True),         # smallest
    (300, 1024, 320, 448, True),   # 16 K steps, N tiles of 256 + 64
])
def test_project_parity(wz, B, D, C, E, bias):
    Z, W1, b1, W2, b2 = _case(B, D, C, E, seed=B + D, bias=bias)
    out = wz.wz_project(Z.cuda(), W1.cuda(), None if b1 is None else b1.cuda(), W2.cuda(),
                        None if b2 is None else b2.cuda())
    torch.cuda.synchronize()
    ref = O.project(_np(Z), _np(W1), _np(b1), _np(W2), _np(b2))
    _check(out.cpu(), ref)


def test_project_full_size_sampled_rows(wz):
    # the 256-frame workload's output size: 18,662 condensed tokens of 3584 channels
    B, D = 18662, 3584
    Z, W1, b1, W2, b2 = _case(B, D, D, D, seed=7)
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    ws = torch.empty(wz.wz_project_workspace_size(B, D), dtype=torch.uint8, device="cuda")
    out = wz.wz_project(Z.cuda(), W1.cuda(), b1.cuda(), W2.cuda(), b2.cuda(), workspace=ws, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    rows = np.array([0, 1, 127, 128, 5000, 9331, 18560, 18661])
    ref = O.project(_np(Z)[rows], _np(W1), _np(b1), _np(W2), _np(b2))
    _check(out.cpu()[rows], ref)


def test_project_argument_errors(wz):
    Z, W1, b1, W2, b2 = _case(4, 64, 64, 64, seed=1)
    with pytest.raises(ValueError):
        wz.wz_project(Z.cuda(), W1.cuda(), b1.cuda(), W2[:, :32].contiguous().cuda(), b2.cuda())
    Zb = torch.randn((4, 96)).to(torch.bfloat16).cuda()           # D not a multiple of 64
    W1b = torch.randn((64, 96)).to(torch.bfloat16).cuda()
    with pytest.raises(wz.WaveZipError):
        wz.wz_project(Zb, W1b, None, W2.cuda(), None)
