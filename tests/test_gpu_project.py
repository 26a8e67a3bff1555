"""Projector P (Eq. 17) on the tensor cores vs the CPU oracle, through the C ABI.

Checked element by element in two stages, with tolerances from the arithmetic.
The call leaves its bf16 hidden layer h in the caller's workspace (as the
header states), so each layer is checked on its own:

- Hidden layer: bf16 operands are exact on both sides; the GPU accumulates the
  first layer in fp32, whose worst-case error is 2^-24 (D + 1) times the sum
  of the magnitudes of the terms (sum_d |z_d W1[c,d]| + |b1_c|), times GELU's
  largest slope 1.13, plus 2^-14 relative and |x| 2^-22 absolute for the fp32
  GELU (x (1 + erff(x / sqrt 2)) / 2 cancels in the negative tail): call that
  e_c.  Both sides then round to bf16 (half an ulp each), so
  |h_gpu - h_oracle| <= e_c + 2^-7 max|h| per element.
- Output, from the GPU's own hidden layer: the second layer's fp32 error is at
  most 2^-24 (C + 1) S_e with S_e = sum_c |W2[e,c] h_c| + |b2_e|, and both
  sides round to bf16 (one ulp, <= 2^-7 |o|; 1e-2 |o| allowed).  So
  |g - o| <= 1e-2 |o| + 2^-24 (C + 1) S_e + 1e-6 per element.
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


def _hidden_ok(hg, Z, W1, b1):
    """The GPU's bf16 hidden layer against the oracle's, element by element."""
    pre = Z @ W1.T + (0.0 if b1 is None else b1[None, :])
    mass = np.abs(Z) @ np.abs(W1).T + (0.0 if b1 is None else np.abs(b1)[None, :])
    g = O.gelu(pre)
    h = O.round_bf16(g)
    e = np.abs(g) * 2.0 ** -14 + np.abs(pre) * 2.0 ** -22 + 1.13 * 2.0 ** -24 * (Z.shape[1] + 1) * mass
    bound = e + 2.0 ** -7 * np.maximum(np.abs(h), np.abs(hg))
    bad = np.abs(hg - h) > bound
    assert not bad.any(), f"hidden layer: {bad.sum()} values off, first at {np.argwhere(bad)[0]}"


def _check(got, hg, W2, b2):
    """The output against the oracle's second layer applied to the GPU's hidden layer."""
    o = O.round_bf16(hg @ W2.T + (0.0 if b2 is None else b2[None, :]))
    S = np.abs(hg) @ np.abs(W2).T + (0.0 if b2 is None else np.abs(b2)[None, :])
    got = got.double().numpy()
    err = np.abs(got - o)
    bound = 1e-2 * np.abs(o) + 2.0 ** -24 * (W2.shape[1] + 1) * S + 1e-6
    assert np.all(err <= bound), f"max |d| {err.max():.3e} at {np.unravel_index(err.argmax(), err.shape)}"


def _run(wz, Z, W1, b1, W2, b2):
    """wz_project with a caller workspace; returns (out, hidden layer) on the host."""
    B, C = Z.shape[0], W1.shape[0]
    ws = torch.empty(wz.wz_project_workspace_size(B, C), dtype=torch.uint8, device="cuda")
    status = torch.zeros(1, dtype=torch.int32, device="cuda")
    out = wz.wz_project(Z.cuda(), W1.cuda(), None if b1 is None else b1.cuda(), W2.cuda(),
                        None if b2 is None else b2.cuda(), workspace=ws, device_status=status)
    torch.cuda.synchronize()
    assert int(status.item()) == 0
    hidden = ws[:B * C * 2].view(torch.bfloat16).view(B, C).cpu()
    return out.cpu(), hidden


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
    out, hidden = _run(wz, Z, W1, b1, W2, b2)
    hg = _np(hidden)
    _hidden_ok(hg, _np(Z), _np(W1), _np(b1))
    _check(out, hg, _np(W2), _np(b2))


def test_project_full_size_sampled_rows(wz):
    # the 256-frame workload's output size: 18,662 condensed tokens of 3584 channels
    B, D = 18662, 3584
    Z, W1, b1, W2, b2 = _case(B, D, D, D, seed=7)
    out, hidden = _run(wz, Z, W1, b1, W2, b2)
    rows = np.array([0, 1, 127, 128, 5000, 9331, 18560, 18661])
    hg = _np(hidden)[rows]
    _hidden_ok(hg, _np(Z)[rows], _np(W1), _np(b1))
    _check(out[rows], hg, _np(W2), _np(b2))


def test_project_argument_errors(wz):
    Z, W1, b1, W2, b2 = _case(4, 64, 64, 64, seed=1)
    with pytest.raises(ValueError):
        wz.wz_project(Z.cuda(), W1.cuda(), b1.cuda(), W2[:, :32].contiguous().cuda(), b2.cuda())
    Zb = torch.randn((4, 96)).to(torch.bfloat16).cuda()           # D not a multiple of 64
    W1b = torch.randn((64, 96)).to(torch.bfloat16).cuda()
    with pytest.raises(wz.WaveZipError):
        wz.wz_project(Zb, W1b, None, W2.cuda(), None)
