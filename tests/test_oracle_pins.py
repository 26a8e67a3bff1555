"""Pins of the CPU oracle to facts outside itself (no GPU needed).

Each check is a function of the oracle module so that the mutation tests at
the end can re-run it against a copy of the oracle with a planted mistake and
see it fail.  Pins used: published filter taps, closed forms of the Haar
transform, perfect reconstruction, vanishing moments, library routines
(numpy convolution, torch adaptive pooling and bilinear interpolation),
brute-force apportionment on tiny inputs, and invariants of the method.
"""

import itertools
import math
import os
import types

import numpy as np
import pytest
import torch

import oracle as O
from oracle import wavezip_oracle as OM

RNG = np.random.default_rng(12345)
SQ2 = math.sqrt(2.0)


def _golden(path):
    rows = []
    with open(path) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append([float(v) for v in line.split()])
    return rows


# ----------------------------------------------------------------------------
# Filters
# ----------------------------------------------------------------------------

def check_haar_filter(o):
    h = o.daubechies_lowpass(1)
    assert h.shape == (2,)
    assert np.allclose(h, [1 / SQ2, 1 / SQ2], atol=1e-15)


def check_db2_closed_form(o, golden_dir):
    rows = _golden(os.path.join(golden_dir, "db2_closed_form.txt"))
    ref = np.array([(a + b * math.sqrt(3.0)) / (4 * SQ2) for a, b in rows])
    assert np.allclose(o.daubechies_lowpass(2), ref, atol=1e-14)


def check_db4_table(o, golden_dir):
    ref = np.array([r[0] for r in _golden(os.path.join(golden_dir, "db4_taps.txt"))])
    assert np.allclose(o.wavelet_filters(4)["rec_lo"], ref, atol=6e-11)


def check_filter_identities(o, p):
    f = o.wavelet_filters(p)
    h, g, F = f["rec_lo"], f["rec_hi"], f["F"]
    assert F == 2 * p
    assert abs(h.sum() - SQ2) < 1e-12
    assert abs((h * h).sum() - 1.0) < 1e-12
    for m in range(1, p):                       # orthogonal to even shifts
        assert abs(np.dot(h[2 * m:], h[:F - 2 * m])) < 1e-12
    assert abs(np.dot(h, g)) < 1e-12            # low/high orthogonal
    k = np.arange(F, dtype=np.float64)
    for j in range(p):                          # vanishing moments of the wavelet
        assert abs(np.dot(k ** j, g)) < 1e-9 * max(1.0, float((k ** j).max()))
    # analysis filters are the time reverses of the synthesis filters
    assert np.array_equal(f["dec_lo"], h[::-1]) and np.array_equal(f["dec_hi"], g[::-1])
    # minimum phase: after dividing out the p-fold zero at z = -1, every zero of
    # sum h[k] z^(F-1-k) lies strictly inside the unit circle
    quot, rem = np.polydiv(h, np.poly([-1.0] * p))
    assert np.abs(rem).max() < 1e-10
    if quot.size > 1:
        assert np.all(np.abs(np.roots(quot)) < 1.0)


def test_haar_filter():
    check_haar_filter(O)


def test_db2_closed_form(golden_dir):
    check_db2_closed_form(O, golden_dir)


def test_db4_published_taps(golden_dir):
    check_db4_table(O, golden_dir)


def check_bior44_published(o, golden_dir):
    rows = _golden(os.path.join(golden_dir, "cdf97_taps.txt"))
    f = o.wavelet_filters(o.BIOR44)
    assert f["F"] == 10
    ana = f["dec_lo"][1:10] / math.sqrt(2.0)             # DC gain 1, 9 taps
    syn = f["rec_lo"][1:8] * math.sqrt(2.0)              # DC gain 2, 7 taps
    for taps, row in ((ana, rows[0]), (syn, rows[1])):
        c = taps.size // 2
        for k, v in enumerate(row):
            assert abs(taps[c + k] - v) < 1e-12 and abs(taps[c - k] - v) < 1e-12


def test_bior44_published_taps(golden_dir):
    check_bior44_published(O, golden_dir)


def test_bior44_biorthogonality_and_moments():
    f = O.wavelet_filters(O.BIOR44)
    F = f["F"]
    # analysis and synthesis lowpass are dual: sum_k h~[k] h[k + 2m] = delta_m
    # (as z-transforms aligned by the layout); checked through perfect
    # reconstruction of every length and of shifted impulses
    for n in (1, 2, 3, 4, 7, 16, 27, 33):
        for mode in ("symmetric", "periodic", "zero"):
            if mode == "periodic" and n < 2:
                continue
            x = RNG.standard_normal(n)
            A, D = O.dwt1d(x, f, mode)
            assert np.allclose(O.idwt1d(A, D, n, f), x, atol=1e-12) or mode == "zero"
    # four vanishing moments on both sides
    k = np.arange(F, dtype=np.float64)
    for hp in (f["dec_hi"], f["rec_hi"]):
        for m in range(4):
            assert abs(np.sum(hp * k ** m)) < 1e-9 * (F ** m)


@pytest.mark.parametrize("p", [1, 2, 3, 4, 5, 6, 8])
def test_filter_identities(p):
    check_filter_identities(O, p)


# ----------------------------------------------------------------------------
# DWT / IDWT
# ----------------------------------------------------------------------------

def check_haar_1d_closed_forms(o):
    f = o.wavelet_filters(1)
    a, b, c, d = 3.0, -1.0, 0.5, 2.0
    cA, cD = o.dwt1d(np.array([a, b]), f)
    assert np.allclose(cA, [(a + b) / SQ2]) and np.allclose(cD, [(a - b) / SQ2])
    cA, cD = o.dwt1d(np.array([a, b, c, d]), f)
    assert np.allclose(cA, [(a + b) / SQ2, (c + d) / SQ2])
    assert np.allclose(cD, [(a - b) / SQ2, (c - d) / SQ2])
    # odd length: the last sample pairs with its mirror image
    cA, cD = o.dwt1d(np.array([a, b, c]), f)
    assert np.allclose(cA, [(a + b) / SQ2, 2 * c / SQ2]) and np.allclose(cD, [(a - b) / SQ2, 0.0])


def check_haar_2d_closed_forms(o):
    f = o.wavelet_filters(1)
    X = np.array([[1.0, 4.0], [-2.0, 0.5]])
    a, b, c, d = X.ravel()
    LL, LH, HL, HH = o.dwt2d(X, f)
    assert np.allclose(LL, [[(a + b + c + d) / 2]])
    assert np.allclose(LH, [[(a - b + c - d) / 2]])   # height low, width high
    assert np.allclose(HL, [[(a + b - c - d) / 2]])
    assert np.allclose(HH, [[(a - b - c + d) / 2]])
    X4 = RNG.standard_normal((4, 4))
    LL, LH, HL, HH = o.dwt2d(X4, f)
    for i in range(2):
        for j in range(2):
            a, b = X4[2 * i, 2 * j], X4[2 * i, 2 * j + 1]
            c, d = X4[2 * i + 1, 2 * j], X4[2 * i + 1, 2 * j + 1]
            assert np.isclose(LL[i, j], (a + b + c + d) / 2)
            assert np.isclose(LH[i, j], (a - b + c - d) / 2)
            assert np.isclose(HL[i, j], (a + b - c - d) / 2)
            assert np.isclose(HH[i, j], (a - b - c + d) / 2)


def check_dwt_vs_numpy_convolution(o, p, mode, n):
    """cA/cD equal the full convolution of the padded signal, every second sample."""
    f = o.wavelet_filters(p)
    F = f["F"]
    x = RNG.standard_normal(n)
    padmode = {"symmetric": "symmetric", "periodic": "wrap", "zero": "constant"}[mode]
    if padmode == "wrap" and F - 1 > n:
        xp = np.array([x[i % n] for i in range(-(F - 1), n + F - 1)])
    else:
        xp = np.pad(x, F - 1, mode=padmode)
    L = o.dwt_len(n, F)
    refA = np.convolve(xp, f["dec_lo"])[F::2][:L]
    refD = np.convolve(xp, f["dec_hi"])[F::2][:L]
    cA, cD = o.dwt1d(x, f, mode)
    assert np.allclose(cA, refA, atol=1e-12) and np.allclose(cD, refD, atol=1e-12)


def check_perfect_reconstruction(o, p, mode, n):
    f = o.wavelet_filters(p)
    x = RNG.standard_normal((n, 3))
    cA, cD = o.dwt1d(x, f, mode)
    assert cA.shape[0] == (n + f["F"] - 1) // 2
    y = o.idwt1d(cA, cD, n, f)
    assert np.abs(y - x).max() < 1e-12


def check_pr_2d(o, p, H, W):
    f = o.wavelet_filters(p)
    X = RNG.standard_normal((H, W, 2))
    bands = o.dwt2d(X, f)
    assert np.abs(o.idwt2d(*bands, H, W, f) - X).max() < 1e-12


def check_constant_map_details_vanish(o, p, H, W):
    f = o.wavelet_filters(p)
    X = np.full((H, W, 3), 1.75)
    LL, LH, HL, HH = o.dwt2d(X, f, "symmetric")
    assert max(np.abs(LH).max(), np.abs(HL).max(), np.abs(HH).max()) < 1e-13
    assert np.allclose(LL, 1.75 * 2.0)          # each axis scales a constant by sum h = sqrt 2


def check_polynomial_interior_details_vanish(o, p):
    """Interior detail coefficients of a degree < p polynomial are 0."""
    f = o.wavelet_filters(p)
    F = f["F"]
    n = 40
    t = np.arange(n, dtype=np.float64)
    x = sum(c * t ** j for j, c in enumerate([0.3, 0.2, -0.01, 1e-4][:p]))
    _, cD = o.dwt1d(x, f, "symmetric")
    interior = [i for i in range(cD.size) if 2 * i + 1 - (F - 1) >= 0 and 2 * i + 1 < n]
    assert interior and np.abs(cD[interior]).max() < 1e-9


def test_haar_1d_closed_forms():
    check_haar_1d_closed_forms(O)


def test_haar_2d_closed_forms():
    check_haar_2d_closed_forms(O)


@pytest.mark.parametrize("mode", ["symmetric", "periodic", "zero"])
@pytest.mark.parametrize("p,n", [(1, 7), (2, 9), (4, 27), (4, 13), (4, 5), (4, 2), (6, 16)])
def test_dwt_vs_numpy_convolution(p, mode, n):
    check_dwt_vs_numpy_convolution(O, p, mode, n)


@pytest.mark.parametrize("mode", ["symmetric", "periodic", "zero"])
@pytest.mark.parametrize("p", [1, 2, 4])
def test_perfect_reconstruction_1d(p, mode):
    for n in range(1, 33):
        check_perfect_reconstruction(O, p, mode, n)


@pytest.mark.parametrize("p,H,W", [(4, 27, 27), (4, 13, 13), (4, 14, 14), (4, 16, 16), (4, 3, 5),
                                   (4, 1, 6), (1, 6, 7), (2, 9, 4)])
def test_perfect_reconstruction_2d(p, H, W):
    check_pr_2d(O, p, H, W)


@pytest.mark.parametrize("p,H,W", [(4, 27, 27), (4, 5, 3), (1, 4, 4), (2, 7, 9)])
def test_constant_map_details_vanish(p, H, W):
    check_constant_map_details_vanish(O, p, H, W)


@pytest.mark.parametrize("p", [2, 3, 4])
def test_polynomial_interior_details_vanish(p):
    check_polynomial_interior_details_vanish(O, p)


# ----------------------------------------------------------------------------
# Pooling and interpolation against torch routines
# ----------------------------------------------------------------------------

def check_adaptive_pool(o, H, W, oh, ow):
    M = RNG.random((H, W))
    ref = torch.nn.functional.adaptive_avg_pool2d(torch.from_numpy(M)[None, None], (oh, ow))[0, 0]
    assert np.allclose(o.adaptive_avg_pool2d(M, oh, ow), ref.numpy(), atol=1e-14)


def check_bilinear(o, H, W, h, w):
    X = RNG.standard_normal((H, W, 3))
    ref = torch.nn.functional.interpolate(torch.from_numpy(X).permute(2, 0, 1)[None], size=(h, w),
                                          mode="bilinear", align_corners=False, antialias=False)
    ref = ref[0].permute(1, 2, 0).numpy()
    assert np.allclose(o.bilinear_resize(X, h, w), ref, atol=1e-12)


@pytest.mark.parametrize("H,W,oh,ow", [(27, 27, 17, 17), (13, 13, 10, 10), (14, 14, 10, 10),
                                       (16, 16, 11, 11), (3, 5, 5, 6), (7, 2, 3, 4), (1, 1, 4, 4)])
def test_adaptive_pool_matches_torch(H, W, oh, ow):
    check_adaptive_pool(O, H, W, oh, ow)


@pytest.mark.parametrize("H,W,h,w", [(27, 27, 9, 9), (27, 27, 10, 8), (13, 13, 5, 4), (14, 14, 7, 7),
                                     (16, 16, 16, 16), (3, 5, 7, 2), (27, 27, 1, 1), (5, 1, 3, 1)])
def test_bilinear_matches_torch(H, W, h, w):
    check_bilinear(O, H, W, h, w)


def test_psi_special_cases():
    X = RNG.standard_normal((6, 8, 2))
    tok, idx = O.psi(X, 48)                              # n = N: identity
    assert np.allclose(tok, X.reshape(48, 2)) and idx[9] == (1, 1)
    tok, _ = O.psi(X, 12)                                # h = H/2, w = W/2: 2x2 means
    pooled = X.reshape(3, 2, 4, 2, 2).mean(axis=(1, 3)).reshape(12, 2)
    assert O.grid_shape(12, 6, 8) == (3, 4)
    assert np.allclose(tok, pooled)


def test_grid_shape_definition():
    from fractions import Fraction
    for H in range(1, 12):
        for W in range(1, 12):
            for n in range(1, H * W + 1):
                h, w = O.grid_shape(n, H, W)
                x = Fraction(n * H, W)
                hc = 1
                while hc * hc < x:
                    hc += 1
                assert h == min(H, hc)
                assert w == -(-n // h) and h * w >= n and w <= W


# ----------------------------------------------------------------------------
# Scorer, VCE, filter
# ----------------------------------------------------------------------------

def test_cosine_closed_forms():
    assert np.isclose(O.cosine(np.array([1.0, 0.0]), np.array([1.0, 1.0])), 1 / SQ2)
    assert O.cosine(np.zeros(3), np.ones(3)) == 0.0
    U = np.array([[3.0, 4.0], [0.0, 0.0], [-1.0, 0.0]])
    a = O.token_saliency(U, np.array([1.0, 0.0]))
    assert np.allclose(a, [0.6, 0.0, -1.0])


def test_scores_scale_invariant():
    X = RNG.standard_normal((4, 3, 3, 16))
    Q = RNG.standard_normal((5, 16))
    r1 = O.condense(X, Q, 0.5, token_frames=[])
    r2 = O.condense(2.5 * X, 0.1 * Q, 0.5, token_frames=[])
    assert np.allclose(r1["a"], r2["a"]) and np.allclose(r1["r"], r2["r"])
    assert np.array_equal(r1["budgets"], r2["budgets"])


def test_frame_relevance_pools_before_cosine():
    U = np.array([[1.0, 0.0], [0.0, 1.0]])
    r, vbar = O.frame_relevance(U, np.array([1.0, 1.0]))
    assert np.allclose(vbar, [0.5, 0.5]) and np.isclose(r, 1.0)
    # the mean of the token cosines would be 1/sqrt2, not 1


def test_visual_change_cases():
    v = RNG.standard_normal(8)
    w = RNG.standard_normal(8)
    w -= np.dot(w, v) / np.dot(v, v) * v                 # orthogonal to v
    vbar = np.stack([v, v, -v, -v, w, w])
    delta, gamma = O.visual_change(vbar)
    assert np.allclose(delta, [0, 0, 2, 0, 1, 0], atol=1e-12)
    assert np.allclose(gamma, [0, 0, 1, 0, 0.5, 0], atol=1e-12)
    d2, g2 = O.visual_change(np.stack([v, v, v]))
    assert np.allclose(d2, 0) and np.all(g2 == 0)


def test_frame_filter():
    delta = np.array([0.0, 0.01, 0.5, 0.02, 0.3])
    assert O.frame_filter(delta, 0.0) == [0, 1, 2, 3, 4]
    assert O.frame_filter(delta, 0.05) == [0, 2, 4]
    assert O.frame_filter(delta, 10.0) == [0]


# ----------------------------------------------------------------------------
# WTA (Eq. 8-10)
# ----------------------------------------------------------------------------

def check_wta_closed_form(o):
    r = np.array([0.3, 0.1, -0.2, 0.4, 0.05])
    g = np.array([0.0, 1.0, 0.25, 0.75, 0.6])
    out = o.wta(r, g)
    for k in range(2):
        mu = 0.5 * (r[2 * k] + r[2 * k + 1])
        dl = 0.5 * (r[2 * k] - r[2 * k + 1])
        gb = 0.5 * (g[2 * k] + g[2 * k + 1])
        assert np.isclose(out[2 * k], mu + gb * dl) and np.isclose(out[2 * k + 1], mu - gb * dl)
    assert np.isclose(out[4], r[4])                      # odd tail passes through
    assert np.allclose(o.wta(r, np.ones(5)), r)          # gate 1: perfect reconstruction
    pm = o.wta(r[:4], np.zeros(4))
    assert np.allclose(pm, [0.2, 0.2, 0.1, 0.1])          # gate 0: pair means


def test_wta_closed_form():
    check_wta_closed_form(O)


@pytest.mark.parametrize("p", [2, 4, 10])
def test_wta_daubechies_unit_gate_is_identity(p):
    r = RNG.standard_normal(23)
    assert np.allclose(O.wta(r, np.ones(23), p), r, atol=1e-12)      # perfect reconstruction


@pytest.mark.parametrize("p", [2, 4])
def test_wta_daubechies_zero_gate_keeps_smooth_signals(p):
    # a polynomial of degree < p has no detail away from the borders, so the
    # gate cannot change the interior of the rectified sequence
    x = np.arange(40, dtype=np.float64)
    r = 0.3 + 0.01 * x - (0.0002 * x * x if p > 2 else 0.0)
    out = O.wta(r, np.zeros(40), p)
    assert np.allclose(out[2 * p:-2 * p], r[2 * p:-2 * p], atol=1e-9)


def test_wta_two_element():
    out = O.wta(np.array([1.0, 0.0]), np.array([0.0, 0.5]))
    assert np.allclose(out, [0.5 + 0.25 * 0.5, 0.5 - 0.25 * 0.5])


def test_wta_length_one():
    assert np.allclose(O.wta(np.array([0.7]), np.array([0.0])), [0.7])


# ----------------------------------------------------------------------------
# Budgets (Eq. 5, Eq. 15)
# ----------------------------------------------------------------------------

def test_global_budget_rounding():
    assert O.global_budget(0.1, 64, 169) == 1082          # 1081.6
    assert O.global_budget(0.1, 256, 729) == 18662         # 18662.4
    assert O.global_budget(0.25, 16, 196) == 784
    assert O.global_budget(0.5, 1, 3) == 2                 # 1.5 rounds away from zero
    assert O.global_budget(1.0, 7, 9) == 63


def check_budget_brute_force(o, L, B, N, seed):
    rng = np.random.default_rng(seed)
    r = rng.uniform(-0.2, 1.0, size=L)
    n, _ = o.allocate_budget(r, B, N)
    assert n.sum() == min(B, L * N) and n.min() >= 0 and n.max() <= N
    w = np.maximum(r, 0)
    if w.sum() == 0:
        w = np.ones(L)
    q = B * w / w.sum()
    if np.any(q > N) or B >= L * N:
        return
    best = None
    for cand in itertools.product(range(N + 1), repeat=L):
        if sum(cand) != B:
            continue
        cost = float(np.sum((np.array(cand) - q) ** 2))
        if best is None or cost < best - 1e-12:
            best, arg = cost, [cand]
        elif abs(cost - best) <= 1e-12:
            arg.append(cand)
    assert tuple(int(v) for v in n) in arg


def test_budget_brute_force():
    for seed in range(60):
        L = 2 + seed % 3
        N = 3 + seed % 4
        B = 1 + (seed * 7) % (L * N)
        check_budget_brute_force(O, L, B, N, seed)


def test_budget_invariants_random():
    for seed in range(40):
        rng = np.random.default_rng(100 + seed)
        L = int(rng.integers(1, 60))
        N = int(rng.integers(1, 50))
        B = int(rng.integers(0, L * N + 20))
        r = rng.normal(0.0, 0.05, size=L) + (0.02 if seed % 2 else 0.0)
        n, _ = O.allocate_budget(r, B, N)
        assert n.sum() == min(B, L * N) and n.min() >= 0 and n.max() <= N


def check_budget_ties_to_earlier(o):
    n, _ = o.allocate_budget(np.ones(4), 6, 10)             # quotas 1.5 each
    assert list(n) == [2, 2, 1, 1]


def test_budget_ties_and_uniform():
    check_budget_ties_to_earlier(O)
    n, _ = O.allocate_budget(np.full(256, 0.3), 18662, 729)
    assert n.max() - n.min() <= 1 and n.sum() == 18662 and np.all(np.diff(n) <= 0)


def test_budget_all_non_positive_is_uniform():
    n, _ = O.allocate_budget(np.array([-0.1, 0.0, -0.3]), 7, 5)
    assert list(n) == [3, 2, 2]


def test_budget_zero_weight_frames_get_nothing():
    n, _ = O.allocate_budget(np.array([0.5, -0.1, 0.25, 0.0]), 9, 10)
    assert list(n) == [6, 0, 3, 0]


def test_budget_caps():
    n, _ = O.allocate_budget(np.array([10.0, 1.0, 1.0]), 12, 6)
    assert list(n) == [6, 3, 3]
    # every positive-weight frame capped: the rest spreads over zero-weight frames
    n, _ = O.allocate_budget(np.array([1.0, -1.0, -1.0]), 10, 4)
    assert list(n) == [4, 3, 3]
    n, _ = O.allocate_budget(np.array([1.0, 0.2]), 50, 10)  # B > L*N
    assert list(n) == [10, 10]
    n, _ = O.allocate_budget(np.array([1.0, 0.2]), 0, 10)
    assert list(n) == [0, 0]


# ----------------------------------------------------------------------------
# WSM (Eq. 11-14) and the whole pass
# ----------------------------------------------------------------------------

def test_wsm_unit_gate_is_identity_and_zero_gate_is_lowpass():
    X = RNG.standard_normal((9, 11, 4))
    M = np.ones((9, 11))
    assert np.allclose(O.wsm(X, M, lam=1.0), X, atol=1e-12)
    f = O.wavelet_filters(4)
    LL, LH, HL, HH = O.dwt2d(X, f)
    low = O.idwt2d(LL, 0 * LH, 0 * HL, 0 * HH, 9, 11, f)
    assert np.allclose(O.wsm(X, M, lam=0.0), low, atol=1e-12)


def test_wsm_is_linear_in_x():
    X1, X2 = RNG.standard_normal((2, 13, 13, 3))
    M = RNG.random((13, 13))
    assert np.allclose(O.wsm(X1 + 2 * X2, M), O.wsm(X1, M) + 2 * O.wsm(X2, M), atol=1e-12)


def test_wsm_gate_scales_detail_only():
    """X~ = low + lambda * detail when M = 1 everywhere (detail = X - low)."""
    X = RNG.standard_normal((10, 10, 2))
    M = np.ones((10, 10))
    low = O.wsm(X, M, lam=0.0)
    assert np.allclose(O.wsm(X, M, lam=1.5), low + 1.5 * (X - low), atol=1e-12)


def test_condense_invariants():
    X = RNG.standard_normal((7, 5, 6, 8))
    Q = RNG.standard_normal((3, 8))
    res = O.condense(X, Q, 0.3)
    B = O.global_budget(0.3, 7, 30)
    assert res["B"] == B and res["count"] == B
    assert res["out_tokens"].shape == (B, 8) and np.all(np.isfinite(res["out_tokens"]))
    idx = res["out_index"]
    for t in range(7):
        rows = idx[res["offsets"][t]:res["offsets"][t + 1]]
        assert np.all(rows[:, 0] == t)
        h, w = O.grid_shape(int(res["budgets"][t]), 5, 6)
        for p, (_, i, j) in enumerate(rows):
            assert (i, j) == (p // w, p % w)


def test_condense_full_ratio_lambda_zero_is_lowpass():
    X = RNG.standard_normal((3, 4, 5, 6))
    Q = RNG.standard_normal((2, 6))
    res = O.condense(X, Q, 1.0, lam=0.0)
    f = O.wavelet_filters(4)
    for t in range(3):
        LL, LH, HL, HH = O.dwt2d(X[t], f)
        low = O.idwt2d(LL, 0 * LH, 0 * HL, 0 * HH, 4, 5, f).reshape(20, 6)
        assert np.allclose(res["out_tokens"][20 * t:20 * (t + 1)], low, atol=1e-12)


def test_condense_tail_rows_when_filter_drops_frames():
    X = np.zeros((4, 2, 2, 4))
    X[:, :, :, 0] = 1.0                                  # four identical frames
    Q = np.ones((1, 4))
    res = O.condense(X, Q, 0.9, tau=0.1)                 # only frame 1 survives
    assert res["keep"] == [0] and res["count"] == 4 and res["B"] == 14
    assert np.all(res["out_index"][4:] == -1) and np.all(res["out_tokens"][4:] == 0)


# ----------------------------------------------------------------------------
# Ablation modes (Section 4 "Ablation Study", Appendix B; reading R18)
# ----------------------------------------------------------------------------

def _aligned_video(T=10, H=4, W=5, D=6, seed=3):
    """Frames whose pooled vector leans on the query by a frame-dependent
    amount, so that r_t spreads over both signs."""
    g = np.random.default_rng(seed)
    Q = g.standard_normal((2, D))
    u = Q.mean(axis=0) / np.linalg.norm(Q.mean(axis=0))
    X = 0.3 * g.standard_normal((T, H, W, D))
    X += np.linspace(-1.0, 1.5, T)[:, None, None, None] * u
    return X, Q


def check_uniform_mode(o):
    X = RNG.standard_normal((9, 4, 5, 6))
    Q = RNG.standard_normal((2, 6))
    res = o.condense(X, Q, 0.37, temporal_mode="uniform")
    B, keep = res["B"], res["keep"]
    base, extra = divmod(B, len(keep))
    expect = np.zeros(9, dtype=np.int64)
    for k, t in enumerate(keep):                          # ties go to the earlier frame
        expect[t] = base + (1 if k < extra else 0)
    assert np.array_equal(res["budgets"], expect)


def check_raw_mode(o):
    X, Q = _aligned_video()
    res = o.condense(X, Q, 0.2, temporal_mode="raw")
    keep, B = res["keep"], res["B"]
    w = np.maximum(res["r"][keep], 0.0)
    q = B * w / w.sum()                                   # Eq. 15 quotas on the raw relevance
    n = res["budgets"][keep]
    assert n.sum() == B and np.all(q < 20)                # no cap binds at this ratio
    assert np.all((n == np.floor(q)) | (n == np.floor(q) + 1))
    frac = q - np.floor(q)
    got = n - np.floor(q)
    # the units beyond the floors went to the largest fractional parts
    assert frac[got == 1].min(initial=np.inf) >= frac[got == 0].max(initial=-np.inf)


def _torch_psi(Xt, n):
    H, W = Xt.shape[:2]
    h, w = OM.grid_shape(n, H, W)
    g = torch.nn.functional.interpolate(torch.from_numpy(Xt).permute(2, 0, 1)[None], size=(h, w),
                                        mode="bilinear", align_corners=False, antialias=False)
    return g[0].permute(1, 2, 0).reshape(h * w, -1)[:n].numpy()


def check_spatial_none(o):
    X, Q = _aligned_video()
    res = o.condense(X, Q, 0.4, spatial_mode="none")
    for t in range(X.shape[0]):
        lo, hi = res["offsets"][t], res["offsets"][t + 1]
        if hi > lo:
            assert np.allclose(res["out_tokens"][lo:hi], _torch_psi(X[t], hi - lo), atol=1e-12)


def check_spatial_saliency(o):
    X, Q = _aligned_video()
    lam = 1.3
    res = o.condense(X, Q, 0.4, lam=lam, spatial_mode="saliency")
    for t in range(X.shape[0]):
        lo, hi = res["offsets"][t], res["offsets"][t + 1]
        if hi > lo:
            A = torch.from_numpy(res["a"][t].reshape(X.shape[1], X.shape[2]))
            M = (A - A.min()) / (A.max() - A.min())
            Xw = lam * M.numpy()[:, :, None] * X[t]
            assert np.allclose(res["out_tokens"][lo:hi], _torch_psi(Xw, hi - lo), atol=1e-12)


def test_uniform_mode_budgets_closed_form():
    check_uniform_mode(O)


def test_raw_mode_apportions_raw_relevance():
    check_raw_mode(O)


def test_spatial_none_is_bilinear_of_features():
    check_spatial_none(O)


def test_spatial_saliency_is_bilinear_of_weighted_features():
    check_spatial_saliency(O)


def test_full_mode_differs_from_ablations():
    X, Q = _aligned_video()
    full = O.condense(X, Q, 0.4)
    for sm in ("saliency", "none"):
        abl = O.condense(X, Q, 0.4, spatial_mode=sm)
        assert np.array_equal(abl["budgets"], full["budgets"])
        assert not np.allclose(abl["out_tokens"], full["out_tokens"])


def test_external_constant_frame_scores_give_uniform_budgets():
    # constant r: the Haar details vanish, r~ = r, every quota is equal
    X = RNG.standard_normal((8, 4, 5, 6))
    Q = RNG.standard_normal((2, 6))
    ext = O.condense(X, Q, 0.3, frame_scores=np.full(8, 0.4))
    uni = O.condense(X, Q, 0.3, temporal_mode="uniform")
    assert np.array_equal(ext["budgets"], uni["budgets"])
    assert np.allclose(ext["r"], 0.4) and np.allclose(ext["r_tilde"], 0.4)


def test_external_flat_token_scores_remove_the_details():
    # a flat saliency map is M = 0 (R11), so G = 0 and the WSM keeps LL only:
    # the same tokens as lambda = 0
    X = RNG.standard_normal((3, 4, 5, 6))
    Q = RNG.standard_normal((2, 6))
    flat = O.condense(X, Q, 0.5, token_scores=np.full((3, 20), 0.7))
    low = O.condense(X, Q, 0.5, lam=0.0)
    assert np.array_equal(flat["budgets"], low["budgets"])
    assert np.allclose(flat["out_tokens"], low["out_tokens"], atol=1e-12)


def check_maxsim_hand_case(o):
    # two orthonormal query rows; one token equal to q_1, one to q_2, one along q_1 + q_2
    D = 4
    Q = np.array([[1.0, 0, 0, 0], [0, 1.0, 0, 0]])
    X = np.zeros((1, 1, 3, D))
    X[0, 0, 0] = [2.0, 0, 0, 0]
    X[0, 0, 1] = [0, 3.0, 0, 0]
    X[0, 0, 2] = [1.0, 1.0, 0, 0]
    res = o.condense(X, Q, 1.0, relevance="maxsim")
    assert np.allclose(res["a"][0], [1.0, 1.0, 1 / math.sqrt(2)], atol=1e-15)
    mean = o.condense(X, Q, 1.0)
    assert np.allclose(mean["a"][0], [1 / math.sqrt(2), 1 / math.sqrt(2), 1.0], atol=1e-15)
    # v_bar = (1, 4/3, 0, 0)/1: r = max of its cosines with q_1 and q_2
    v = np.array([3.0, 4.0, 0, 0]) / 3
    assert abs(res["r"][0] - 4.0 / 5.0) < 1e-15 and abs(mean["r"][0] - 7.0 / (5 * math.sqrt(2))) < 1e-15
    assert np.allclose(res["vbar"][0], v)


def test_maxsim_hand_case():
    check_maxsim_hand_case(O)


def test_maxsim_with_one_query_row_is_the_similarity_branch():
    X = RNG.standard_normal((6, 4, 5, 8))
    Q = RNG.standard_normal((1, 8))
    a, b = O.condense(X, Q, 0.3, relevance="maxsim"), O.condense(X, Q, 0.3)
    assert np.array_equal(a["budgets"], b["budgets"])
    assert np.allclose(a["a"], b["a"], atol=1e-15) and np.allclose(a["r"], b["r"], atol=1e-15)
    assert np.allclose(a["out_tokens"], b["out_tokens"], atol=1e-13)


# ----------------------------------------------------------------------------
# Projector P (Eq. 17, reading R21) against torch's CPU routines
# ----------------------------------------------------------------------------

def check_gelu(o):
    x = np.linspace(-6.0, 6.0, 241)
    ref = torch.nn.functional.gelu(torch.from_numpy(x), approximate="none").numpy()
    assert np.allclose(o.gelu(x), ref, atol=1e-15, rtol=1e-14)


def check_project(o):
    g = np.random.default_rng(5)
    Z = g.standard_normal((7, 24))
    W1, b1 = g.standard_normal((40, 24)) / 5, g.standard_normal(40)
    W2, b2 = g.standard_normal((16, 40)) / 6, g.standard_normal(16)
    t = lambda a: torch.from_numpy(a)
    hid = torch.nn.functional.gelu(torch.nn.functional.linear(t(Z), t(W1), t(b1)))
    ref = torch.nn.functional.linear(hid.to(torch.bfloat16).double(), t(W2), t(b2)).numpy()
    assert np.allclose(o.project(Z, W1, b1, W2, b2), ref, atol=1e-12)
    ref32 = torch.nn.functional.linear(hid, t(W2), t(b2)).numpy()
    assert np.allclose(o.project(Z, W1, b1, W2, b2, hidden_bf16=False), ref32, atol=1e-12)


def test_gelu_matches_torch():
    check_gelu(O)


def test_project_matches_torch_linear():
    check_project(O)


def test_project_identity_weights():
    Z = RNG.standard_normal((5, 8))
    eye = np.eye(8)
    out = O.project(Z, eye, None, eye, None)
    assert np.allclose(out, O.round_bf16(O.gelu(Z)), atol=0)


# ----------------------------------------------------------------------------
# Multi-level option of the wavelet modules (reading R23)
# ----------------------------------------------------------------------------

def check_multilevel_wta_hand_case(o):
    """Haar, two levels, on one block of four samples (worked by hand): the
    level-1 gates are the pair means of gamma (0.4, 0.5), the level-2 gate
    their mean (0.45); block mean 3, pair means 2 and 4."""
    r = np.array([1.0, 3.0, 2.0, 6.0])
    g = np.array([0.2, 0.6, 1.0, 0.0])
    # pair means after level 2: 3 -/+ 0.45 * (2 - 4) / 2; then -/+ gate * half-difference
    assert np.allclose(o.wta(r, g, 1, 2), [2.15, 2.95, 2.45, 4.45], atol=1e-12)


def check_multilevel_zero_gate_is_block_mean(o):
    r = np.array([1.0, 3.0, 2.0, 6.0, 0.0, 4.0, 8.0, 8.0])
    assert np.allclose(o.wta(r, np.zeros(8), 1, 2), np.repeat([3.0, 5.0], 4), atol=1e-12)
    assert np.allclose(o.wta(r, np.zeros(8), 1, 3), np.full(8, 4.0), atol=1e-12)
    X = RNG.standard_normal((8, 8, 2))
    blocks = X.reshape(2, 4, 2, 4, 2).mean(axis=(1, 3))
    expect = np.repeat(np.repeat(blocks, 4, axis=0), 4, axis=1)
    assert np.allclose(o.wsm(X, np.ones((8, 8)), lam=0.0, p=1, levels=2), expect, atol=1e-12)


def check_multilevel_wsm_level2_gate(o):
    """Haar, two levels, a 4x4 map constant on 2x2 blocks (no level-1 detail):
    the blocks b become mean + G_2 (b - mean) with G_2 = lambda * mean(M),
    the saliency map pooled to the 1x1 grid of level 2."""
    b = np.array([[1.0, -2.0], [0.5, 3.5]])
    X = np.repeat(np.repeat(b, 2, axis=0), 2, axis=1)[:, :, None]
    M = np.linspace(0.0, 1.0, 16).reshape(4, 4)
    lam = 1.25
    g2 = lam * M.mean()
    mu = b.mean()
    expect = np.repeat(np.repeat(mu + g2 * (b - mu), 2, axis=0), 2, axis=1)[:, :, None]
    assert np.allclose(o.wsm(X, M, lam=lam, p=1, levels=2), expect, atol=1e-12)


def test_multilevel_wta_hand_case():
    check_multilevel_wta_hand_case(O)


def test_multilevel_zero_gate_is_block_mean():
    check_multilevel_zero_gate_is_block_mean(O)


def test_multilevel_wsm_level2_gate():
    check_multilevel_wsm_level2_gate(O)


@pytest.mark.parametrize("p", [1, 2, 4, 44])
@pytest.mark.parametrize("levels", [2, 3, 4])
def test_multilevel_unit_gate_is_identity(p, levels):
    for L in (1, 2, 5, 23, 64):
        r = RNG.standard_normal(L)
        assert np.allclose(O.wta(r, np.ones(L), p, levels), r, atol=1e-11)
    for H, W in ((4, 4), (9, 11), (27, 27)):
        X = RNG.standard_normal((H, W, 2))
        assert np.allclose(O.wsm(X, np.ones((H, W)), lam=1.0, p=p, levels=levels), X, atol=1e-10)


def test_multilevel_one_level_is_the_single_level_module():
    r, g = RNG.standard_normal(19), RNG.random(19)
    X, M = RNG.standard_normal((13, 13, 3)), RNG.random((13, 13))
    assert np.array_equal(O.wta(r, g, 4, 1), O.wta(r, g, 4))
    assert np.array_equal(O.wsm(X, M, 1.5, 4, "symmetric", 1), O.wsm(X, M, 1.5, 4))


def test_multilevel_condense_invariants():
    X = RNG.standard_normal((9, 7, 8, 4))
    Q = RNG.standard_normal((3, 4))
    res = O.condense(X, Q, 0.3, wta_levels=3, wsm_levels=2)
    assert res["budgets"].sum() == O.global_budget(0.3, 9, 56)
    assert np.all(np.isfinite(res["out_tokens"]))


# ----------------------------------------------------------------------------
# Mutation tests: a planted mistake in the oracle makes a pin fail
# ----------------------------------------------------------------------------

def _mutant(**overrides):
    m = types.ModuleType("oracle_mutant")
    m.__dict__.update({k: v for k, v in OM.__dict__.items() if not k.startswith("__")})
    m.__dict__.update(overrides)
    # functions look globals up in their own module dict; rebind them to the mutant
    for k, v in list(m.__dict__.items()):
        if isinstance(v, types.FunctionType) and k not in overrides:
            m.__dict__[k] = types.FunctionType(v.__code__, m.__dict__, k, v.__defaults__, v.__closure__)
    return m


def _fails(fn, *args):
    try:
        fn(*args)
    except AssertionError:
        return True
    return False


def test_mutation_idwt_offset_breaks_pr():
    def idwt1d_bad(cA, cD, n, filt, axis=0):          # synthesis offset F-1 instead of F-2
        F, L = filt["F"], cA.shape[0]
        x = np.zeros((n,) + cA.shape[1:])
        for k in range(n):
            for i in range(L):
                t = k + F - 1 - 2 * i
                if 0 <= t < F:
                    x[k] += filt["rec_lo"][t] * cA[i] + filt["rec_hi"][t] * cD[i]
        return x
    m = _mutant(idwt1d=idwt1d_bad)
    assert _fails(check_perfect_reconstruction, m, 4, "symmetric", 12)


def test_mutation_highpass_sign_breaks_pins(golden_dir):
    good = OM.wavelet_filters

    def filters_bad(p):
        f = good(p)
        f = dict(f)
        f["rec_hi"] = np.array([f["rec_lo"][f["F"] - 1 - k] for k in range(f["F"])])  # dropped (-1)^k
        f["dec_hi"] = f["rec_hi"][::-1].copy()
        return f
    m = _mutant(wavelet_filters=filters_bad)
    assert _fails(check_filter_identities, m, 4)
    assert _fails(check_haar_1d_closed_forms, m)


def test_mutation_band_swap_breaks_haar_2d():
    def dwt2d_bad(X, filt, mode="symmetric"):
        LL, LH, HL, HH = OM.dwt2d(X, filt, mode)
        return LL, HL, LH, HH
    assert _fails(check_haar_2d_closed_forms, _mutant(dwt2d=dwt2d_bad))


def test_mutation_wrong_extension_breaks_convolution_pin():
    def ext_bad(i, n, mode):
        if 0 <= i < n:
            return i
        if mode == "symmetric":                        # whole-sample instead of half-sample
            k = i % (2 * n - 2) if n > 1 else 0
            return k if k < n else 2 * n - 2 - k
        return OM.extend_index(i, n, mode)
    assert _fails(check_dwt_vs_numpy_convolution, _mutant(extend_index=ext_bad), 4, "symmetric", 13)


def test_mutation_pool_bins_break_torch_pin():
    def pool_bad(M, oh, ow):
        H, W = M.shape
        out = np.zeros((oh, ow))
        for i in range(oh):
            r0, r1 = (i * H) // oh, max((i * H) // oh + 1, ((i + 1) * H) // oh)
            for j in range(ow):
                c0, c1 = (j * W) // ow, max((j * W) // ow + 1, ((j + 1) * W) // ow)
                out[i, j] = M[r0:r1, c0:c1].mean()
        return out
    assert _fails(check_adaptive_pool, _mutant(adaptive_avg_pool2d=pool_bad), 27, 27, 17, 17)


def test_mutation_align_corners_breaks_bilinear_pin():
    def src_bad(i, in_size, out_size):
        s = i * (in_size - 1) / max(out_size - 1, 1)
        i0 = min(int(math.floor(s)), in_size - 1)
        return i0, min(i0 + 1, in_size - 1), s - i0
    assert _fails(check_bilinear, _mutant(bilinear_source=src_bad), 27, 27, 9, 9)


def test_mutation_gate_on_approximation_breaks_wta():
    def wta_bad(r_M, gamma_M, p=1):
        r_M = np.asarray(r_M, dtype=np.float64)
        L = r_M.size
        filt = OM.wavelet_filters(p)
        A, D = OM.dwt1d(r_M, filt, "symmetric")
        gbar = np.array([0.5 * (gamma_M[OM.extend_index(2 * k, L, "symmetric")]
                                + gamma_M[OM.extend_index(2 * k + 1, L, "symmetric")])
                         for k in range(D.size)])
        return OM.idwt1d(gbar * A, D, L, filt)
    assert _fails(check_wta_closed_form, _mutant(wta=wta_bad))


def test_mutation_tie_rule_breaks_pin():
    src = OM.allocate_budget

    def alloc_bad(r, B, N):
        n, info = src(np.asarray(r)[::-1], B, N)
        return n[::-1].copy(), info
    assert _fails(check_budget_ties_to_earlier, _mutant(allocate_budget=alloc_bad))


def test_mutation_saliency_map_without_normalisation_breaks_saliency_pin():
    m = _mutant(saliency_map=lambda a_t, H, W: np.asarray(a_t, dtype=np.float64).reshape(H, W))
    assert _fails(check_spatial_saliency, m)


def test_mutation_budget_without_remainders_breaks_uniform_pin():
    def floors_only(r_tilde, B, N):
        w = np.maximum(np.asarray(r_tilde, dtype=np.float64), 0.0)
        n = np.floor(B * w / w.sum()).astype(np.int64)
        return n, {"alloc_gap": math.inf, "cap_gap": math.inf, "max_r": 1.0}
    m = _mutant(allocate_budget=floors_only)
    assert _fails(check_uniform_mode, m)


def test_mutation_bior44_normalisation_breaks_published_pin(golden_dir):
    def unit_sum():
        h, ht = OM.cdf97_lowpass()
        return h / h.sum(), ht / ht.sum()                # a plausible slip: DC gain 1, not sqrt(2)
    m = _mutant(cdf97_lowpass=unit_sum)
    assert _fails(check_bior44_published, m, golden_dir)


def test_mutation_tanh_gelu_breaks_gelu_pin():
    tanh_gelu = lambda x: 0.5 * np.asarray(x) * (1 + np.tanh(math.sqrt(2 / math.pi) * (np.asarray(x) + 0.044715 * np.asarray(x) ** 3)))
    m = _mutant(gelu=tanh_gelu)
    assert _fails(check_gelu, m)


def test_mutation_dropped_bias_breaks_project_pin():
    original = OM.project
    m = _mutant(project=lambda Z, W1, b1, W2, b2, hidden_bf16=True: original(Z, W1, None, W2, b2, hidden_bf16))
    assert _fails(check_project, m)


def test_mutation_maxsim_min_breaks_hand_case():
    original = OM.condense

    def min_condense(X, Q, ratio, **kw):
        res = original(X, Q, ratio, **kw)
        if kw.get("relevance") == "maxsim":              # planted: min over the rows instead of max
            Xr = np.asarray(X, dtype=np.float64)
            T, H, W, D = Xr.shape
            res["a"] = np.array([np.min([OM.token_saliency(Xr[t].reshape(H * W, D), q) for q in Q], axis=0)
                                 for t in range(T)])
        return res
    m = _mutant(condense=min_condense)
    assert _fails(check_maxsim_hand_case, m)


def test_mutation_level2_gate_from_gamma_breaks_multilevel_pin():
    def wta_bad(r_M, gamma_M, p=1, levels=1):         # planted: every level gated by gamma's pair means
        A = np.asarray(r_M, dtype=np.float64)
        filt = OM.wavelet_filters(p)
        n0 = A.size
        g1 = lambda k: 0.5 * (gamma_M[OM.extend_index(2 * k, n0, "symmetric")]
                              + gamma_M[OM.extend_index(2 * k + 1, n0, "symmetric")])
        details, lengths = [], []
        for _ in range(levels):
            n = A.size
            A_next, D = OM.dwt1d(A, filt, "symmetric")
            details.append(np.array([g1(k) for k in range(D.size)]) * D)
            lengths.append(n)
            A = A_next
        for j in reversed(range(levels)):
            A = OM.idwt1d(A, details[j], lengths[j], filt)
        return A
    assert _fails(check_multilevel_wta_hand_case, _mutant(wta=wta_bad))


def test_mutation_gated_level1_approximation_breaks_multilevel_pin():
    original = OM.wsm

    def wsm_bad(X_m, M_m, lam=1.5, p=4, mode="symmetric", levels=1):   # planted: LL of level 1 gated too
        if levels == 1:
            return original(X_m, M_m, lam, p, mode)
        filt = OM.wavelet_filters(p)
        LL, LH, HL, HH = OM.dwt2d(X_m, filt, mode)
        G = OM.as_float32(lam) * OM.adaptive_avg_pool2d(M_m, LL.shape[0], LL.shape[1])
        G = G.reshape(G.shape + (1,) * (X_m.ndim - 2))
        inner = original(LL, OM.adaptive_avg_pool2d(M_m, LL.shape[0], LL.shape[1]), lam, p, mode, levels - 1)
        return OM.idwt2d(G * inner, G * LH, G * HL, G * HH, X_m.shape[0], X_m.shape[1], filt)
    assert _fails(check_multilevel_zero_gate_is_block_mean, _mutant(wsm=wsm_bad))
