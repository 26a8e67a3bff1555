"""CPU oracle for the WaveZip video-token condensation pass (arXiv 2607.23265).

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py`` (its ``cpu_baseline`` leg and its ``--impl reference`` arm) may
import this module.  The CUDA library never calls it, shares no code with it,
and must fail loudly instead of falling back to it.

This is a plain, slow, float64 restatement of the method, step by step in the
paper's order and notation (Section 3):

  query embedding u_q            Section 3.2.1 (global query embedding)
  token saliency a_{t,n}         Section 3.2.1, "Spatial Saliency"
  saliency map M_t               Eq. 6
  frame relevance r_t            Section 3.2.1, "Temporal Relevance"
  visual change delta_t, gamma_t Eq. 7 and the min-max gate after it
  frame filter  M = {t: d>=tau}  Section 3.2.2, "Frame Filter"
  WTA                            Eq. 8-10 (single-level Haar DWT)
  WSM                            Eq. 11-14 (single-level db4 2D DWT)
  Token Assigner budgets n_m     Eq. 15 with the constraint of Eq. 5
  bilinear condensation Psi      Eq. 16
  concatenation                  Eq. 18 (projector P of Eq. 17 = identity)

Library primitives used as single steps: matrix-vector products, means and
norms (numpy), polynomial roots (numpy.roots).  There is no blocking, fusion or
reordering beyond the definitions.

Readings of points the paper leaves open (each is a choice, not a verified
fact; the same list is kept in the design notes):
  R1  u_q is the mean of the Lq query rows (the paper uses one global vector).
  R2  the "similarity" scorer: the base features serve as u_{t,n}.
  R3  cosine with a zero norm is 0.
  R4  delta_t is clamped to [0, 2] and compares adjacent ORIGINAL frames.
  R5  a constant delta sequence gives gamma = 0.
  R6  frame 1 is always retained (delta_1 = 0 would otherwise drop it for tau>0);
      tau defaults to 0 (the filter keeps every frame).
  R7  WTA boundary: half-sample symmetric extension (an odd last sample pairs
      with itself, so its detail is 0 and it passes through).
  R8  P_down of Eq. 9 is the mean of the two (extended) gate samples of a pair.
  R9  B = round-half-away(rho * T * N), N_v counted before compression.
  R10 Eq. 15 "Round" cannot meet Eq. 5 exactly; budgets are apportioned by the
      largest-remainder rule (ties to the earlier frame), capped at N with the
      excess re-apportioned; all-non-positive relevance gives uniform weights;
      if every positive-weight frame is capped the rest goes uniformly to the
      remaining retained frames; if B > |M| N every retained frame keeps N.
  R11 the rank-preserving normalisation of Eq. 6 is per-frame min-max (range 0
      gives M = 0).
  R12 "db4" is the 8-tap Daubechies filter with 4 vanishing moments (the
      PyWavelets/MATLAB name), derived here by spectral factorisation.
  R13 DWT boundary: half-sample symmetric extension by default ("zero" and
      "periodic" are selectable); output length floor((n+F-1)/2).
  R14 P_down of Eq. 12 is adaptive average pooling (bins floor(i*H/h') ..
      ceil((i+1)*H/h')-1), gate lambda = 1.5.
  R15 Eq. 13 applies G on the whole detail bands (values <1 suppress, >1
      amplify); LL is unchanged.
  R16 Psi: n_m becomes an h_m x w_m grid, h_m = min(H, ceil(sqrt(n_m H / W))),
      w_m = ceil(n_m / h_m); bilinear with half-pixel centres
      (align_corners=False, no antialias); the first n_m points in raster
      order are kept; the index map records (t, i, j).
  R17 the output dtype is the input dtype; rows that cannot be produced
      (B > sum of budgets) carry index -1 and zero tokens.
  R18 the ablation modes of Section 4 ("Ablation Study") and Appendix B:
      temporal "raw" (Raw Top-k) apportions B with the same rule over
      max(r_t, 0) of the retained frames instead of max(r~, 0); temporal
      "uniform" apportions B over the retained frames with equal weights (the
      quotas are then exactly equal and the tie rule alone decides, so their
      rounding is not a decision margin); spatial "saliency" (Saliency-Only)
      replaces the WSM by the plain saliency weighting X~_m = lambda * M_m * X_m
      in the token domain; spatial "none" (the module ablation's Uniform / WTA
      rows) condenses X_m itself.  The default modes are the full method.
  R20 "bior4.4" is the biorthogonal CDF 9/7 pair (the PyWavelets name, as
      for db4), with 10-tap arrays laid out as in that library: analysis
      lowpass in dec_lo[1..9], synthesis lowpass in rec_lo[1..7]; the paper
      evaluates it for both WTA and WSM ("Wavelet Basis" ablation).
  R21 the projector P of Eq. 17 (applied after Psi, Eq. 16-18) is the two-
      layer MLP of LLaVA-style models, P(z) = W2 GELU(W1 z + b1) + b2 with the
      exact (erf) GELU; its weights are the caller's.  The hidden layer is
      rounded to the tokens' dtype (bf16), as a bf16 model stores it.
  R22 a max-over-query scorer ("maxsim") for queries of several rows: the
      query is not pooled; a_{t,n} = max_j cos(u_{t,n}, q_j) and
      r_t = max_j cos(v_bar_t, q_j) over the Lq rows q_j (with one row it is
      the similarity branch itself).
  R23 a multi-level option for both wavelet modules (the paper keeps one
      level, Section 4 "Wavelet Basis"; one level stays the default).  With
      J levels the DWT cascades on the approximation band.  WTA: the gate of
      level j's details is the pairwise mean (R8) of level j-1's gate, the
      gate of level 0 being gamma; the inverse cascades back.  WSM: the
      detail bands of level j are gated by G_j = lambda * P_down(M_m) with
      P_down the adaptive average pool (R14) of the saliency map to level
      j's subband grid; the approximation of level J is not gated.
  R19 an external scorer (Section 3.2.1 names BLIP-style matchers as
      alternatives to the similarity branch) may supply the token saliency
      a_{t,n} and / or the frame relevance r_t; the pooled features still come
      from X, since delta_t (Eq. 7) compares frames, not scores.
"""

from __future__ import annotations

import math
from math import comb

import numpy as np

MODES = ("symmetric", "zero", "periodic")


# ----------------------------------------------------------------------------
# Daubechies filters (Section 3.2.3: Haar for WTA, db4 for WSM)
# ----------------------------------------------------------------------------

def daubechies_lowpass(p: int) -> np.ndarray:
    """Minimum-phase Daubechies scaling filter with p vanishing moments (2p taps).

    Spectral factorisation: |m0(w)|^2 = cos^{2p}(w/2) P(sin^2(w/2)) with
    P(y) = sum_{k<p} C(p-1+k, k) y^k.  Each root y of P gives the pair z, 1/z
    solving (2 - z - 1/z)/4 = y; the root inside the unit circle is kept.  The
    filter is the coefficient list of (z+1)^p * prod(z - z_i), normalised so that
    sum h = sqrt(2).  p = 1 is Haar.
    """
    if p < 1:
        raise ValueError("p >= 1")
    coeff_ascending = [comb(p - 1 + k, k) for k in range(p)]
    zeros = []
    if p > 1:
        for y in np.roots(coeff_ascending[::-1]):
            b = 4.0 * y - 2.0                      # z^2 + b z + 1 = 0
            disc = np.sqrt(b * b - 4.0 + 0j)
            z1, z2 = (-b + disc) / 2.0, (-b - disc) / 2.0
            zeros.append(z1 if abs(z1) < 1.0 else z2)
    h = np.real(np.poly([-1.0] * p + zeros))
    return h * (math.sqrt(2.0) / h.sum())


BIOR44 = 44     # identifier of the biorthogonal wavelet bior4.4 (CDF 9/7)


def cdf97_lowpass():
    """(h, h~): the 7-tap synthesis and 9-tap analysis lowpass filters of bior4.4.

    Same product polynomial as db4 (p = 4): cos^8(w/2) P(sin^2(w/2)), split
    into two symmetric (zero-phase) factors cos^4 q(sin^2) and cos^4 q~(sin^2)
    with q q~ = P: the real root of P goes to q (7 taps), the complex pair to
    q~ (9 taps) (Cohen, Daubechies, Feauveau 1992).  sin^2(w/2) is
    (-z + 2 - 1/z) / 4 and cos^2(w/2) is (z + 2 + 1/z) / 4; each filter is
    normalised to sum sqrt(2).
    """
    P = [comb(3 + k, k) for k in range(4)]               # 1 + 4y + 10y^2 + 20y^3
    roots = np.roots(P[::-1])
    y_r = float(np.real(roots[np.argmin(np.abs(np.imag(roots)))]))
    y_c = roots[np.argmax(np.imag(roots))]
    cos4 = np.array([1.0, 4.0, 6.0, 4.0, 1.0]) / 16.0
    s_taps = np.array([-1.0, 2.0, -1.0]) / 4.0            # sin^2(w/2)
    q = np.array([0.0, 1.0, 0.0]) - s_taps / y_r
    alpha = float(np.real(1.0 / y_c + 1.0 / np.conj(y_c)))
    beta = float(np.real(1.0 / (y_c * np.conj(y_c))))
    qt = (np.array([0.0, 0.0, 1.0, 0.0, 0.0]) - alpha * np.pad(s_taps, 1)
          + beta * np.convolve(s_taps, s_taps))
    h = np.convolve(cos4, q)
    ht = np.convolve(cos4, qt)
    return h * (math.sqrt(2.0) / h.sum()), ht * (math.sqrt(2.0) / ht.sum())


def wavelet_filters(p: int) -> dict:
    """Analysis / synthesis filter bank of the orthogonal wavelet db<p>, or of
    bior4.4 for p = BIOR44.

    db<p>: rec_lo is the minimum-phase filter, dec_lo its reverse, and the
    high-pass pair is the alternating flip: rec_hi[k] = (-1)^k rec_lo[F-1-k].
    bior4.4 (reading R20): F = 10 taps; the 9-tap analysis lowpass occupies
    dec_lo[1..9] and the 7-tap synthesis lowpass rec_lo[1..7]; each high-pass
    filter is the alternating flip of the OTHER side's lowpass
    (rec_hi[k] = (-1)^k dec_lo[F-1-k] reversed, dec_hi from rec_lo).
    """
    if p == BIOR44:
        h, ht = cdf97_lowpass()
        F = 10
        rec_lo = np.zeros(F)
        rec_lo[1:8] = h
        ht_pad = np.zeros(F)
        ht_pad[0:9] = ht
        dec_lo = ht_pad[::-1].copy()
        rec_hi = np.array([(-1.0) ** k * ht_pad[F - 1 - k] for k in range(F)])
        g = np.array([(-1.0) ** k * rec_lo[F - 1 - k] for k in range(F)])
        return {"dec_lo": dec_lo, "dec_hi": g[::-1].copy(), "rec_lo": rec_lo, "rec_hi": rec_hi, "F": F}
    rec_lo = daubechies_lowpass(p)
    F = rec_lo.size
    rec_hi = np.array([(-1.0) ** k * rec_lo[F - 1 - k] for k in range(F)])
    return {"dec_lo": rec_lo[::-1].copy(), "dec_hi": rec_hi[::-1].copy(),
            "rec_lo": rec_lo, "rec_hi": rec_hi, "F": F}


# ----------------------------------------------------------------------------
# Single-level DWT / IDWT (Eq. 8, 10, 11, 14)
# ----------------------------------------------------------------------------

def extend_index(i: int, n: int, mode: str):
    """Index of the sample that position i of the extended signal copies.

    Returns None where the extension is zero.
    """
    if 0 <= i < n:
        return i
    if mode == "zero":
        return None
    if mode == "periodic":
        return i % n
    if mode == "symmetric":            # half-sample symmetric: x[-1-k] = x[k]
        k = i % (2 * n)
        return k if k < n else 2 * n - 1 - k
    raise ValueError(mode)


def dwt_len(n: int, F: int) -> int:
    return (n + F - 1) // 2


def dwt1d(x: np.ndarray, filt: dict, mode: str = "symmetric", axis: int = 0):
    """Single-level DWT along `axis`.

    Definition: with x^ the extended signal,
      cA[i] = sum_j dec_lo[j] * x^[2i + 1 - j],
      cD[i] = sum_j dec_hi[j] * x^[2i + 1 - j],   i = 0 .. floor((n+F-1)/2)-1.
    """
    x = np.moveaxis(np.asarray(x, dtype=np.float64), axis, 0)
    n, F = x.shape[0], filt["F"]
    L = dwt_len(n, F)
    cA = np.zeros((L,) + x.shape[1:])
    cD = np.zeros((L,) + x.shape[1:])
    for i in range(L):
        for j in range(F):
            src = extend_index(2 * i + 1 - j, n, mode)
            if src is None:
                continue
            cA[i] += filt["dec_lo"][j] * x[src]
            cD[i] += filt["dec_hi"][j] * x[src]
    return np.moveaxis(cA, 0, axis), np.moveaxis(cD, 0, axis)


def idwt1d(cA: np.ndarray, cD: np.ndarray, n: int, filt: dict, axis: int = 0):
    """Single-level inverse DWT along `axis`, returning n samples.

    Definition (upsample, filter with the synthesis pair, keep the n samples
    that start at offset F-2):
      x[k] = sum_i cA[i] rec_lo[k + F - 2 - 2i] + cD[i] rec_hi[k + F - 2 - 2i].
    """
    cA = np.moveaxis(np.asarray(cA, dtype=np.float64), axis, 0)
    cD = np.moveaxis(np.asarray(cD, dtype=np.float64), axis, 0)
    F, L = filt["F"], cA.shape[0]
    x = np.zeros((n,) + cA.shape[1:])
    for k in range(n):
        for i in range(L):
            t = k + F - 2 - 2 * i
            if 0 <= t < F:
                x[k] += filt["rec_lo"][t] * cA[i] + filt["rec_hi"][t] * cD[i]
    return np.moveaxis(x, 0, axis)


def dwt2d(X: np.ndarray, filt: dict, mode: str = "symmetric"):
    """Single-level 2D DWT of an (H, W, ...) map (Eq. 11).

    Rows (axis 0, height) first, then columns (axis 1, width).  The first band
    letter is the height filter, the second the width filter: LL, LH, HL, HH.
    """
    lo, hi = dwt1d(X, filt, mode, axis=0)
    LL, LH = dwt1d(lo, filt, mode, axis=1)
    HL, HH = dwt1d(hi, filt, mode, axis=1)
    return LL, LH, HL, HH


def idwt2d(LL, LH, HL, HH, H: int, W: int, filt: dict):
    """Inverse of dwt2d (Eq. 14), cropped to the original H x W."""
    lo = idwt1d(LL, LH, W, filt, axis=1)
    hi = idwt1d(HL, HH, W, filt, axis=1)
    return idwt1d(lo, hi, H, filt, axis=0)


# ----------------------------------------------------------------------------
# Cross-Modal Scorer (Section 3.2.1), similarity branch
# ----------------------------------------------------------------------------

def cosine(u: np.ndarray, v: np.ndarray) -> float:
    """cos(u, v); 0 when either norm is 0 (reading R3)."""
    nu, nv = float(np.linalg.norm(u)), float(np.linalg.norm(v))
    if nu == 0.0 or nv == 0.0:
        return 0.0
    return float(np.dot(u, v) / (nu * nv))


def query_embedding(Q: np.ndarray) -> np.ndarray:
    """u_q: mean of the query rows (reading R1)."""
    return np.asarray(Q, dtype=np.float64).mean(axis=0)


def token_saliency(U: np.ndarray, u_q: np.ndarray) -> np.ndarray:
    """a_{t,n} = cos(u_{t,n}, u_q) for the N tokens (rows) of one frame."""
    U = np.asarray(U, dtype=np.float64)
    nq = float(np.linalg.norm(u_q))
    nu = np.linalg.norm(U, axis=1)
    dots = U @ u_q
    out = np.zeros(U.shape[0])
    ok = (nu > 0) & (nq > 0)
    out[ok] = dots[ok] / (nu[ok] * nq)
    return out


def frame_relevance(U: np.ndarray, u_q: np.ndarray):
    """Average-pool the frame's tokens, then r_t = cos(v_bar_t, u_q).

    Returns (r_t, v_bar_t); the same pooled v_bar_t feeds Eq. 7.
    """
    vbar = np.asarray(U, dtype=np.float64).mean(axis=0)
    return cosine(vbar, u_q), vbar


def saliency_map(a_t: np.ndarray, H: int, W: int) -> np.ndarray:
    """M_t (Eq. 6): reshape to H x W, per-frame min-max (reading R11)."""
    A = np.asarray(a_t, dtype=np.float64).reshape(H, W)
    lo, hi = A.min(), A.max()
    if hi > lo:
        return (A - lo) / (hi - lo)
    return np.zeros((H, W))


# ----------------------------------------------------------------------------
# Visual Change Estimator (Section 3.2.2)
# ----------------------------------------------------------------------------

def visual_change(vbar: np.ndarray):
    """delta_t (Eq. 7) and gamma_t = min-max_t(delta_t)."""
    T = vbar.shape[0]
    delta = np.zeros(T)
    for t in range(1, T):
        delta[t] = min(2.0, max(0.0, 1.0 - cosine(vbar[t], vbar[t - 1])))
    lo, hi = delta.min(), delta.max()
    gamma = (delta - lo) / (hi - lo) if hi > lo else np.zeros(T)
    return delta, gamma


def frame_filter(delta: np.ndarray, tau: float) -> list:
    """Retained set M = {t : delta_t >= tau}, temporal order; frame 1 kept (R6)."""
    return [0] + [t for t in range(1, delta.shape[0]) if delta[t] >= tau]


# ----------------------------------------------------------------------------
# Wavelet Temporal Allocator (Eq. 8-10)
# ----------------------------------------------------------------------------

def wta(r_M: np.ndarray, gamma_M: np.ndarray, p: int = 1, levels: int = 1) -> np.ndarray:
    """Rectified relevance r~ = IDWT(A, Gamma_bar * D) with (A, D) = DWT(r).

    Gamma_bar_k is the mean of the extended gate samples 2k and 2k+1 (R8); the
    extension is the DWT's half-sample symmetric one (R7).  With levels > 1
    (R23) the DWT cascades on A, level j's gate is the same pairwise mean of
    level j-1's gate, and the inverse cascades back.
    """
    A = np.asarray(r_M, dtype=np.float64)
    g = np.asarray(gamma_M, dtype=np.float64)
    filt = wavelet_filters(p)
    details, lengths = [], []
    for _ in range(levels):
        n = A.size
        A_next, D = dwt1d(A, filt, "symmetric")
        gbar = np.array([0.5 * (g[extend_index(2 * k, n, "symmetric")]
                                + g[extend_index(2 * k + 1, n, "symmetric")])
                         for k in range(D.size)])
        details.append(gbar * D)
        lengths.append(n)
        A, g = A_next, gbar
    for j in reversed(range(levels)):
        A = idwt1d(A, details[j], lengths[j], filt)
    return A


# ----------------------------------------------------------------------------
# Token Assigner budgets (Eq. 5, Eq. 15)
# ----------------------------------------------------------------------------

def as_float32(x: float) -> float:
    """The C interface carries rho, lambda and tau as 32-bit floats."""
    return float(np.float32(x))


def global_budget(ratio: float, T: int, N: int) -> int:
    """B = rho * N_v rounded half away from zero, N_v = T * N (reading R9)."""
    x = as_float32(ratio) * T * N
    return int(math.floor(x + 0.5))


def allocate_budget(r_tilde: np.ndarray, B: int, N: int):
    """Integer budgets n_m >= 0 with sum n_m = B (Eq. 5), quotas per Eq. 15.

    Largest-remainder apportionment with caps at N (reading R10).  Returns
    (n, margins) where margins holds the distances of the decisions from their
    boundaries in quota units (see decision_margins).
    """
    r_tilde = np.asarray(r_tilde, dtype=np.float64)
    L = r_tilde.size
    n = np.zeros(L, dtype=np.int64)
    info = {"alloc_gap": math.inf, "cap_gap": math.inf,
            "max_r": float(r_tilde.max()) if L else 0.0}
    if L == 0 or B <= 0:
        return n, info
    if B >= L * N:
        n[:] = N
        return n, info
    w = np.maximum(r_tilde, 0.0)
    if not np.any(w > 0):
        w = np.ones(L)
    active = list(range(L))
    remaining = B
    while True:
        act = [m for m in active if w[m] > 0]
        weights = {m: w[m] for m in act}
        if not act:                                   # every positive frame capped
            act = list(active)
            weights = {m: 1.0 for m in act}
        S = 0.0
        for m in act:
            S += weights[m]
        q = {m: remaining * weights[m] / S for m in act}
        for m in act:
            info["cap_gap"] = min(info["cap_gap"], abs(q[m] - N))
        capped = [m for m in act if q[m] > N]
        if capped:
            for m in capped:
                n[m] = N
                active.remove(m)
            remaining -= N * len(capped)
            continue
        fl = {m: math.floor(q[m]) for m in act}
        R = remaining - sum(fl.values())
        frac = {m: q[m] - fl[m] for m in act}
        order = sorted(act, key=lambda m: (-frac[m], m))
        for m in act:
            n[m] = fl[m]
        for m in order[:R]:
            n[m] += 1
        f = [frac[m] for m in order]
        K = len(f)
        upper = f[R - 1] if R > 0 else f[K - 1] + 1.0
        lower = f[R] if R < K else f[0] - 1.0
        info["alloc_gap"] = upper - lower
        return n, info


# ----------------------------------------------------------------------------
# Wavelet Spatial Modulator (Eq. 11-14)
# ----------------------------------------------------------------------------

def adaptive_avg_pool2d(M: np.ndarray, oh: int, ow: int) -> np.ndarray:
    """Average over bins rows floor(i*H/oh) .. ceil((i+1)*H/oh)-1 (same for columns)."""
    H, W = M.shape
    out = np.zeros((oh, ow))
    for i in range(oh):
        r0, r1 = (i * H) // oh, -((-(i + 1) * H) // oh)
        for j in range(ow):
            c0, c1 = (j * W) // ow, -((-(j + 1) * W) // ow)
            out[i, j] = M[r0:r1, c0:c1].mean()
    return out


def wsm(X_m: np.ndarray, M_m: np.ndarray, lam: float = 1.5, p: int = 4,
        mode: str = "symmetric", levels: int = 1) -> np.ndarray:
    """X~_m = IDWT2(LL, G*LH, G*HL, G*HH) with G = lambda * P_down(M_m).

    levels > 1 (R23): the DWT2 cascades on LL; level j's detail bands are
    gated by lambda * P_down(M_m) pooled to level j's subband grid.
    """
    filt = wavelet_filters(p)
    LL = X_m
    bands, sizes = [], []
    for _ in range(levels):
        sizes.append(LL.shape[:2])
        LL, LH, HL, HH = dwt2d(LL, filt, mode)
        G = as_float32(lam) * adaptive_avg_pool2d(M_m, LL.shape[0], LL.shape[1])
        G = G.reshape(G.shape + (1,) * (X_m.ndim - 2))
        bands.append((G * LH, G * HL, G * HH))
    for j in reversed(range(levels)):
        H, W = sizes[j]
        LL = idwt2d(LL, *bands[j], H, W, filt)
    return LL


# ----------------------------------------------------------------------------
# Psi: budget-guided bilinear interpolation (Eq. 16) and packing (Eq. 18)
# ----------------------------------------------------------------------------

def grid_shape(n: int, H: int, W: int):
    """(h_m, w_m): h = min(H, ceil(sqrt(n H / W))), w = ceil(n / h) (reading R16).

    ceil(sqrt(x)) for the rational x = nH/W is the least h with h*h*W >= n*H,
    evaluated exactly in integers.
    """
    if n <= 0:
        return 0, 0
    h = math.isqrt((n * H) // W)
    while h * h * W < n * H:
        h += 1
    while h > 1 and (h - 1) * (h - 1) * W >= n * H:
        h -= 1
    h = min(H, max(1, h))
    return h, -(-n // h)


def bilinear_source(i: int, in_size: int, out_size: int):
    """Half-pixel source coordinate (align_corners=False): (i0, i1, weight of i1)."""
    s = (i + 0.5) * (in_size / out_size) - 0.5
    s = max(s, 0.0)
    i0 = min(int(math.floor(s)), in_size - 1)
    i1 = min(i0 + 1, in_size - 1)
    return i0, i1, s - i0


def bilinear_resize(Xt: np.ndarray, h: int, w: int) -> np.ndarray:
    """Bilinear resample of an (H, W, D) map to (h, w, D)."""
    H, W = Xt.shape[:2]
    out = np.zeros((h, w) + Xt.shape[2:])
    for i in range(h):
        y0, y1, ly = bilinear_source(i, H, h)
        for j in range(w):
            x0, x1, lx = bilinear_source(j, W, w)
            out[i, j] = ((1 - ly) * ((1 - lx) * Xt[y0, x0] + lx * Xt[y0, x1])
                         + ly * ((1 - lx) * Xt[y1, x0] + lx * Xt[y1, x1]))
    return out


def psi(Xt_tilde: np.ndarray, n: int):
    """Psi(X~_m, n_m): the first n_m points of the h_m x w_m grid in raster order."""
    H, W = Xt_tilde.shape[:2]
    h, w = grid_shape(n, H, W)
    grid = bilinear_resize(Xt_tilde, h, w).reshape((h * w,) + Xt_tilde.shape[2:])
    idx = [(p // w, p % w) for p in range(n)]
    return grid[:n], idx


# ----------------------------------------------------------------------------
# Whole pass C_WaveZip(X, Q) (Section 3.2, Eq. 18)
# ----------------------------------------------------------------------------

TEMPORAL_MODES = ("wta", "raw", "uniform")
SPATIAL_MODES = ("wsm", "saliency", "none")


def condense(X, Q, ratio: float, lam: float = 1.5, tau: float = 0.0,
             wta_wavelet: int = 1, wsm_wavelet: int = 4, mode: str = "symmetric",
             token_frames=None, temporal_mode: str = "wta", spatial_mode: str = "wsm",
             token_scores=None, frame_scores=None, relevance: str = "mean",
             wta_levels: int = 1, wsm_levels: int = 1) -> dict:
    """Condense features X (T, H, W, D) for query Q (Lq, D) to B tokens.

    token_frames: optional iterable of frame indices; when given, the WSM and
    Psi steps run only for those frames (budgets, offsets and the index map are
    always complete), and out_tokens rows of other frames are left as NaN.
    temporal_mode / spatial_mode: the ablation modes of reading R18.
    token_scores (T, N) / frame_scores (T,): an external scorer's a_{t,n} and
    r_t (reading R19), replacing the similarity branch's values.
    relevance: "mean" (u_q = mean query row, R1) or "maxsim" (reading R22).
    wta_levels / wsm_levels: decomposition levels of the two modules (R23).
    """
    if temporal_mode not in TEMPORAL_MODES or spatial_mode not in SPATIAL_MODES or relevance not in ("mean", "maxsim"):
        raise ValueError("unknown mode")
    X = np.asarray(X, dtype=np.float64)
    T, H, W, D = X.shape
    N = H * W
    u_q = query_embedding(Q)
    a = np.zeros((T, N))
    r = np.zeros(T)
    vbar = np.zeros((T, D))
    for t in range(T):
        U = X[t].reshape(N, D)
        a[t] = token_saliency(U, u_q)
        r[t], vbar[t] = frame_relevance(U, u_q)
        if relevance == "maxsim":
            Qr = np.asarray(Q, dtype=np.float64)
            a[t] = np.max([token_saliency(U, q) for q in Qr], axis=0)
            r[t] = max(cosine(vbar[t], q) for q in Qr)
    if token_scores is not None:
        a = np.asarray(token_scores, dtype=np.float64).reshape(T, N).copy()
    if frame_scores is not None:
        r = np.asarray(frame_scores, dtype=np.float64).reshape(T).copy()
    delta, gamma = visual_change(vbar)
    keep = frame_filter(delta, as_float32(tau))
    r_tilde_M = wta(r[keep], gamma[keep], wta_wavelet, wta_levels)
    B = global_budget(ratio, T, N)
    if temporal_mode == "wta":
        n_M, margins = allocate_budget(r_tilde_M, B, N)
    elif temporal_mode == "raw":
        n_M, margins = allocate_budget(r[keep], B, N)
    else:
        n_M, margins = allocate_budget(np.ones(len(keep)), B, N)
        margins["alloc_gap"] = math.inf        # equal quotas: the tie rule decides (R18)
    budgets = np.zeros(T, dtype=np.int64)
    r_tilde = np.full(T, np.nan)
    for k, t in enumerate(keep):
        budgets[t] = n_M[k]
        r_tilde[t] = r_tilde_M[k]
    offsets = np.zeros(T + 1, dtype=np.int64)
    offsets[1:] = np.cumsum(budgets)
    count = int(offsets[-1])
    out_tokens = np.zeros((B, D))
    out_index = np.full((B, 3), -1, dtype=np.int64)
    frames = set(range(T)) if token_frames is None else set(token_frames)
    for t in range(T):
        n = int(budgets[t])
        if n == 0:
            continue
        h, w = grid_shape(n, H, W)
        for p in range(n):
            out_index[offsets[t] + p] = (t, p // w, p % w)
        if t in frames:
            if spatial_mode == "wsm":
                Xt = wsm(X[t], saliency_map(a[t], H, W), lam, wsm_wavelet, mode, wsm_levels)
            elif spatial_mode == "saliency":
                Xt = lam * saliency_map(a[t], H, W)[:, :, None] * X[t]
            else:
                Xt = X[t]
            tok, _ = psi(Xt, n)
            out_tokens[offsets[t]:offsets[t] + n] = tok
        else:
            out_tokens[offsets[t]:offsets[t] + n] = np.nan
    margins = dict(margins)
    if tau > 0 and T > 1:
        margins["tau_gap"] = float(np.min(np.abs(delta[1:] - as_float32(tau))))
    return {"out_tokens": out_tokens, "out_index": out_index, "budgets": budgets,
            "offsets": offsets, "count": count, "B": B, "a": a, "r": r,
            "vbar": vbar, "delta": delta, "gamma": gamma, "keep": keep,
            "r_tilde": r_tilde, "u_q": u_q, "margins": margins}


def decision_margins(result: dict) -> float:
    """Smallest distance of any integer decision from its boundary.

    alloc_gap: gap between the last awarded and first unawarded fractional
    quota (largest remainder, circular); cap_gap: |q_m - N|; max_r: |max r~|
    (the all-non-positive fallback); tau_gap: |delta_t - tau| when tau > 0.
    """
    m = result["margins"]
    vals = [m.get("alloc_gap", math.inf), m.get("cap_gap", math.inf),
            abs(m.get("max_r", math.inf)), m.get("tau_gap", math.inf)]
    return float(min(vals))


# ----------------------------------------------------------------------------
# Projector P (Eq. 17), applied to the condensed tokens (reading R21)
# ----------------------------------------------------------------------------

def gelu(x: np.ndarray) -> np.ndarray:
    """GELU(x) = x Phi(x) = x (1 + erf(x / sqrt 2)) / 2, elementwise."""
    x = np.asarray(x, dtype=np.float64)
    return np.array([0.5 * v * (1.0 + math.erf(v / math.sqrt(2.0))) for v in x.ravel()]).reshape(x.shape)


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round to bfloat16 (nearest, ties to even) and back to float64."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float64)).to(torch.bfloat16).double().numpy()


def project(Z: np.ndarray, W1: np.ndarray, b1, W2: np.ndarray, b2, hidden_bf16: bool = True) -> np.ndarray:
    """P(Z) = GELU(Z W1^T + b1) W2^T + b2 for tokens Z (B, D), W1 (C, D), W2 (E, C).

    A bias of None is zero.  With hidden_bf16 the hidden layer is rounded to
    bfloat16 between the two layers (reading R21).
    """
    Z = np.asarray(Z, dtype=np.float64)
    Hd = Z @ np.asarray(W1, dtype=np.float64).T
    if b1 is not None:
        Hd = Hd + np.asarray(b1, dtype=np.float64)[None, :]
    Hd = gelu(Hd)
    if hidden_bf16:
        Hd = round_bf16(Hd)
    out = Hd @ np.asarray(W2, dtype=np.float64).T
    if b2 is not None:
        out = out + np.asarray(b2, dtype=np.float64)[None, :]
    return out
