"""Seeded synthetic inputs for the WaveZip condensation pass.

This module is shared by the tests, the benchmark and the oracle checks.  It
holds only input construction (random fields, query vectors, shapes) and none
of the method's arithmetic.

Recipe (stands in for the paper's LLaVA-Video / LLaVA-OneVision features on
EgoSchema, LongVideoBench and VideoMME, which are not available here):

* every frame is a spatially smooth Gaussian random field on the H x W token
  grid, independently per channel: white N(0,1) noise smoothed along H and W by
  a Gaussian of length-scale 3 tokens (half-sample symmetric boundary), each
  smoothing row normalised to unit L2 norm so every position has variance 1;
* over time the field follows AR(1), F_t = a F_{t-1} + sqrt(1-a^2) E_t, with a
  fresh independent field at each scene cut (cut frames uniform without
  replacement over frames 2..T);
* i.i.d. N(0, 0.1^2) noise is added to every feature;
* optional salient patches: 3x3-token patches at random places, each present
  over a random contiguous span of T/8 frames, adding +2 * (unit mean query);
* the query has Lq rows with i.i.d. N(0, 1/D) entries (std 1/sqrt(D)).

Shapes follow the paper's workloads: 64 frames by default and 16-128 in the
frame-budget ablation, 196 tokens per frame, keep ratios 0.1-0.25.
"""

from __future__ import annotations

import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass

import numpy as np
import torch

DTYPES = {"bf16": torch.bfloat16, "f32": torch.float32}


@dataclass
class VideoSpec:
    T: int
    H: int
    W: int
    D: int
    dtype: str = "bf16"
    Lq: int = 32
    ratio: float = 0.1
    ar: float = 0.95
    cuts: int = 3
    patches: int = 0
    seed: int = 0
    length_scale: float = 3.0
    noise: float = 0.1

    @property
    def N(self) -> int:
        return self.H * self.W


# The five workloads: a tiny fp32 case, the paper's 64-frame default at
# 13x13 tokens, a 128-frame case with query-correlated objects, the 256-frame
# HBM-roofline case and a 32-video serving batch.
CONFIGS = {
    "tiny_f32_16x14x14": VideoSpec(T=16, H=14, W=14, D=896, dtype="f32", Lq=16,
                                   ratio=0.25, ar=0.9, cuts=1, seed=1001),
    "video64_13x13_bf16": VideoSpec(T=64, H=13, W=13, D=3584, Lq=32, ratio=0.1,
                                    ar=0.95, cuts=3, seed=1002),
    "video128_16x16_objects": VideoSpec(T=128, H=16, W=16, D=3584, Lq=64, ratio=0.1,
                                        ar=0.95, cuts=6, patches=4, seed=1003),
    "video256_27x27_bf16": VideoSpec(T=256, H=27, W=27, D=3584, Lq=64, ratio=0.1,
                                     ar=0.95, cuts=12, seed=1004),
}
BATCH_NAME = "serving32x64_13x13_bf16"


def batch_specs(V: int = 32, T: int = 64, H: int = 13, W: int = 13, D: int = 3584):
    """The serving batch: per-video seeds 2000+v, Lq ~ U[8,128], rho in {0.05,0.1,0.25}."""
    rng = np.random.Generator(np.random.PCG64(3000))
    lqs = rng.integers(8, 129, size=V)
    ratios = rng.choice(np.array([0.05, 0.1, 0.25]), size=V)
    return [VideoSpec(T=T, H=H, W=W, D=D, Lq=int(lqs[v]), ratio=float(ratios[v]),
                      ar=0.95, cuts=3, seed=2000 + v) for v in range(V)]


def smoothing_matrix(n: int, length_scale: float) -> np.ndarray:
    """Gaussian smoothing along one axis with half-sample symmetric folding.

    Row y holds the weights of input positions for output y, normalised to
    unit L2 norm so that smoothed white noise has unit variance everywhere.
    """
    radius = int(math.ceil(3.0 * length_scale))
    K = np.zeros((n, n))
    for y in range(n):
        for o in range(-radius, radius + 1):
            k = (y + o) % (2 * n)
            k = k if k < n else 2 * n - 1 - k
            K[y, k] += math.exp(-0.5 * (o / length_scale) ** 2)
        K[y] /= np.linalg.norm(K[y])
    return K


def _frame_draws(seq, KH, KW, D, noise):
    """Smoothed field E_t and the i.i.d. noise of one frame (its own stream)."""
    rng = np.random.Generator(np.random.PCG64(seq))
    H, W = KH.shape[0], KW.shape[0]
    E = rng.standard_normal((H, W * D), dtype=np.float32).astype(np.float64)
    F = np.matmul(KH, E).reshape(H, W, D)
    F = np.matmul(KW[None], F)
    Z = rng.standard_normal((H, W, D), dtype=np.float32)
    return F, noise * Z


def make_video(spec: VideoSpec, device=None):
    """Return (features [T,H,W,D], query [Lq,D]) as torch tensors of spec.dtype.

    With device=None the features are drawn on the CPU from numpy streams
    (reproducible on any machine).  With a CUDA device the same recipe draws
    the per-frame noise from a torch generator on that device (much faster for
    gigabyte-sized inputs; different random numbers, same distribution).  The
    query, cuts and patches come from the numpy stream either way.
    Also returns a dict with the scene-cut frames and patch placements.
    """
    rng = np.random.Generator(np.random.PCG64(spec.seed))
    T, H, W, D = spec.T, spec.H, spec.W, spec.D
    dt = DTYPES[spec.dtype]
    q = rng.standard_normal((spec.Lq, D)) / math.sqrt(D)
    qmean = q.mean(axis=0)
    qhat = qmean / np.linalg.norm(qmean)
    ncut = min(spec.cuts, max(T - 1, 0))
    cuts = sorted(int(c) for c in rng.choice(np.arange(1, T), size=ncut, replace=False)) if ncut else []
    patches = []
    span = max(1, T // 8)
    for _ in range(spec.patches):
        y0 = int(rng.integers(0, max(1, H - 2)))
        x0 = int(rng.integers(0, max(1, W - 2)))
        t0 = int(rng.integers(0, max(1, T - span + 1)))
        patches.append((t0, t0 + span, y0, x0))
    KH = smoothing_matrix(H, spec.length_scale)
    KW = smoothing_matrix(W, spec.length_scale)
    meta = {"cuts": cuts, "patches": patches}
    if device is not None and torch.device(device).type != "cpu":
        X = _make_frames_torch(spec, KH, KW, qhat, cuts, patches, torch.device(device))
        return X, torch.from_numpy(q).to(dt).to(device), meta
    X = torch.empty((T, H, W, D), dtype=dt)
    a = spec.ar
    F = None
    cutset = set(cuts)
    seqs = np.random.SeedSequence(spec.seed).spawn(T)
    workers = max(1, min(16, os.cpu_count() or 1))
    with ThreadPoolExecutor(max_workers=workers) as pool:
        pending = [pool.submit(_frame_draws, seqs[t], KH, KW, D, spec.noise)
                   for t in range(min(T, 2 * workers))]
        for t in range(T):
            E, Z = pending[t].result()
            pending[t] = None
            nxt = t + 2 * workers
            if nxt < T:
                pending.append(pool.submit(_frame_draws, seqs[nxt], KH, KW, D, spec.noise))
            if F is None or t in cutset:
                F = E
            else:
                F = a * F + math.sqrt(1.0 - a * a) * E
            frame = F + Z
            for (t0, t1, y0, x0) in patches:
                if t0 <= t < t1:
                    frame[y0:y0 + 3, x0:x0 + 3, :] += 2.0 * qhat
            X[t] = torch.from_numpy(frame).to(dt)
    Q = torch.from_numpy(q).to(dt)
    return X, Q, meta


def _make_frames_torch(spec, KH, KW, qhat, cuts, patches, device):
    """The frame recipe of make_video with torch draws on `device` (float32)."""
    T, H, W, D = spec.T, spec.H, spec.W, spec.D
    g = torch.Generator(device=device).manual_seed(spec.seed)
    kh = torch.from_numpy(KH).float().to(device)
    kw = torch.from_numpy(KW).float().to(device)
    qv = torch.from_numpy(qhat).float().to(device)
    X = torch.empty((T, H, W, D), dtype=DTYPES[spec.dtype], device=device)
    a = spec.ar
    cutset = set(cuts)
    F = None
    for t in range(T):
        E = torch.randn((H, W * D), generator=g, device=device)
        E = torch.matmul(kh, E).reshape(H, W, D)
        E = torch.matmul(kw.unsqueeze(0), E)
        F = E if (F is None or t in cutset) else a * F + math.sqrt(1.0 - a * a) * E
        frame = F + spec.noise * torch.randn((H, W, D), generator=g, device=device)
        for (t0, t1, y0, x0) in patches:
            if t0 <= t < t1:
                frame[y0:y0 + 3, x0:x0 + 3, :] += 2.0 * qv
        X[t] = frame.to(X.dtype)
    return X


def make_batch(specs):
    """Concatenate videos of equal shape: features [V,T,H,W,D], queries [sum Lq, D]."""
    xs, qs = [], []
    for s in specs:
        X, Q, _ = make_video(s)
        xs.append(X)
        qs.append(Q)
    return torch.stack(xs), torch.cat(qs, dim=0)


def random_video(T, H, W, D, Lq, dtype="bf16", seed=0, scale=1.0):
    """Plain i.i.d. N(0, scale^2) features and query, for edge-case tests."""
    g = torch.Generator().manual_seed(seed)
    X = (torch.randn((T, H, W, D), generator=g, dtype=torch.float64) * scale).to(DTYPES[dtype])
    Q = torch.randn((Lq, D), generator=g, dtype=torch.float64).to(DTYPES[dtype])
    return X, Q
