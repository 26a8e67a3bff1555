"""The oracle's condensation pass with its per-frame steps spread over a pool
of processes: the second CPU baseline (test and baseline infrastructure only,
like the rest of this package; the product path never imports it).

Frames are independent in two of the pass's steps: the similarity branch of
the Cross-Modal Scorer (Section 3.2.1: a_{t,n}, v_bar_t, r_t) and the WSM with
Psi (Eq. 11-16).  Those run in worker processes, a few frames per job, on the
features shared through one block of shared memory (bf16 bit patterns,
widened to fp64 exactly in the worker).  The steps that couple the frames
(Eq. 7, the frame filter, the WTA of Eq. 8-10, the budgets of Eq. 5 / 15) run
in the parent.  Every step calls the same oracle function on the same fp64
operands as `condense`, so the budgets and the index map are the same and the
tokens agree to the last few ulps (a BLAS call may block its sums differently
in another process).  Default options only (mean query row, WTA + WSM).
"""
from __future__ import annotations

import multiprocessing as mp
from multiprocessing import shared_memory

import numpy as np

from . import wavezip_oracle as O


def _bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """bfloat16 bit patterns (uint16) -> float64, exactly."""
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _frames_f64(name: str, shape, t0: int, t1: int) -> np.ndarray:
    shm = shared_memory.SharedMemory(name=name)
    try:
        bits = np.ndarray(shape, dtype=np.uint16, buffer=shm.buf)
        X = _bf16_bits_to_f64(bits[t0:t1])
        del bits
    finally:
        shm.close()
    return X


def _relevance_job(job):
    name, shape, t0, t1, u_q = job
    T, H, W, D = shape
    X = _frames_f64(name, shape, t0, t1)
    out = []
    for k in range(t1 - t0):
        U = X[k].reshape(H * W, D)
        r, vbar = O.frame_relevance(U, u_q)
        out.append((O.token_saliency(U, u_q), r, vbar))
    return t0, out


def _condense_job(job):
    name, shape, items, lam, p, mode = job
    T, H, W, D = shape
    res = []
    for t, n, a_t in items:
        X = _frames_f64(name, shape, t, t + 1)[0]
        Xt = O.wsm(X, O.saliency_map(a_t, H, W), lam, p, mode)
        tok, _ = O.psi(Xt, n)
        res.append((t, tok))
    return res


def spawn_pool(workers: int):
    """A pool of `workers` spawned processes (safe after CUDA is initialised
    in the parent), reusable across calls of the drivers below."""
    return mp.get_context("spawn").Pool(workers)


def condense_parallel(bits: np.ndarray, Q, ratio: float, workers: int, lam: float = 1.5,
                      wsm_wavelet: int = 4, mode: str = "symmetric", frames_per_job: int = 2,
                      pool=None) -> dict:
    """`condense(X, Q, ratio)` for X given as bf16 bit patterns `bits` (T, H, W, D)
    uint16, with the per-frame steps on `workers` processes (spawned), or on
    the given `pool` of spawn_pool()."""
    bits = np.ascontiguousarray(bits, dtype=np.uint16)
    T, H, W, D = bits.shape
    N = H * W
    shape = (T, H, W, D)
    u_q = O.query_embedding(Q)
    shm = shared_memory.SharedMemory(create=True, size=bits.nbytes)
    own = pool is None
    try:
        view = np.ndarray(shape, dtype=np.uint16, buffer=shm.buf)
        view[...] = bits
        del view
        if own:
            pool = spawn_pool(workers)
        a = np.zeros((T, N))
        r = np.zeros(T)
        vbar = np.zeros((T, D))
        jobs = [(shm.name, shape, t0, min(T, t0 + frames_per_job), u_q)
                for t0 in range(0, T, frames_per_job)]
        for t0, out in pool.imap_unordered(_relevance_job, jobs):
            for k, (a_t, r_t, v_t) in enumerate(out):
                a[t0 + k], r[t0 + k], vbar[t0 + k] = a_t, r_t, v_t
        delta, gamma = O.visual_change(vbar)
        keep = O.frame_filter(delta, O.as_float32(0.0))
        r_tilde_M = O.wta(r[keep], gamma[keep], 1)
        B = O.global_budget(ratio, T, N)
        n_M, _ = O.allocate_budget(r_tilde_M, B, N)
        budgets = np.zeros(T, dtype=np.int64)
        for k, t in enumerate(keep):
            budgets[t] = n_M[k]
        offsets = np.zeros(T + 1, dtype=np.int64)
        offsets[1:] = np.cumsum(budgets)
        items = [(t, int(budgets[t]), a[t]) for t in range(T) if budgets[t] > 0]
        jobs = [(shm.name, shape, items[i:i + frames_per_job], lam, wsm_wavelet, mode)
                for i in range(0, len(items), frames_per_job)]
        out_tokens = np.zeros((B, D))
        for res in pool.imap_unordered(_condense_job, jobs):
            for t, tok in res:
                out_tokens[offsets[t]:offsets[t] + len(tok)] = tok
    finally:
        if own and pool is not None:
            pool.terminate()
        shm.close()
        shm.unlink()
    out_index = np.full((B, 3), -1, dtype=np.int64)
    for t in range(T):
        n = int(budgets[t])
        if n:
            h, w = O.grid_shape(n, H, W)
            for p in range(n):
                out_index[offsets[t] + p] = (t, p // w, p % w)
    return {"out_tokens": out_tokens, "out_index": out_index, "budgets": budgets, "offsets": offsets,
            "count": int(offsets[-1]), "B": B, "r": r, "delta": delta}


def _video_job(job):
    path, shape, v, q, ratio = job
    bits = np.load(path, mmap_mode="r")
    X = _bf16_bits_to_f64(np.asarray(bits[v]))
    del bits
    res = O.condense(X, q, ratio)
    return v, {k: res[k] for k in ("budgets", "out_index", "out_tokens", "count")}


def condense_videos_parallel(path: str, Qs, ratios, pool) -> list:
    """`condense(X_v, Q_v, ratio_v)` of every video of a batch, one video per
    job on `pool` (spawn_pool()).  `path` is a .npy file of bf16 bit patterns
    [V][T][H][W][D] uint16 that the workers map read-only; Qs[v] is video v's
    [Lq_v][D] query (fp64)."""
    bits = np.load(path, mmap_mode="r")
    shape = bits.shape
    del bits
    jobs = [(path, shape, v, np.asarray(Qs[v], dtype=np.float64), float(ratios[v])) for v in range(shape[0])]
    out = [None] * shape[0]
    for v, res in pool.imap_unordered(_video_job, jobs):
        out[v] = res
    return out
