"""Shared helpers for the GPU parity tests (CUDA path vs the CPU oracle)."""

import numpy as np
import torch

import oracle as O
import workload as wl

# Decision margins below this are rejected when choosing seeds (quota units).
MIN_MARGIN = 1e-4
ATOL, RTOL = 1e-3, 2e-2


def to_np64(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().double().numpy()


def oracle_run(X, Q, ratio, **kw):
    return O.condense(to_np64(X), to_np64(Q), ratio, **kw)


def accepted_video(spec: wl.VideoSpec, tries: int = 8, **kw):
    """Generate the spec's video, advancing the seed by 10000 until every
    integer decision of the oracle (with options kw) is at least MIN_MARGIN
    from its boundary."""
    seed = spec.seed
    for _ in range(tries):
        s = wl.VideoSpec(**{**spec.__dict__, "seed": seed})
        X, Q, meta = wl.make_video(s)
        ref = oracle_run(X, Q, s.ratio, token_frames=[], **kw)
        if O.decision_margins(ref) >= MIN_MARGIN:
            return s, X, Q, ref
        seed += 10000
    raise AssertionError(f"no seed with margins >= {MIN_MARGIN} from {spec.seed}")


def accepted_random(T, H, W, D, Lq, ratio, seed=0, dtype="bf16", tries=20, **kw):
    for k in range(tries):
        X, Q = wl.random_video(T, H, W, D, Lq, dtype=dtype, seed=seed + 1000 * k)
        ref = oracle_run(X, Q, ratio, token_frames=[], **kw)
        if O.decision_margins(ref) >= MIN_MARGIN:
            return X, Q
    raise AssertionError("no random input with safe margins")


def round_like(x: np.ndarray, dtype: torch.dtype) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(x)).to(dtype).double().numpy()


def assert_tokens_close(got: np.ndarray, ref: np.ndarray, what="tokens"):
    assert got.shape == ref.shape, (got.shape, ref.shape)
    err = np.abs(got - ref)
    bound = ATOL + RTOL * np.abs(ref)
    bad = err > bound
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {bad.sum()} of {bad.size} outside |d| <= {ATOL} + {RTOL}|o|; "
                             f"first at {tuple(i)}: got {got[tuple(i)]} ref {ref[tuple(i)]}; "
                             f"max |d| {err.max():.3e}")


def assert_relevance_close(rel: np.ndarray, ref: dict):
    """The [T][4] per-frame outputs (r, delta, gamma, r~) against the oracle:
    r and delta to 1e-5, gamma to 1e-4, and r~ of Eq. 10 to 1e-5 on the
    retained frames and NaN on the filtered ones."""
    rel = np.asarray(rel, dtype=np.float64)
    assert np.allclose(rel[:, 0], ref["r"], atol=1e-5, rtol=0), "r"
    assert np.allclose(rel[:, 1], ref["delta"], atol=1e-5, rtol=0), "delta"
    assert np.allclose(rel[:, 2], ref["gamma"], atol=1e-4, rtol=0), "gamma"
    rt, rr = rel[:, 3], ref["r_tilde"]
    assert np.array_equal(np.isnan(rt), np.isnan(rr)), "r~: filtered frames differ"
    keep = ~np.isnan(rr)
    err = np.abs(rt[keep] - rr[keep])
    assert err.size == 0 or err.max() <= 1e-5, f"r~: max |d| {err.max():.3e}"


def compare_condense(out: dict, ref: dict, dtype: torch.dtype, frames=None):
    """Budgets, offsets and the index map bit-exact; tokens within tolerance;
    the per-frame relevance outputs (with r~) when the call returned them."""
    if out.get("relevance") is not None and "r_tilde" in ref:
        assert_relevance_close(out["relevance"].cpu().double().numpy().reshape(-1, 4), ref)
    budgets = out["budgets"].cpu().numpy().astype(np.int64)
    assert np.array_equal(budgets, ref["budgets"]), f"budgets differ at {np.nonzero(budgets != ref['budgets'])[0][:10]}"
    assert int(out["count"].cpu()[0]) == ref["count"]
    idx = out["index"].cpu().numpy().astype(np.int64)
    assert np.array_equal(idx, ref["out_index"]), "index map differs"
    tok = to_np64(out["tokens"])
    rt = round_like(ref["out_tokens"], dtype)
    if frames is None:
        assert_tokens_close(tok, rt)
    else:
        for t in frames:
            a, b = ref["offsets"][t], ref["offsets"][t + 1]
            assert_tokens_close(tok[a:b], rt[a:b], what=f"tokens of frame {t}")


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.view(torch.int16).numpy() if t.dtype == torch.bfloat16 else t.numpy()


def _tensor(a: np.ndarray) -> torch.Tensor:
    t = torch.from_numpy(a)
    return t.view(torch.bfloat16) if a.dtype == np.int16 else t


_REF_KEYS = ("out_tokens", "out_index", "budgets", "offsets", "count", "r", "delta", "gamma", "r_tilde")


def _accept_and_condense(spec: wl.VideoSpec):
    s, X, Q, _ = accepted_video(spec, tries=4)
    ref = oracle_run(X, Q, s.ratio)
    return s, _bits(X), _bits(Q), {k: ref[k] for k in _REF_KEYS}


def oracle_videos(specs, workers: int = 8):
    """accepted_video and the full oracle condensation of every spec, on a
    pool of spawned processes (safe after CUDA is initialised in the parent).
    Returns [(spec, X, Q, ref)] in the order of `specs`."""
    import multiprocessing as mp
    from concurrent.futures import ProcessPoolExecutor
    with ProcessPoolExecutor(max_workers=max(1, min(workers, len(specs))),
                             mp_context=mp.get_context("spawn")) as pool:
        res = list(pool.map(_accept_and_condense, specs))
    return [(s, _tensor(x), _tensor(q), ref) for s, x, q, ref in res]
