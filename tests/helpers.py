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


def compare_condense(out: dict, ref: dict, dtype: torch.dtype, frames=None):
    """Budgets, offsets and the index map bit-exact; tokens within tolerance."""
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
