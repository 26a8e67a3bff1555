"""Python binding of the WaveZip C ABI (include/wavezip.h).

Argument marshalling only: every function allocates its outputs as torch
tensors on the inputs' device, passes raw device pointers and the current
CUDA stream to the library, and raises WaveZipError on a nonzero status.  All
computation happens in the CUDA kernels of libwavezip.so; there is no other
implementation to fall back to, and importing fails if the library is absent.
"""

from __future__ import annotations

import contextlib
import ctypes as C
import os

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libwavezip.so")
LIB_CHECKED_PATH = os.path.join(_HERE, "libwavezip_checked.so")   # bounds-checked build (WZ_CHECKED)

OK, ERR_INVALID_ARG, ERR_UNSUPPORTED, ERR_CUDA, ERR_NO_MEMORY, ERR_WORKSPACE = 0, -1, -2, -3, -4, -5
DTYPE_BF16, DTYPE_F32 = 0, 1
MODE_SYMMETRIC, MODE_ZERO, MODE_PERIODIC = 0, 1, 2
PATH_AUTO, PATH_TENSOR, PATH_SIMT = 0, 1, 2
MODES = {"symmetric": MODE_SYMMETRIC, "zero": MODE_ZERO, "periodic": MODE_PERIODIC}
PATHS = {"auto": PATH_AUTO, "tensor": PATH_TENSOR, "simt": PATH_SIMT}
WAVELET_HAAR, WAVELET_DB4, WAVELET_BIOR44 = 1, 4, 44
TEMPORAL_WTA, TEMPORAL_RAW, TEMPORAL_UNIFORM = 0, 1, 2
SPATIAL_WSM, SPATIAL_SALIENCY, SPATIAL_NONE = 0, 1, 2
TEMPORAL_MODES = {"wta": TEMPORAL_WTA, "raw": TEMPORAL_RAW, "uniform": TEMPORAL_UNIFORM}
SPATIAL_MODES = {"wsm": SPATIAL_WSM, "saliency": SPATIAL_SALIENCY, "none": SPATIAL_NONE}
RELEVANCE_MEAN, RELEVANCE_MAXSIM = 0, 1
RELEVANCE_MODES = {"mean": RELEVANCE_MEAN, "maxsim": RELEVANCE_MAXSIM}
MAX_LQ_MAXSIM = 128
MAX_LEVELS = 4


def _enum(table, v):
    return table[v] if isinstance(v, str) else int(v)


def _f32_scores(x: torch.Tensor, shape, name: str) -> torch.Tensor:
    if x.dtype != torch.float32 or not x.is_cuda or tuple(x.shape) != tuple(shape):
        raise ValueError(f"{name} must be a float32 CUDA tensor of shape {tuple(shape)}")
    return x.contiguous()


class WaveZipError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {status_string(status)} ({status})")


class CondenseArgs(C.Structure):
    _fields_ = [
        ("features", C.c_void_p), ("T", C.c_int), ("H", C.c_int), ("W", C.c_int), ("D", C.c_int),
        ("dtype", C.c_int), ("query", C.c_void_p), ("Lq", C.c_int), ("ratio", C.c_float),
        ("lam", C.c_float), ("tau", C.c_float), ("wta_wavelet", C.c_int), ("wsm_wavelet", C.c_int),
        ("mode", C.c_int), ("path", C.c_int), ("temporal_mode", C.c_int), ("spatial_mode", C.c_int),
        ("token_scores", C.c_void_p), ("frame_scores", C.c_void_p), ("relevance_mode", C.c_int),
        ("wta_levels", C.c_int), ("wsm_levels", C.c_int),
        ("out_tokens", C.c_void_p), ("out_index", C.c_void_p),
        ("out_budgets", C.c_void_p), ("out_count", C.c_void_p), ("out_relevance", C.c_void_p),
        ("workspace", C.c_void_p), ("workspace_bytes", C.c_size_t), ("device_status", C.c_void_p),
        ("kernel_events", C.POINTER(C.c_void_p)), ("stream", C.c_void_p),
    ]


class BatchArgs(C.Structure):
    _fields_ = [
        ("V", C.c_int), ("features", C.c_void_p), ("T", C.c_int), ("H", C.c_int), ("W", C.c_int),
        ("D", C.c_int), ("dtype", C.c_int), ("queries", C.c_void_p), ("Lq", C.POINTER(C.c_int32)),
        ("ratio", C.POINTER(C.c_float)), ("lam", C.c_float), ("tau", C.c_float),
        ("wta_wavelet", C.c_int), ("wsm_wavelet", C.c_int), ("mode", C.c_int), ("path", C.c_int),
        ("temporal_mode", C.c_int), ("spatial_mode", C.c_int),
        ("token_scores", C.c_void_p), ("frame_scores", C.c_void_p), ("relevance_mode", C.c_int),
        ("wta_levels", C.c_int), ("wsm_levels", C.c_int),
        ("out_tokens", C.c_void_p), ("out_index", C.c_void_p), ("row_offsets", C.POINTER(C.c_int64)),
        ("out_budgets", C.c_void_p), ("out_count", C.c_void_p), ("out_relevance", C.c_void_p),
        ("workspace", C.c_void_p), ("workspace_bytes", C.c_size_t), ("device_status", C.c_void_p),
        ("kernel_events", C.POINTER(C.c_void_p)), ("stream", C.c_void_p),
    ]

class ProjectArgs(C.Structure):
    _fields_ = [
        ("tokens", C.c_void_p), ("B", C.c_int64), ("D", C.c_int), ("w1", C.c_void_p), ("b1", C.c_void_p),
        ("C", C.c_int), ("w2", C.c_void_p), ("b2", C.c_void_p), ("E", C.c_int), ("out", C.c_void_p),
        ("workspace", C.c_void_p), ("workspace_bytes", C.c_size_t), ("device_status", C.c_void_p),
        ("stream", C.c_void_p),
    ]


NUM_KERNELS = 6
KERNEL_NAMES = ("query_pool", "relevance", "frame_stats", "temporal", "spatial", "condense")


def _load(path: str = LIB_PATH):
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it with `python -m paper_2607_23265_gb300.build` "
                          "(the WaveZip path has no non-CUDA implementation)")
    lib = C.CDLL(path)
    vp, i, f, sz, i64 = C.c_void_p, C.c_int, C.c_float, C.c_size_t, C.c_int64
    sig = {
        "wz_budget_size": (i64, [i, i, i, f]),
        "wz_condense": (i, [vp, i, i, i, i, vp, i, f, vp, vp, vp]),
        "wz_condense_args_init": (None, [C.POINTER(CondenseArgs)]),
        "wz_condense_workspace_size": (sz, [i, i, i, i, i, f]),
        "wz_condense_ex": (i, [C.POINTER(CondenseArgs)]),
        "wz_condense_host": (i, [C.POINTER(CondenseArgs)]),
        "wz_batch_args_init": (None, [C.POINTER(BatchArgs)]),
        "wz_batch_rows": (i64, [i, i, i, i, C.POINTER(C.c_float), C.POINTER(C.c_int64)]),
        "wz_batch_workspace_size": (sz, [i, i, i, i, i, i, C.POINTER(C.c_float)]),
        "wz_condense_batch": (i, [C.POINTER(BatchArgs)]),
        "wz_relevance": (i, [vp, i, i, i, i, i, vp, i, vp, vp, vp, vp, sz, vp, vp]),
        "wz_relevance_workspace_size": (sz, [i, i, i, i]),
        "wz_relevance_static": (i, [vp, i, i, i, i, i, vp, i, vp, vp, vp, vp, vp]),
        "wz_project_workspace_size": (sz, [i64, i]),
        "wz_project": (i, [C.POINTER(ProjectArgs)]),
        "wz_dwt_len": (i, [i, i]),
        "wz_wavelet_filters": (i, [i] + [C.POINTER(C.c_double)] * 4),
        "wz_dwt1d": (i, [vp, i, i, i, i, vp, vp, vp]),
        "wz_idwt1d": (i, [vp, vp, i, i, i, vp, vp]),
        "wz_dwt2d": (i, [vp, i, i, i, i, i, i, i, vp, vp, vp, vp, vp]),
        "wz_idwt2d": (i, [vp, vp, vp, vp, i, i, i, i, i, vp, vp]),
        "wz_status_string": (C.c_char_p, [i]),
        "wz_version": (i, []),
        "wz_graph_cache": (i, [i, C.POINTER(C.c_int64)]),
        "wz_selftest_bounded_wait": (i, [C.c_uint64, vp, vp]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


_lib = _load()


def status_string(status: int) -> str:
    return _lib.wz_status_string(int(status)).decode()


def _check(status: int, where: str):
    if status != OK:
        raise WaveZipError(status, where)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return DTYPE_BF16
    if t.dtype == torch.float32:
        return DTYPE_F32
    raise TypeError(f"features must be bfloat16 or float32, got {t.dtype}")


def _stream(stream, device) -> int:
    if stream is None:
        stream = torch.cuda.current_stream(device)
    return int(stream.cuda_stream)


def _ptr(t):
    return None if t is None else t.data_ptr()


def _cuda_contig(t: torch.Tensor, name: str) -> torch.Tensor:
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    return t.contiguous()


# --------------------------------------------------------------------------
# Condensation
# --------------------------------------------------------------------------

def wz_budget_size(T: int, H: int, W: int, ratio: float) -> int:
    return int(_lib.wz_budget_size(T, H, W, ratio))


def wz_condense_workspace_size(T, H, W, D, dtype=DTYPE_BF16, ratio=0.1) -> int:
    return int(_lib.wz_condense_workspace_size(T, H, W, D, dtype, ratio))


def wz_condense(features: torch.Tensor, query: torch.Tensor, ratio: float, stream=None):
    """wz_condense: bf16 [T,H,W,D] features, [Lq,D] query -> (tokens [B,D], index [B,3])."""
    features = _cuda_contig(features, "features")
    query = _cuda_contig(query, "query")
    T, H, W, D = features.shape
    B = wz_budget_size(T, H, W, ratio)
    if B < 0:
        raise WaveZipError(ERR_INVALID_ARG, "wz_condense")
    tokens = torch.empty((B, D), dtype=features.dtype, device=features.device)
    index = torch.empty((B, 3), dtype=torch.int32, device=features.device)
    st = _lib.wz_condense(features.data_ptr(), T, H, W, D, query.data_ptr(), query.shape[0], ratio,
                          tokens.data_ptr(), index.data_ptr(), _stream(stream, features.device))
    _check(st, "wz_condense")
    return tokens, index


def _out(t, shape, dtype, dev, name):
    """A caller-given output tensor (checked) or a new one."""
    if t is None:
        return torch.empty(shape, dtype=dtype, device=dev)
    if tuple(t.shape) != tuple(shape) or t.dtype != dtype or t.device != dev or not t.is_contiguous():
        raise ValueError(f"{name}: expected a contiguous {dtype} tensor of shape {tuple(shape)} on {dev}")
    return t


def wz_condense_ex(features: torch.Tensor, query: torch.Tensor, ratio: float, *, lam: float = 1.5,
                   tau: float = 0.0, wsm_wavelet: int = 4, mode="symmetric", path="auto",
                   temporal_mode="wta", spatial_mode="wsm", wta_wavelet: int = 1,
                   token_scores: torch.Tensor | None = None, frame_scores: torch.Tensor | None = None,
                   relevance="mean", wta_levels: int = 1, wsm_levels: int = 1, workspace: torch.Tensor | None = None, out_tokens=None, out_index=None,
                   out_budgets=None, out_count=None, out_relevance=None,
                   device_status: torch.Tensor | None = None, kernel_events=None, stream=None):
    """wz_condense_ex.  Returns a dict with tokens, index, budgets, count and relevance.

    kernel_events: optional list of 2*NUM_KERNELS recorded torch.cuda.Event
    objects; event 2k / 2k+1 is recorded right before / after kernel k.
    token_scores [T, H*W] / frame_scores [T]: float32 device tensors of an
    external scorer (None: the similarity branch's own scores).
    relevance: "mean" (the mean query row) or "maxsim" (maximum cosine over
    the query rows; bf16 features, D % 64 == 0, at most 128 query rows).
    wta_levels / wsm_levels: decomposition levels of the two wavelet modules
    (1..4; the DWT cascades on the approximation band).
    out_*: optional preallocated outputs; with a workspace and the same
    buffers on every call, repeated calls replay one captured CUDA graph."""
    features = _cuda_contig(features, "features")
    query = _cuda_contig(query, "query")
    T, H, W, D = features.shape
    dev = features.device
    B = wz_budget_size(T, H, W, ratio)
    if B < 0:
        raise WaveZipError(ERR_INVALID_ARG, "wz_condense_ex")
    tokens = out_tokens if out_tokens is not None else torch.empty((B, D), dtype=features.dtype, device=dev)
    index = out_index if out_index is not None else torch.empty((B, 3), dtype=torch.int32, device=dev)
    budgets = _out(out_budgets, (T,), torch.int32, dev, "out_budgets")
    count = _out(out_count, (1,), torch.int32, dev, "out_count")
    rel = _out(out_relevance, (T, 4), torch.float32, dev, "out_relevance")
    a = CondenseArgs()
    _lib.wz_condense_args_init(C.byref(a))
    a.features, a.T, a.H, a.W, a.D = features.data_ptr(), T, H, W, D
    a.dtype = _dtype_code(features)
    a.query, a.Lq, a.ratio = query.data_ptr(), query.shape[0], ratio
    a.lam, a.tau, a.wsm_wavelet, a.wta_wavelet = lam, tau, wsm_wavelet, wta_wavelet
    a.mode = MODES[mode] if isinstance(mode, str) else int(mode)
    a.path = PATHS[path] if isinstance(path, str) else int(path)
    a.temporal_mode = _enum(TEMPORAL_MODES, temporal_mode)
    a.spatial_mode = _enum(SPATIAL_MODES, spatial_mode)
    a.relevance_mode = _enum(RELEVANCE_MODES, relevance)
    a.wta_levels, a.wsm_levels = wta_levels, wsm_levels
    if token_scores is not None:
        token_scores = _f32_scores(token_scores, (T, H * W), "token_scores")
        a.token_scores = token_scores.data_ptr()
    if frame_scores is not None:
        frame_scores = _f32_scores(frame_scores, (T,), "frame_scores")
        a.frame_scores = frame_scores.data_ptr()
    a.out_tokens, a.out_index = tokens.data_ptr(), index.data_ptr()
    a.out_budgets, a.out_count, a.out_relevance = budgets.data_ptr(), count.data_ptr(), rel.data_ptr()
    if workspace is not None:
        a.workspace, a.workspace_bytes = workspace.data_ptr(), workspace.numel() * workspace.element_size()
    a.device_status = _ptr(device_status)
    if kernel_events is not None:
        handles = (C.c_void_p * (2 * NUM_KERNELS))(*[e.cuda_event for e in kernel_events])
        a.kernel_events = handles
    a.stream = _stream(stream, dev)
    _check(_lib.wz_condense_ex(C.byref(a)), "wz_condense_ex")
    return {"tokens": tokens, "index": index, "budgets": budgets, "count": count, "relevance": rel}


def wz_condense_host(features: torch.Tensor, query: torch.Tensor, ratio: float, out_tokens: torch.Tensor,
                     out_index: torch.Tensor, *, lam: float = 1.5, tau: float = 0.0, wsm_wavelet: int = 4,
                     wta_wavelet: int = 1, mode="symmetric", path="auto", relevance="mean", stream=None):
    """wz_condense_host: features [T,H,W,D] and query [Lq,D] in (pinned) host memory, out_tokens [B,D]
    and out_index [B,3] host tensors filled once the stream has run the call."""
    for t, name in ((features, "features"), (query, "query"), (out_tokens, "out_tokens"), (out_index, "out_index")):
        if t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous host tensor")
    T, H, W, D = features.shape
    a = CondenseArgs()
    _lib.wz_condense_args_init(C.byref(a))
    a.features, a.T, a.H, a.W, a.D = features.data_ptr(), T, H, W, D
    a.dtype = _dtype_code(features)
    a.query, a.Lq, a.ratio = query.data_ptr(), query.shape[0], ratio
    a.lam, a.tau, a.wsm_wavelet, a.wta_wavelet = lam, tau, wsm_wavelet, wta_wavelet
    a.mode = MODES[mode] if isinstance(mode, str) else int(mode)
    a.path = PATHS[path] if isinstance(path, str) else int(path)
    a.relevance_mode = _enum(RELEVANCE_MODES, relevance)
    a.out_tokens, a.out_index = out_tokens.data_ptr(), out_index.data_ptr()
    a.stream = _stream(stream, torch.device("cuda", torch.cuda.current_device()))
    _check(_lib.wz_condense_host(C.byref(a)), "wz_condense_host")


def wz_batch_rows(V, T, H, W, ratios):
    r = (C.c_float * V)(*ratios)
    offs = (C.c_int64 * (V + 1))()
    rows = _lib.wz_batch_rows(V, T, H, W, r, offs)
    if rows < 0:
        raise WaveZipError(ERR_INVALID_ARG, "wz_batch_rows")
    return int(rows), [int(o) for o in offs]


def wz_condense_batch(features: torch.Tensor, queries: torch.Tensor, Lq, ratios, *, lam: float = 1.5,
                      tau: float = 0.0, wsm_wavelet: int = 4, mode="symmetric", path="auto",
                      temporal_mode="wta", spatial_mode="wsm", wta_wavelet: int = 1, relevance="mean",
                      wta_levels: int = 1, wsm_levels: int = 1, workspace: torch.Tensor | None = None, out_tokens=None, out_index=None,
                      out_budgets=None, out_count=None, out_relevance=None,
                      device_status: torch.Tensor | None = None, kernel_events=None, stream=None):
    """wz_condense_batch: features [V,T,H,W,D], queries [sum Lq, D].  Options as
    for wz_condense_ex; kernel_events brackets each kernel of the whole batch."""
    features = _cuda_contig(features, "features")
    queries = _cuda_contig(queries, "queries")
    V, T, H, W, D = features.shape
    dev = features.device
    rows, offs = wz_batch_rows(V, T, H, W, ratios)
    tokens = out_tokens if out_tokens is not None else torch.empty((rows, D), dtype=features.dtype, device=dev)
    index = out_index if out_index is not None else torch.empty((rows, 3), dtype=torch.int32, device=dev)
    budgets = _out(out_budgets, (V, T), torch.int32, dev, "out_budgets")
    count = _out(out_count, (V,), torch.int32, dev, "out_count")
    rel = _out(out_relevance, (V, T, 4), torch.float32, dev, "out_relevance")
    lq = (C.c_int32 * V)(*[int(x) for x in Lq])
    rt = (C.c_float * V)(*[float(x) for x in ratios])
    ro = (C.c_int64 * (V + 1))()
    a = BatchArgs()
    _lib.wz_batch_args_init(C.byref(a))
    a.V, a.features, a.T, a.H, a.W, a.D = V, features.data_ptr(), T, H, W, D
    a.dtype = _dtype_code(features)
    a.queries, a.Lq, a.ratio = queries.data_ptr(), lq, rt
    a.lam, a.tau, a.wsm_wavelet, a.wta_wavelet = lam, tau, wsm_wavelet, wta_wavelet
    a.mode = MODES[mode] if isinstance(mode, str) else int(mode)
    a.path = PATHS[path] if isinstance(path, str) else int(path)
    a.temporal_mode = _enum(TEMPORAL_MODES, temporal_mode)
    a.spatial_mode = _enum(SPATIAL_MODES, spatial_mode)
    a.relevance_mode = _enum(RELEVANCE_MODES, relevance)
    a.wta_levels, a.wsm_levels = wta_levels, wsm_levels
    a.out_tokens, a.out_index, a.row_offsets = tokens.data_ptr(), index.data_ptr(), ro
    a.out_budgets, a.out_count, a.out_relevance = budgets.data_ptr(), count.data_ptr(), rel.data_ptr()
    if workspace is not None:
        a.workspace, a.workspace_bytes = workspace.data_ptr(), workspace.numel() * workspace.element_size()
    a.device_status = _ptr(device_status)
    if kernel_events is not None:
        handles = (C.c_void_p * (2 * NUM_KERNELS))(*[e.cuda_event for e in kernel_events])
        a.kernel_events = handles
    a.stream = _stream(stream, dev)
    _check(_lib.wz_condense_batch(C.byref(a)), "wz_condense_batch")
    return {"tokens": tokens, "index": index, "budgets": budgets, "count": count, "relevance": rel,
            "row_offsets": [int(ro[v]) for v in range(V + 1)]}


def wz_batch_workspace_size(V, T, H, W, D, dtype, ratios) -> int:
    rt = (C.c_float * V)(*[float(x) for x in ratios])
    return int(_lib.wz_batch_workspace_size(V, T, H, W, D, dtype, rt))


# --------------------------------------------------------------------------
# Relevance and DWT
# --------------------------------------------------------------------------

def wz_relevance(features: torch.Tensor, query: torch.Tensor, *, frame_mean: bool = False,
                 workspace: torch.Tensor | None = None, device_status: torch.Tensor | None = None, stream=None):
    """(token_scores [T,H*W], frame_scores [T], frame_mean [T,D] or None).
    device_status: optional [1] int32 word that a bounded wait which gives up
    ORs a nonzero code into (the caller zeroes it)."""
    features = _cuda_contig(features, "features")
    query = _cuda_contig(query, "query")
    T, H, W, D = features.shape
    dev = features.device
    ts = torch.empty((T, H * W), dtype=torch.float32, device=dev)
    fs = torch.empty((T,), dtype=torch.float32, device=dev)
    fm = torch.empty((T, D), dtype=torch.float32, device=dev) if frame_mean else None
    wsp, wsb = (workspace.data_ptr(), workspace.numel() * workspace.element_size()) if workspace is not None else (None, 0)
    st = _lib.wz_relevance(features.data_ptr(), T, H, W, D, _dtype_code(features), query.data_ptr(),
                           query.shape[0], ts.data_ptr(), fs.data_ptr(), _ptr(fm), wsp, wsb,
                           _ptr(device_status), _stream(stream, dev))
    _check(st, "wz_relevance")
    return ts, fs, fm


def wz_relevance_static(features: torch.Tensor, query: torch.Tensor, *, frame_mean: bool = False,
                        out=None, device_status: torch.Tensor | None = None, stream=None):
    """wz_relevance_static: the scores of wz_relevance without any device allocation
    (its sums live in a fixed array inside the library; see include/wavezip.h).
    out: optional (token_scores, frame_scores, frame_mean or None) tensors to
    write, so that the call itself allocates nothing on the torch side either.
    The call runs with the features' device current (the library picks the
    fixed array of the current device)."""
    features = _cuda_contig(features, "features")
    query = _cuda_contig(query, "query")
    T, H, W, D = features.shape
    dev = features.device
    if out is None:
        ts = torch.empty((T, H * W), dtype=torch.float32, device=dev)
        fs = torch.empty((T,), dtype=torch.float32, device=dev)
        fm = torch.empty((T, D), dtype=torch.float32, device=dev) if frame_mean else None
    else:
        ts, fs, fm = out
    with torch.cuda.device(dev):
        st = _lib.wz_relevance_static(features.data_ptr(), T, H, W, D, _dtype_code(features), query.data_ptr(),
                                      query.shape[0], ts.data_ptr(), fs.data_ptr(), _ptr(fm), _ptr(device_status),
                                      _stream(stream, dev))
    _check(st, "wz_relevance_static")
    return ts, fs, fm


def wz_relevance_workspace_size(T, H, W, D) -> int:
    return int(_lib.wz_relevance_workspace_size(T, H, W, D))


def wz_dwt_len(n: int, wavelet: int = 4) -> int:
    return int(_lib.wz_dwt_len(n, wavelet))


def wavelet_taps(wavelet: int) -> int:
    return 10 if wavelet == WAVELET_BIOR44 else 2 * wavelet


def wz_wavelet_filters(wavelet: int = 4):
    F = wavelet_taps(wavelet)
    bufs = [(C.c_double * F)() for _ in range(4)]
    _check(_lib.wz_wavelet_filters(wavelet, *bufs), "wz_wavelet_filters")
    return {k: [float(x) for x in b] for k, b in zip(("dec_lo", "dec_hi", "rec_lo", "rec_hi"), bufs)}


def wz_dwt1d(x: torch.Tensor, wavelet: int = 4, mode="symmetric", stream=None):
    x = _cuda_contig(x, "x").float()
    rows, L = x.shape
    Lo = wz_dwt_len(L, wavelet)
    cA = torch.empty((rows, Lo), dtype=torch.float32, device=x.device)
    cD = torch.empty_like(cA)
    st = _lib.wz_dwt1d(x.data_ptr(), rows, L, wavelet, MODES[mode] if isinstance(mode, str) else mode,
                       cA.data_ptr(), cD.data_ptr(), _stream(stream, x.device))
    _check(st, "wz_dwt1d")
    return cA, cD


def wz_idwt1d(cA: torch.Tensor, cD: torch.Tensor, L: int, wavelet: int = 4, stream=None):
    cA = _cuda_contig(cA, "cA").float()
    cD = _cuda_contig(cD, "cD").float()
    x = torch.empty((cA.shape[0], L), dtype=torch.float32, device=cA.device)
    st = _lib.wz_idwt1d(cA.data_ptr(), cD.data_ptr(), cA.shape[0], L, wavelet, x.data_ptr(),
                        _stream(stream, cA.device))
    _check(st, "wz_idwt1d")
    return x


def wz_dwt2d(features: torch.Tensor, wavelet: int = 4, mode="symmetric", stream=None):
    features = _cuda_contig(features, "features")
    T, H, W, D = features.shape
    hp, wp = wz_dwt_len(H, wavelet), wz_dwt_len(W, wavelet)
    bands = [torch.empty((T, hp, wp, D), dtype=torch.float32, device=features.device) for _ in range(4)]
    st = _lib.wz_dwt2d(features.data_ptr(), T, H, W, D, _dtype_code(features), wavelet,
                       MODES[mode] if isinstance(mode, str) else mode, *[b.data_ptr() for b in bands],
                       _stream(stream, features.device))
    _check(st, "wz_dwt2d")
    return tuple(bands)


def wz_idwt2d(LL, LH, HL, HH, H: int, W: int, wavelet: int = 4, stream=None):
    bands = [_cuda_contig(b, "band").float() for b in (LL, LH, HL, HH)]
    T, _, _, D = bands[0].shape
    out = torch.empty((T, H, W, D), dtype=torch.float32, device=bands[0].device)
    st = _lib.wz_idwt2d(*[b.data_ptr() for b in bands], T, H, W, D, wavelet, out.data_ptr(),
                        _stream(stream, bands[0].device))
    _check(st, "wz_idwt2d")
    return out


def wz_version() -> int:
    return int(_lib.wz_version())


def wz_graph_cache(capacity: int = -1) -> dict:
    """Set the replay cache's capacity (0 disables it; negative only
    queries).  Returns the capacity in force before the call and the cache's
    counters after it: graphs kept, replays and captures."""
    st = (C.c_int64 * 3)()
    prev = int(_lib.wz_graph_cache(int(capacity), st))
    return {"previous_capacity": prev, "kept": int(st[0]), "replays": int(st[1]), "captures": int(st[2])}


STATUS_WAIT_TIMEOUT = 0x100
STATUS_BOUNDS = 0x200


@contextlib.contextmanager
def checked_library():
    """Route this module's calls to the bounds-checked build of the library
    (libwavezip_checked.so) while the block runs: the same kernels, whose
    global writes check their index and set STATUS_BOUNDS instead of writing
    out of range."""
    global _lib
    saved = _lib
    _lib = _load(LIB_CHECKED_PATH)
    try:
        yield
    finally:
        _lib = saved


def wz_selftest_bounded_wait(timeout_ns: int, device_status: torch.Tensor | None = None, stream=None) -> torch.Tensor:
    """Launch the bounded-wait self-test; returns the [1] int32 status tensor
    (STATUS_WAIT_TIMEOUT set once the kernel has given up)."""
    if device_status is None:
        device_status = torch.zeros((1,), dtype=torch.int32, device="cuda")
    _check(_lib.wz_selftest_bounded_wait(int(timeout_ns), device_status.data_ptr(),
                                         _stream(stream, device_status.device)), "wz_selftest_bounded_wait")
    return device_status


def wz_project_workspace_size(B: int, C_: int) -> int:
    return int(_lib.wz_project_workspace_size(int(B), int(C_)))


def wz_project(tokens: torch.Tensor, w1: torch.Tensor, b1, w2: torch.Tensor, b2, *, out=None,
               workspace: torch.Tensor | None = None, device_status: torch.Tensor | None = None, stream=None):
    """wz_project: GELU(tokens w1^T + b1) w2^T + b2, bf16 in and out (b1, b2 float32 or None)."""
    tokens = _cuda_contig(tokens, "tokens")
    w1 = _cuda_contig(w1, "w1")
    w2 = _cuda_contig(w2, "w2")
    for t, name in ((tokens, "tokens"), (w1, "w1"), (w2, "w2")):
        if t.dtype != torch.bfloat16:
            raise TypeError(f"{name} must be bfloat16")
    B, D = tokens.shape
    C_, E = w1.shape[0], w2.shape[0]
    if w1.shape[1] != D or w2.shape[1] != C_:
        raise ValueError("shapes: tokens [B, D], w1 [C, D], w2 [E, C]")
    biases = []
    for b, n, name in ((b1, C_, "b1"), (b2, E, "b2")):
        if b is not None:
            b = _cuda_contig(b, name)
            if b.dtype != torch.float32 or b.shape != (n,):
                raise ValueError(f"{name} must be float32 of shape ({n},)")
        biases.append(b)
    res = out if out is not None else torch.empty((B, E), dtype=torch.bfloat16, device=tokens.device)
    a = ProjectArgs()
    a.tokens, a.B, a.D, a.w1, a.C, a.w2, a.E = tokens.data_ptr(), B, D, w1.data_ptr(), C_, w2.data_ptr(), E
    a.b1, a.b2 = _ptr(biases[0]), _ptr(biases[1])
    a.out = res.data_ptr()
    if workspace is not None:
        a.workspace, a.workspace_bytes = workspace.data_ptr(), workspace.numel() * workspace.element_size()
    a.device_status = _ptr(device_status)
    a.stream = _stream(stream, tokens.device)
    _check(_lib.wz_project(C.byref(a)), "wz_project")
    return res
