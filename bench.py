#!/usr/bin/env python
"""Benchmark of the WaveZip condensation pass on GB300.

Metric: video frames condensed per second per GB300 (the whole pass: query
pooling, relevance, visual change, WTA, budgets, WSM operator and the fused
condensation GEMM) on the 256-frame 27x27x3584 bf16 workload (~1.3 GB of
tokens, larger than L2, so no L2 flush is needed between steps), with the
achieved HBM bandwidth of the dominant kernel against the measured peak.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--config NAME]

--config picks one of the five synthetic workloads (default: the 256-frame
video); `serving32x64_13x13_bf16` condenses 32 videos in one wz_condense_batch
launch sequence.  The input is the recipe's CPU draw (workload.py), the same
tensor the parity tests compare.  Under torchrun every rank condenses its own
independent inputs (replicas, weak scaling); the time is the max over ranks.
`--impl reference` times the CPU oracle on the host cores instead, the whole
workload per step.  The cpu_baseline leg runs the oracle on the very input the
GPU condensed and reports, beside its time, whether the GPU's outputs of the
timed step match it (budgets and index map bit-exact, tokens within the
stated tolerance).
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "video frames/sec condensed per GB300 (and GB/s vs ~8 TB/s HBM roofline)"
UNIT = "frames/s"
WORKLOAD = "video256_27x27_bf16"
KERNELS = ("query_pool", "relevance", "frame_stats", "temporal", "spatial", "condense")
KERNEL_SOURCES = {"query_pool": "relevance.cu", "relevance": "relevance.cu", "frame_stats": "relevance.cu",
                  "temporal": "temporal.cu", "spatial": "spatial_tc.cu", "condense": "condense_tc.cu"}
L2_BYTES = 129 * 10**6          # GB300 L2
L2_FLUSH_BYTES = 512 << 20
BATCH_CPU_VIDEOS = 16           # cpu_baseline sample of the serving batch: its first 16 videos (~12 s on one core)


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--config", default=WORKLOAD,
                   choices=["tiny_f32_16x14x14", "video64_13x13_bf16", "video128_16x16_objects",
                            "video256_27x27_bf16", "serving32x64_13x13_bf16"])
    p.add_argument("--path", default="auto", choices=["auto", "tensor", "simt"])
    p.add_argument("--e2e-steps", type=int, default=5)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--projector-steps", type=int, default=10,
                   help="also time the projector P (Eq. 17) on the condensed tokens; 0 skips it")
    p.add_argument("--maxsim-steps", type=int, default=10,
                   help="also time the step with the max-over-query scorer; 0 skips it")
    p.add_argument("--graph-steps", type=int, default=20,
                   help="also time the step replayed from a captured CUDA graph; 0 skips it")
    p.add_argument("--variant-steps", type=int, default=5,
                   help="also time the wavelet, level, ablation and external-score variants; 0 skips them")
    return p.parse_args()


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def replica_spec(spec, rank):
    """Each rank condenses its own independent video (replicas, weak scaling)."""
    import workload as wl
    return wl.VideoSpec(**{**spec.__dict__, "seed": spec.seed + 7919 * rank})


class Workload:
    """One benchmark workload: one video, or the serving batch of videos of
    one shape (per-video Lq, ratio and seed)."""

    def __init__(self, name, specs, batch):
        self.name, self.specs, self.batch = name, specs, batch
        s = specs[0]
        self.T, self.H, self.W, self.D, self.dtype = s.T, s.H, s.W, s.D, s.dtype
        self.frames = len(specs) * s.T


def workload(name, rank=0):
    import workload as wl
    if name == wl.BATCH_NAME:
        return Workload(name, [replica_spec(s, rank) for s in wl.batch_specs()], True)
    return Workload(name, [replica_spec(wl.CONFIGS[name], rank)], False)


def draw_inputs(w):
    """Host tensors of the workload: features [T,H,W,D] (or [V,T,H,W,D]) and
    the query rows [Lq,D] (or all videos' rows, [sum Lq, D])."""
    import torch
    import workload as wl
    pairs = [wl.make_video(s)[:2] for s in w.specs]
    if not w.batch:
        return pairs[0]
    return torch.stack([x for x, _ in pairs]), torch.cat([q for _, q in pairs])


def max_over_ranks(x, world, device=None):
    """The slowest rank's value (the job time); a no-op on one rank."""
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_value(frames_per_rank, world, ms):
    """Whole-job frames/s: every rank's frames over the slowest rank's time."""
    return frames_per_rank * world / (ms * 1e-3)


def config_dict(w):
    s = w.specs[0]
    esz = 2 if w.dtype == "bf16" else 4
    fb = w.frames * w.H * w.W * w.D * esz
    d = {"workload": w.name, "T": w.T, "H": w.H, "W": w.W, "D": w.D}
    if w.batch:
        d.update({"videos": len(w.specs), "Lq": [x.Lq for x in w.specs], "ratio": [x.ratio for x in w.specs],
                  "seed": [x.seed for x in w.specs]})
    else:
        d.update({"Lq": s.Lq, "ratio": s.ratio, "seed": s.seed})
    d.update({"features_dtype": w.dtype, "feature_bytes": fb,
              "input": "the recipe's CPU draw (workload.py), the tensor the parity tests use",
              "l2": ("inputs larger than L2 (no flush needed)" if fb > L2_BYTES else
                     "inputs smaller than L2: L2 flushed (512 MB written) before each timed step, "
                     "each step timed alone"),
              "parallelism": "replicas"})
    return d


def measured_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


def measured_tensor_peak():
    """Measured dense bf16 TFLOP/s (burst, sustained) of the GB300s."""
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    except (OSError, KeyError, ValueError):
        return 1900.0, 1700.0, "fallback"


def time_projector(wz, tokens, steps, dev):
    """P (Eq. 17) on this step's condensed tokens [B][D] with random weights of
    an LLM-sized MLP (C = E = D), timed with CUDA events after warm-up."""
    import torch
    B, D = tokens.shape
    g = torch.Generator(device=dev).manual_seed(17)
    w1 = (torch.randn((D, D), device=dev, generator=g) / D ** 0.5).to(torch.bfloat16)
    w2 = (torch.randn((D, D), device=dev, generator=g) / D ** 0.5).to(torch.bfloat16)
    b1 = torch.zeros(D, device=dev)
    b2 = torch.zeros(D, device=dev)
    ws = torch.empty((wz.wz_project_workspace_size(B, D),), dtype=torch.uint8, device=dev)
    out = torch.empty((B, D), dtype=torch.bfloat16, device=dev)
    for _ in range(3):
        wz.wz_project(tokens, w1, b1, w2, b2, out=out, workspace=ws)
    torch.cuda.synchronize(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(steps):
        wz.wz_project(tokens, w1, b1, w2, b2, out=out, workspace=ws)
    e1.record()
    torch.cuda.synchronize(dev)
    ms = e0.elapsed_time(e1) / steps
    # for comparison only (not the product path): PyTorch's cuBLAS GEMMs with
    # torch's erf GELU on the same operands, timed the same way
    b1b = b1.to(torch.bfloat16)
    b2b = b2.to(torch.bfloat16)

    def library():
        hid = torch.nn.functional.gelu(torch.addmm(b1b, tokens, w1.t()))
        return torch.addmm(b2b, hid, w2.t())

    for _ in range(3):
        library()
    torch.cuda.synchronize(dev)
    e0.record()
    for _ in range(steps):
        library()
    e1.record()
    torch.cuda.synchronize(dev)
    lib_ms = e0.elapsed_time(e1) / steps
    flop = 2 * 2.0 * B * D * D
    burst, sustained, kind = measured_tensor_peak()
    achieved = flop / (ms * 1e-3) / 1e12
    return {"config": {"B": B, "D": D, "C": D, "E": D, "hidden": "bf16", "activation": "gelu (erf)"},
            "ms": round(ms, 5), "bound": "tensor", "achieved": round(achieved, 1), "unit": "TFLOP/s",
            "peak": sustained, "frac": round(achieved / sustained, 4), "frac_of_burst": round(achieved / burst, 4),
            "peak_source": kind + " (sustained: a kernel timed in a back-to-back loop)", "launches": 2 * steps,
            "cublas_gelu_ms": round(lib_ms, 5)}


def single_outputs(X, ratio, wz):
    """Caller-owned outputs of one video's call (a stable argument set)."""
    import torch
    T, H, W, D = X.shape
    B = wz.wz_budget_size(T, H, W, ratio)
    return {"out_tokens": torch.empty((B, D), dtype=X.dtype, device=X.device),
            "out_index": torch.empty((B, 3), dtype=torch.int32, device=X.device),
            "out_budgets": torch.empty((T,), dtype=torch.int32, device=X.device),
            "out_count": torch.empty((1,), dtype=torch.int32, device=X.device),
            "out_relevance": torch.empty((T, 4), dtype=torch.float32, device=X.device)}


def time_maxsim(wz, X, Q, ratio, ws, status, steps, dev):
    """The whole step with the max-over-query scorer (same workload), plain
    and with kernel events.  For one video with frames of >= 128 tokens the
    library runs it as one pass over the features (maxsim_pass_kernel: the
    token x query-row GEMM on the tensor cores, the token norms and the
    per-frame channel sums from the same tiles), bracketed by the relevance
    events; otherwise the relevance pass and the per-video GEMM, whose span
    lies between the relevance pass's end event and frame_stats' start."""
    import torch
    stream = torch.cuda.current_stream(dev)
    T, H, W, D = X.shape
    Lq = Q.shape[0]
    Lqp = (Lq + 15) // 16 * 16
    fused = H * W >= 128 and D % 64 == 0 and D <= 4096 and Lqp <= 128
    outs = single_outputs(X, ratio, wz)

    def step(events=None):
        return wz.wz_condense_ex(X, Q, ratio, workspace=ws, device_status=status, relevance="maxsim",
                                 kernel_events=events, **outs)

    for _ in range(3):
        res = step()
    torch.cuda.synchronize(dev)
    active = int((res["budgets"] > 0).sum())
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for _ in range(steps):
        step()
    t1.record(stream)
    torch.cuda.synchronize(dev)
    ms = t0.elapsed_time(t1) / steps
    rel, fs = KERNELS.index("relevance"), KERNELS.index("frame_stats")
    spans, kern = [], {k: [] for k in KERNELS}
    for _ in range(steps):
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * len(KERNELS))]
        for e in ev:
            e.record(stream)   # creates the CUDA event behind the handle
        step(ev)
        torch.cuda.synchronize(dev)
        spans.append(ev[2 * rel].elapsed_time(ev[2 * rel + 1]) if fused else ev[2 * rel + 1].elapsed_time(ev[2 * fs]))
        for j, k in enumerate(KERNELS):
            kern[k].append(ev[2 * j].elapsed_time(ev[2 * j + 1]))
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}: a bounded wait timed out")
    span_ms = statistics.mean(spans)
    tok = T * H * W
    # the features once, a_{t,n} out (the unfused GEMM also reads the ||u|| the relevance pass left)
    nbytes = tok * D * X.element_size() + (4 if fused else 8) * tok
    flop = 2.0 * tok * D * (2 * Lqp)                     # hi and lo halves of the Lqp padded rows
    peak, peak_kind = measured_peak()
    gb_s = nbytes / (span_ms * 1e-3) / 1e9
    name = "pass" if fused else "gemm"
    return {"Lq": Lq, "active_frames": active, "ms_per_step": round(ms, 5), "frames_per_s": round(T / (ms * 1e-3), 1),
            "fused": fused,
            name: {"ms": round(span_ms, 5), "bound": "hbm", "achieved": round(gb_s, 1), "unit": "GB/s",
                   "peak": peak, "frac": round(gb_s / peak, 4), "peak_source": peak_kind,
                   "tflop_s": round(flop / (span_ms * 1e-3) / 1e12, 1)},
            "kernels_ms": {k: round(statistics.mean(v), 5) for k, v in kern.items()},
            "launches_per_step": len(KERNELS) + (1 if fused else 2)}


VARIANTS = [   # (name, wz_condense_ex options): the paper's variant rows on the same video
    ("wta_db4", dict(wta_wavelet=4)),
    ("wsm_haar", dict(wsm_wavelet=1)),
    ("wsm_bior44", dict(wsm_wavelet=44)),
    ("wta_levels3", dict(wta_levels=3)),
    ("wsm_levels2", dict(wsm_levels=2)),
    ("wsm_levels3", dict(wsm_levels=3)),
    ("alloc_raw", dict(temporal_mode="raw")),
    ("alloc_uniform", dict(temporal_mode="uniform")),
    ("spatial_saliency_only", dict(spatial_mode="saliency")),
    ("spatial_none", dict(spatial_mode="none")),
    ("external_scores", None),   # caller-supplied a_{t,n} and r_t
]


def time_variants(wz, X, Q, ratio, ws, status, steps, dev):
    """Each variant: 3 warm-up steps, `steps` plain timed steps, then the same
    steps with kernel events for the per-kernel times."""
    import torch
    stream = torch.cuda.current_stream(dev)
    T, H, W, D = X.shape
    g = torch.Generator(device=dev).manual_seed(23)
    ext = dict(token_scores=torch.rand((T, H * W), device=dev, generator=g),
               frame_scores=0.1 + 0.2 * torch.randn((T,), device=dev, generator=g))
    out = {}
    outs = single_outputs(X, ratio, wz)
    for name, kw in VARIANTS:
        kw = ext if kw is None else kw

        def step(events=None):
            return wz.wz_condense_ex(X, Q, ratio, workspace=ws, device_status=status, kernel_events=events,
                                     **kw, **outs)

        for _ in range(3):
            res = step()
        torch.cuda.synchronize(dev)
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        for _ in range(steps):
            step()
        t1.record(stream)
        torch.cuda.synchronize(dev)
        ms = t0.elapsed_time(t1) / steps
        kern = {k: [] for k in KERNELS}
        for _ in range(steps):
            ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * len(KERNELS))]
            for e in ev:
                e.record(stream)
            step(ev)
            torch.cuda.synchronize(dev)
            for j, k in enumerate(KERNELS):
                kern[k].append(ev[2 * j].elapsed_time(ev[2 * j + 1]))
        out[name] = {"options": {k: v for k, v in kw.items() if not hasattr(v, "shape")} or "external a, r",
                     "ms_per_step": round(ms, 5), "frames_per_s": round(T / (ms * 1e-3), 1),
                     "active_frames": int((res["budgets"] > 0).sum()),
                     "kernels_ms": {k: round(statistics.mean(v), 5) for k, v in kern.items()}}
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}: a bounded wait timed out")
    return out


def source_hash(fname):
    """Hash of a kernel's source file and every shared header it can include."""
    csrc = os.path.join(ROOT, "paper_2607_23265_gb300", "csrc")
    paths = [os.path.join(csrc, fname)] + sorted(os.path.join(csrc, h) for h in os.listdir(csrc) if h.endswith(".cuh"))
    paths.append(os.path.join(ROOT, "include", "wavezip.h"))
    h = hashlib.sha256()
    for p in paths:
        with open(p, "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel, workload_name):
    """dram bytes per launch from the committed ncu summary of this workload,
    if the kernel's source is unchanged since the capture; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(kernel)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("source_sha256_16") != source_hash(KERNEL_SOURCES[kernel]):
        return None
    if rec.get("workload", WORKLOAD).split()[0] != workload_name:
        return None
    return rec.get("dram_bytes_per_launch")


class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.rows = []
        self.proc = None
        try:
            self.proc = subprocess.Popen(["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                                          "-i", str(gpu_index), "-lms", "200"],
                                         stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 9:
                self.rows.append(parts)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.3)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm = [float(r[1]) for r in self.rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in self.rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in self.rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(self.rows)}


# The parity tolerance of condensed tokens for bf16 inputs with fp32
# accumulation: |gpu - oracle| <= 1e-3 + 2e-2 |oracle|, the oracle's value
# rounded to the output dtype first.
TOK_ATOL, TOK_RTOL = 1e-3, 2e-2

_BASELINE_CODE = r"""
import json, sys, time
sys.path.insert(0, %(root)r)
import numpy as np
import oracle as O

d = %(dir)r
meta = json.load(open(d + "/meta.json"))
bits = np.load(d + "/x.npy", mmap_mode="r")
gpu = np.load(d + "/gpu.npz")
Qs = [np.load(d + "/q%%d.npy" %% v) for v in range(meta["V"])]

def f64(a):
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    return a.astype(np.float64)

def bf16_round(x):     # round to nearest even bfloat16, as the output dtype
    f = x.astype(np.float32).view(np.uint32).astype(np.uint64)
    f = (f + 0x7FFF + ((f >> 16) & 1)) & 0xFFFF0000
    return f.astype(np.uint32).view(np.float32).astype(np.float64)

videos = meta["videos"]            # the bounded sample: these videos, whole
secs, frames, res = 0.0, 0, {}
for v in videos:
    x = f64(bits[v] if meta["batch"] else bits)
    t = time.perf_counter()
    r = O.condense(x, Qs[v], meta["ratios"][v])
    secs += time.perf_counter() - t
    frames += x.shape[0]
    res[v] = r
# parity of the GPU's outputs of the timed step on the same input
ok_b = ok_i = ok_t = True
worst, maxerr, rows = 0.0, 0.0, 0
for v in videos:
    r = res[v]
    a, b = meta["row_offsets"][v], meta["row_offsets"][v + 1]
    ok_b &= bool(np.array_equal(gpu["budgets"][v].astype(np.int64), r["budgets"]))
    ok_i &= bool(np.array_equal(gpu["index"][a:b].astype(np.int64), r["out_index"]))
    ref = bf16_round(r["out_tokens"]) if meta["dtype"] == "bf16" else r["out_tokens"].astype(np.float32).astype(np.float64)
    g = gpu["tokens"][a:b].astype(np.float64)
    err = np.abs(g - ref)
    bound = %(atol)r + %(rtol)r * np.abs(ref)
    ok_t &= bool((err <= bound).all())
    if err.size:
        worst = max(worst, float((err / bound).max()))
        maxerr = max(maxerr, float(err.max()))
    rows += b - a
print(json.dumps({"seconds": secs, "frames": frames, "parity": {
    "videos": len(videos), "rows": int(rows), "budgets_equal": ok_b, "index_equal": ok_i,
    "tokens_within_tolerance": ok_t, "max_abs_err": maxerr, "worst_err_over_bound": worst,
    "tolerance": "|g - o| <= %(atol)r + %(rtol)r |o|"}}))
"""

_PARALLEL_CODE = r"""
import json, os, sys, time
sys.path.insert(0, %(root)r)
import numpy as np
from oracle.parallel import condense_parallel, condense_videos_parallel, spawn_pool

d = %(dir)r
meta = json.load(open(d + "/meta.json"))
Qs = [np.load(d + "/q%%d.npy" %% v) for v in range(meta["V"])]
n = os.cpu_count()
pool = spawn_pool(n)
try:
    pool.map(abs, range(n))                     # workers up before the clock starts
    if meta["batch"]:
        t = time.perf_counter()
        condense_videos_parallel(d + "/x.npy", Qs, meta["ratios"], pool)
        dt = time.perf_counter() - t
    else:
        bits = np.load(d + "/x.npy")
        t = time.perf_counter()
        condense_parallel(bits, Qs[0], meta["ratios"][0], n, pool=pool)
        dt = time.perf_counter() - t
finally:
    pool.terminate()
print(json.dumps({"seconds": dt, "frames": meta["frames"], "cores": n}))
"""


def _oracle_env():
    return dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1",
                CUDA_VISIBLE_DEVICES="")


def write_inputs(d, w, Xh, Qh, gpu=None):
    """The step's host inputs (and optionally the GPU's outputs) for the
    oracle legs, in directory d: x.npy (bf16 bit patterns or f32), q<v>.npy
    (fp64), meta.json, gpu.npz."""
    import numpy as np
    import torch
    x = Xh.view(torch.int16).numpy().view(np.uint16) if Xh.dtype == torch.bfloat16 else Xh.numpy()
    np.save(os.path.join(d, "x.npy"), x)
    q0 = 0
    for v, s in enumerate(w.specs):
        np.save(os.path.join(d, f"q{v}.npy"), Qh[q0:q0 + s.Lq].double().numpy())
        q0 += s.Lq
    rows = [0]
    for s in w.specs:
        rows.append(rows[-1] + int(round_half_away(s.ratio * s.T * s.H * s.W)))
    meta = {"V": len(w.specs), "batch": w.batch, "dtype": w.dtype, "ratios": [s.ratio for s in w.specs],
            "row_offsets": rows, "frames": w.frames, "videos": list(range(len(w.specs)))}
    if gpu is not None:
        tok, idx, bud = gpu
        np.savez(os.path.join(d, "gpu.npz"), tokens=tok.float().numpy(), index=idx.numpy(),
                 budgets=bud.reshape(len(w.specs), -1).numpy())
    return meta


def round_half_away(x):
    import math
    return math.floor(x + 0.5)


def cpu_baseline(d, meta, w):
    """The oracle, as it stands, on one host core, on the bench's own input
    (the tensor the GPU condensed): the whole video, or for the serving batch
    the first videos (a bounded sample, ~15 s).  Also checks the GPU's outputs
    of the timed step against the oracle's on that sample."""
    meta = dict(meta)
    if w.batch:
        meta["videos"] = list(range(BATCH_CPU_VIDEOS))
    with open(os.path.join(d, "meta.json"), "w") as f:
        json.dump(meta, f)
    code = _BASELINE_CODE % {"root": ROOT, "dir": d, "atol": TOK_ATOL, "rtol": TOK_RTOL}
    res = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=_oracle_env(),
                         timeout=1200)
    if res.returncode != 0:
        return {"value": None, "unit": UNIT, "cores": 1, "kind": "oracle", "error": res.stderr[-400:]}, None
    r = json.loads(res.stdout.strip().splitlines()[-1])
    sample = (f"the whole {w.T}-frame video the GPU condensed ({w.H}x{w.W}x{w.D} {w.dtype}), fp64 oracle"
              if not w.batch else
              f"the first {BATCH_CPU_VIDEOS} of the {len(w.specs)} videos the GPU condensed "
              f"({w.T} frames of {w.H}x{w.W}x{w.D} {w.dtype} each), fp64 oracle")
    return ({"value": r["frames"] / r["seconds"], "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample,
             "seconds": r["seconds"]}, r["parity"])


def cpu_baseline_parallel(d, meta, w):
    """The second CPU baseline: the oracle's independent steps over a pool of
    spawned processes, one per host core (frames of the video, or whole
    videos of the batch), on the same input as cpu_baseline."""
    if w.dtype != "bf16":
        return None
    with open(os.path.join(d, "meta.json"), "w") as f:
        json.dump(meta, f)
    code = _PARALLEL_CODE % {"root": ROOT, "dir": d}
    res = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=_oracle_env(),
                         timeout=1200)
    if res.returncode != 0:
        return {"value": None, "unit": UNIT, "kind": "oracle over a process pool", "error": res.stderr[-400:]}
    r = json.loads(res.stdout.strip().splitlines()[-1])
    what = "videos" if w.batch else "frames"
    return {"value": r["frames"] / r["seconds"], "unit": UNIT, "cores": r["cores"],
            "kind": f"oracle, {what} over a process pool (one process per core)",
            "sample": f"the whole workload the GPU condensed ({w.frames} frames)", "seconds": r["seconds"]}


def run_reference(args, w, world, rank):
    """The oracle on the host cores, one whole workload per step: the frames
    of the video (or the videos of the batch) spread over one spawned process
    per core, as `oracle/parallel.py` drives it; the fp32 workload (16 small
    frames) on one core."""
    if rank != 0:
        return
    import tempfile

    import numpy as np
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    import oracle as O
    from oracle.parallel import condense_parallel, condense_videos_parallel, spawn_pool
    Xh, Qh = draw_inputs(w)
    n = os.cpu_count() or 1
    Qs, q0 = [], 0
    for s in w.specs:
        Qs.append(Qh[q0:q0 + s.Lq].double().numpy())
        q0 += s.Lq
    with tempfile.TemporaryDirectory() as d:
        pool = None
        if w.dtype == "f32":
            x = Xh.double().numpy()
            cores, kind = 1, "oracle (one core)"

            def step():
                O.condense(x, Qs[0], w.specs[0].ratio)
        else:
            import torch
            pool = spawn_pool(n)
            pool.map(abs, range(n))
            cores = n
            bits = Xh.view(torch.int16).numpy().view(np.uint16)
            if w.batch:
                path = os.path.join(d, "x.npy")
                np.save(path, bits)
                kind = "oracle, videos over a process pool (one process per core)"

                def step():
                    condense_videos_parallel(path, Qs, [s.ratio for s in w.specs], pool)
            else:
                kind = "oracle, frames over a process pool (one process per core)"

                def step():
                    condense_parallel(bits, Qs[0], w.specs[0].ratio, n, pool=pool)
        try:
            for _ in range(args.warmup):
                step()
            t0 = time.perf_counter()
            for _ in range(args.steps):
                step()
            dt = time.perf_counter() - t0
        finally:
            if pool is not None:
                pool.terminate()
    value = w.frames * args.steps / dt
    sample = f"the whole workload per step ({w.frames} frames, the same recipe and seeds as the GPU arm)"
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_dict(w),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": kind, "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def algorithmic_bytes(w, budgets, rows):
    """Bytes each kernel must move per launch (the whole workload).  budgets:
    [V][T] per-frame token counts; rows: total condensed rows."""
    esz = 2 if w.dtype == "bf16" else 4
    N, D, T, V = w.H * w.W, w.D, w.T, len(w.specs)
    K_pad = (N + 31) // 32 * 32
    active = int((budgets > 0).sum())
    return {
        "relevance": V * T * N * D * esz + V * T * N * 4,
        "condense": active * N * D * esz + rows * D * esz + rows * K_pad * 4,
        # operator rows written (bf16 hi + lo) and the pooled gate of each
        # active frame read (db4: (H + 7) / 2 x (W + 7) / 2)
        "spatial": rows * K_pad * 4 + active * ((w.H + 7) // 2) * ((w.W + 7) // 2) * 4,
        "frame_stats": None, "query_pool": None, "temporal": None,
    }


def run_ours(args, w, world, rank, local):
    import tempfile

    import torch
    import torch.distributed as dist

    import paper_2607_23265_gb300.build as build
    build.build()
    import paper_2607_23265_gb300.wavezip as wz

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    Xh, Qh = draw_inputs(w)                       # host tensors (the recipe's CPU draw)
    X, Q = Xh.to(dev), Qh.to(dev)
    ratios = [s.ratio for s in w.specs]
    Lqs = [s.Lq for s in w.specs]
    if w.batch:
        rows, _ = wz.wz_batch_rows(len(w.specs), w.T, w.H, w.W, ratios)
        wsb = wz.wz_batch_workspace_size(len(w.specs), w.T, w.H, w.W, w.D, wz._dtype_code(X), ratios)
    else:
        rows = wz.wz_budget_size(w.T, w.H, w.W, ratios[0])
        wsb = wz.wz_condense_workspace_size(w.T, w.H, w.W, w.D, wz._dtype_code(X), ratios[0])
    ws = torch.empty((wsb,), dtype=torch.uint8, device=dev)
    status = torch.zeros((1,), dtype=torch.int32, device=dev)
    tokens = torch.empty((rows, w.D), dtype=X.dtype, device=dev)
    index = torch.empty((rows, 3), dtype=torch.int32, device=dev)
    # every output caller-owned: the same argument set on every call, which the
    # library's replay cache turns into one captured graph per step
    lead = (len(w.specs),) if w.batch else ()
    outs = {"out_budgets": torch.empty(lead + (w.T,), dtype=torch.int32, device=dev),
            "out_count": torch.empty(lead or (1,), dtype=torch.int32, device=dev),
            "out_relevance": torch.empty(lead + (w.T, 4), dtype=torch.float32, device=dev)}
    stream = torch.cuda.current_stream(dev)
    flush_l2 = X.numel() * X.element_size() <= L2_BYTES

    def step(events=None):
        if w.batch:
            return wz.wz_condense_batch(X, Q, Lqs, ratios, workspace=ws, out_tokens=tokens, out_index=index,
                                        device_status=status, path=args.path, kernel_events=events, **outs)
        return wz.wz_condense_ex(X, Q, ratios[0], workspace=ws, out_tokens=tokens, out_index=index,
                                 device_status=status, path=args.path, kernel_events=events, **outs)

    def barrier():
        torch.cuda.synchronize(dev)
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    evs = []
    for _ in range(args.steps):
        row = [torch.cuda.Event(enable_timing=True) for _ in range(2 * len(KERNELS))]
        for e in row:
            e.record(stream)
        evs.append(row)
    for _ in range(max(3, args.warmup)):
        res = step()
    barrier()
    gpu_index = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")[local] \
        if os.environ.get("CUDA_VISIBLE_DEVICES") else str(local)
    sampler = ClockSampler(gpu_index)
    time.sleep(0.4)
    barrier()
    # timed region: K steps through the public call.  With the caller's
    # workspace and outputs the same on every step, the library replays the
    # graph it captured of the six launches (programmatic-dependency edges
    # inside it); the warm-up steps made and captured it.  Inputs smaller than
    # L2 would stay in it from one step to the next, so for them every step is
    # timed alone with L2 flushed (a 512 MB buffer written) before it.
    flush = torch.empty((L2_FLUSH_BYTES,), dtype=torch.uint8, device=dev) if flush_l2 else None

    def timed_steps():
        # returns (outputs, device ms per step, host us per call: the wall time
        # of the loop that enqueues the steps, which runs ahead of the device)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        if flush_l2:
            marks = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                     for _ in range(args.steps)]
            t0.record(stream)
            h0 = time.perf_counter()
            for k in range(args.steps):
                flush.zero_()
                marks[k][0].record(stream)
                r = step()
                marks[k][1].record(stream)
            h1 = time.perf_counter()
            t1.record(stream)
            barrier()
            return r, sum(a.elapsed_time(b) for a, b in marks) / args.steps, (h1 - h0) * 1e6 / args.steps
        t0.record(stream)
        h0 = time.perf_counter()
        for k in range(args.steps):
            r = step()
        h1 = time.perf_counter()
        t1.record(stream)
        barrier()
        return r, t0.elapsed_time(t1) / args.steps, (h1 - h0) * 1e6 / args.steps

    cache0 = wz.wz_graph_cache(-1)
    res, step_ms, host_us = timed_steps()
    cache1 = wz.wz_graph_cache(-1)
    # the same K steps with the replay cache off: six launches per step
    cap = wz.wz_graph_cache(0)["previous_capacity"]
    for _ in range(3):
        step()
    barrier()
    _, direct_ms, direct_host_us = timed_steps()
    wz.wz_graph_cache(cap)
    for _ in range(3):
        step()
    barrier()
    # the same K steps again with an event pair around every kernel: the
    # per-kernel durations (an event between two launches removes their
    # overlap, so this pass is slower per step and reported separately)
    t2 = torch.cuda.Event(enable_timing=True)
    t3 = torch.cuda.Event(enable_timing=True)
    t2.record(stream)
    for k in range(args.steps):
        res = step(evs[k])
    t3.record(stream)
    barrier()
    clocks = sampler.stop()
    ms = max_over_ranks(step_ms, world, dev)
    direct_ms = max_over_ranks(direct_ms, world, dev)
    ms_instr = max_over_ranks(t2.elapsed_time(t3) / args.steps, world, dev)
    kern_ms = {name: statistics.mean(evs[k][2 * j].elapsed_time(evs[k][2 * j + 1]) for k in range(args.steps))
               for j, name in enumerate(KERNELS)}
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}: a bounded wait timed out")
    budgets = res["budgets"].cpu()
    gpu_out = (tokens.cpu(), index.cpu(), budgets)

    # end to end through the public API: pinned host buffers in, results out
    Xp = Xh.pin_memory()
    Qp = Qh.pin_memory()
    tok_h = torch.empty((rows, w.D), dtype=X.dtype).pin_memory()
    idx_h = torch.empty((rows, 3), dtype=torch.int32).pin_memory()
    if w.batch:
        Xd = torch.empty_like(X)
        Qd = torch.empty_like(Q)

        def e2e_step():
            # copies in, the batch call, copies out, all on the stream
            Xd.copy_(Xp, non_blocking=True)
            Qd.copy_(Qp, non_blocking=True)
            wz.wz_condense_batch(Xd, Qd, Lqs, ratios, workspace=ws, out_tokens=tokens, out_index=index,
                                 device_status=status, path=args.path, **outs)
            tok_h.copy_(tokens, non_blocking=True)
            idx_h.copy_(index, non_blocking=True)
        e2e_path = "pinned host -> device copies, wz_condense_batch, device -> pinned host copies on one stream"
    else:
        def e2e_step():
            # the C-ABI call on host buffers: copies in, the pass, copies out, all on the stream
            wz.wz_condense_host(Xp, Qp, ratios[0], tok_h, idx_h, path=args.path)
        e2e_path = "wz_condense_host (C ABI, pinned host buffers)"

    e2e_ms = None
    if args.e2e_steps > 0:
        e2e_step()
        barrier()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.e2e_steps):
            e2e_step()
        e1.record(stream)
        barrier()
        e2e_ms = max_over_ranks(e0.elapsed_time(e1) / args.e2e_steps, world, dev)

    # the same step captured once in a CUDA graph and replayed (launches of the
    # six kernels submitted as one graph)
    graph = None
    if args.graph_steps > 0 and not w.batch:
        gs = torch.cuda.Stream(dev)
        gs.wait_stream(stream)
        with torch.cuda.stream(gs):
            wz.wz_condense_ex(X, Q, ratios[0], workspace=ws, out_tokens=tokens, out_index=index,
                              device_status=status, path=args.path, stream=gs)
        torch.cuda.synchronize(dev)
        cg = torch.cuda.CUDAGraph()
        with torch.cuda.graph(cg, stream=gs):
            wz.wz_condense_ex(X, Q, ratios[0], workspace=ws, out_tokens=tokens, out_index=index,
                              device_status=status, path=args.path, stream=gs)
        for _ in range(3):
            cg.replay()
        barrier()
        g0, g1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        for _ in range(args.graph_steps):
            cg.replay()
        g1.record(stream)
        barrier()
        gms = max_over_ranks(g0.elapsed_time(g1) / args.graph_steps, world, dev)
        graph = {"ms_per_step": round(gms, 5), "value": job_value(w.frames, world, gms), "unit": UNIT,
                 "steps": args.graph_steps}
        del cg

    single_bf16 = not w.batch and X.dtype == torch.bfloat16
    projector = time_projector(wz, tokens, args.projector_steps, dev) \
        if args.projector_steps > 0 and single_bf16 and w.D % 64 == 0 else None
    maxsim = time_maxsim(wz, X, Q, ratios[0], ws, status, args.maxsim_steps, dev) \
        if args.maxsim_steps > 0 and single_bf16 and w.D % 64 == 0 else None
    variants = time_variants(wz, X, Q, ratios[0], ws, status, args.variant_steps, dev) \
        if args.variant_steps > 0 and not w.batch else None

    if rank == 0:
        peak, peak_kind = measured_peak()
        ab = algorithmic_bytes(w, budgets.reshape(len(w.specs), -1), rows)
        dominant = max(KERNELS, key=lambda k: kern_ms[k])
        kern = {}
        for k in KERNELS:
            entry = {"ms": round(kern_ms[k], 5), "share": round(kern_ms[k] / sum(kern_ms.values()), 4)}
            if ab.get(k):
                entry["bytes"] = ab[k]
                entry["gb_s"] = round(ab[k] / (kern_ms[k] * 1e-3) / 1e9, 1)
                entry["frac"] = round(ab[k] / (kern_ms[k] * 1e-3) / 1e9 / peak, 4)
            kern[k] = entry
        bytes_dom = ab.get(dominant)
        achieved = bytes_dom / (kern_ms[dominant] * 1e-3) / 1e9 if bytes_dom else None
        out = {
            "metric": METRIC, "value": job_value(w.frames, world, ms), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
            "data": "synthetic", "config": config_dict(w),
            "tokens_out_per_s": rows * world / (ms * 1e-3),
            "roofline": {"bound": "hbm", "kernel": dominant, "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak if achieved else None,
                         "traffic": recorded_traffic(dominant, w.name), "peak_source": peak_kind,
                         "frac_of_8000": achieved / 8000.0 if achieved else None},
            "kernels": kern,
            "ms_per_step_with_kernel_events": ms_instr,
            "active_frames": int((budgets > 0).sum()), "rows": rows,
            "e2e": {"value": job_value(w.frames, world, e2e_ms) if e2e_ms else None, "unit": UNIT, "path": e2e_path,
                    "h2d_bytes_per_step": X.numel() * X.element_size() + Q.numel() * Q.element_size(),
                    "d2h_bytes_per_step": tokens.numel() * tokens.element_size() + index.numel() * 4},
            "clocks": clocks,
            "gpu_launches": len(KERNELS) * args.steps,
            "projector": projector,
            "launch": {"replay_cache": {"replays_in_timed_steps": cache1["replays"] - cache0["replays"],
                                        "captures_in_timed_steps": cache1["captures"] - cache0["captures"],
                                        "host_us_per_call": round(host_us, 1)},
                       "direct_launches": {"ms_per_step": round(direct_ms, 5),
                                           "value": job_value(w.frames, world, direct_ms), "unit": UNIT,
                                           "host_us_per_call": round(direct_host_us, 1)}},
            "graph": graph,
            "maxsim": maxsim,
            "variants": variants,
        }
        if world == 1 and not args.no_cpu_baseline:
            with tempfile.TemporaryDirectory() as d:
                meta = write_inputs(d, w, Xh, Qh, gpu_out)
                out["cpu_baseline"], out["parity"] = cpu_baseline(d, meta, w)
                out["cpu_baseline_parallel"] = cpu_baseline_parallel(d, meta, w)
        print(json.dumps(out))
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    world, rank, local = dist_setup()
    w = workload(args.config, rank)
    if args.impl == "reference":
        run_reference(args, w, world, rank)
    else:
        run_ours(args, w, world, rank, local)


if __name__ == "__main__":
    main()
