#!/usr/bin/env python
"""Benchmark of the WaveZip condensation pass on GB300.

Metric: video frames condensed per second per GB300 (the whole pass: query
pooling, relevance, visual change, WTA, budgets, WSM operator and the fused
condensation GEMM) on the 256-frame 27x27x3584 bf16 workload (~1.3 GB of
tokens, larger than L2, so no L2 flush is needed between steps), with the
achieved HBM bandwidth of the dominant kernel against the measured peak.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Under torchrun every rank condenses its own independent video (replicas, weak
scaling); the time is the max over ranks.  `--impl reference` times the CPU
oracle on a bounded sample of the same workload instead.
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
                  "temporal": "temporal.cu", "spatial": "spatial.cu", "condense": "condense_tc.cu"}
CPU_SAMPLE_FRAMES = 256         # oracle sample for the cpu_baseline leg: the whole 256-frame video (~15 s on one core)
REF_SAMPLE_FRAMES = 16          # oracle sample per step of the reference arm


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--config", default=WORKLOAD)
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


def config_dict(spec, name):
    return {"workload": name, "T": spec.T, "H": spec.H, "W": spec.W, "D": spec.D, "Lq": spec.Lq,
            "ratio": spec.ratio, "features_dtype": spec.dtype, "seed": spec.seed,
            "feature_bytes": spec.T * spec.H * spec.W * spec.D * (2 if spec.dtype == "bf16" else 4),
            "l2": "inputs larger than L2 (no flush needed)", "parallelism": "replicas"}


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
    flop = 2 * 2.0 * B * D * D
    burst, sustained, kind = measured_tensor_peak()
    achieved = flop / (ms * 1e-3) / 1e12
    return {"config": {"B": B, "D": D, "C": D, "E": D, "hidden": "bf16", "activation": "gelu (erf)"},
            "ms": round(ms, 5), "bound": "tensor", "achieved": round(achieved, 1), "unit": "TFLOP/s",
            "peak": sustained, "frac": round(achieved / sustained, 4), "frac_of_burst": round(achieved / burst, 4),
            "peak_source": kind + " (sustained: a kernel timed in a back-to-back loop)", "launches": 2 * steps}


def time_maxsim(wz, X, Q, ratio, ws, status, steps, dev):
    """The whole step with the max-over-query scorer (same workload), plain
    and with kernel events; the token x query-row GEMM (and the small
    query-row kernel before it) is the span between the relevance pass's
    end event and frame_stats' start event."""
    import torch
    stream = torch.cuda.current_stream(dev)
    T, H, W, D = X.shape
    Lq = Q.shape[0]
    Lqp = (Lq + 15) // 16 * 16

    def step(events=None):
        return wz.wz_condense_ex(X, Q, ratio, workspace=ws, device_status=status, relevance="maxsim",
                                 kernel_events=events)

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
        spans.append(ev[2 * rel + 1].elapsed_time(ev[2 * fs]))
        for j, k in enumerate(KERNELS):
            kern[k].append(ev[2 * j].elapsed_time(ev[2 * j + 1]))
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}: a bounded wait timed out")
    gemm_ms = statistics.mean(spans)
    tok = T * H * W
    nbytes = tok * D * X.element_size() + 2 * 4 * tok   # features once, ||u|| in and a_{t,n} out
    flop = 2.0 * tok * D * (2 * Lqp)                     # hi and lo halves of the Lqp padded rows
    peak, peak_kind = measured_peak()
    gb_s = nbytes / (gemm_ms * 1e-3) / 1e9
    return {"Lq": Lq, "active_frames": active, "ms_per_step": round(ms, 5), "frames_per_s": round(T / (ms * 1e-3), 1),
            "gemm": {"ms": round(gemm_ms, 5), "bound": "hbm", "achieved": round(gb_s, 1), "unit": "GB/s",
                     "peak": peak, "frac": round(gb_s / peak, 4), "peak_source": peak_kind,
                     "tflop_s": round(flop / (gemm_ms * 1e-3) / 1e12, 1)},
            "kernels_ms": {k: round(statistics.mean(v), 5) for k, v in kern.items()},
            "launches_per_step": len(KERNELS) + 2}


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
    for name, kw in VARIANTS:
        kw = ext if kw is None else kw

        def step(events=None):
            return wz.wz_condense_ex(X, Q, ratio, workspace=ws, device_status=status, kernel_events=events, **kw)

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


def recorded_traffic(kernel):
    """dram bytes per launch from the committed ncu summary, if the kernel's
    source is unchanged since the capture; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as f:
            rec = json.load(f).get(kernel)
    except (OSError, ValueError):
        return None
    if not rec or rec.get("source_sha256_16") != source_hash(KERNEL_SOURCES[kernel]):
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


def cpu_baseline(spec, frames):
    """Time the oracle, as it stands, on one host core: a `frames`-frame video
    drawn with the same recipe.  Runs in a fresh interpreter pinned to one BLAS
    thread."""
    code = (
        "import json,sys,time; sys.path.insert(0, %r)\n"
        "import workload as wl, oracle as O\n"
        "s = wl.VideoSpec(T=%d, H=%d, W=%d, D=%d, dtype=%r, Lq=%d, ratio=%r, ar=%r, cuts=%d, seed=%d)\n"
        "X, Q, _ = wl.make_video(s)\n"
        "x, q = X.double().numpy(), Q.double().numpy()\n"
        "t = time.perf_counter(); O.condense(x, q, s.ratio); dt = time.perf_counter() - t\n"
        "print(json.dumps({'seconds': dt, 'frames': s.T}))\n"
    ) % (ROOT, frames, spec.H, spec.W, spec.D, spec.dtype, spec.Lq, spec.ratio, spec.ar,
         max(1, spec.cuts * frames // spec.T), spec.seed)
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    res = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=900)
    if res.returncode != 0:
        return {"value": None, "unit": UNIT, "cores": 1, "kind": "oracle", "error": res.stderr[-400:]}
    r = json.loads(res.stdout.strip().splitlines()[-1])
    return {"value": r["frames"] / r["seconds"], "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"first {frames} frames of the workload recipe ({spec.H}x{spec.W}x{spec.D} "
                      f"{spec.dtype}, Lq={spec.Lq}, ratio={spec.ratio}) condensed by the fp64 oracle",
            "seconds": r["seconds"]}


def cpu_baseline_parallel(spec, frames):
    """The oracle's per-frame steps spread over every host core (spawned
    processes, frames sharing one block of shared memory), the coupling steps
    in the parent: the second CPU baseline.  Same video as cpu_baseline."""
    code = (
        "import json,os,sys,time; sys.path.insert(0, %r)\n"
        "import numpy as np, torch, workload as wl\n"
        "from oracle.parallel import condense_parallel\n"
        "s = wl.VideoSpec(T=%d, H=%d, W=%d, D=%d, dtype=%r, Lq=%d, ratio=%r, ar=%r, cuts=%d, seed=%d)\n"
        "X, Q, _ = wl.make_video(s)\n"
        "bits, q = X.view(torch.int16).numpy().view(np.uint16), Q.double().numpy()\n"
        "n = os.cpu_count()\n"
        "t = time.perf_counter(); condense_parallel(bits, q, s.ratio, n); dt = time.perf_counter() - t\n"
        "print(json.dumps({'seconds': dt, 'frames': s.T, 'cores': n}))\n"
    ) % (ROOT, frames, spec.H, spec.W, spec.D, spec.dtype, spec.Lq, spec.ratio, spec.ar,
         max(1, spec.cuts * frames // spec.T), spec.seed)
    env = dict(os.environ, OPENBLAS_NUM_THREADS="1", OMP_NUM_THREADS="1", MKL_NUM_THREADS="1",
               CUDA_VISIBLE_DEVICES="")
    if spec.dtype != "bf16":
        return None
    res = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=900)
    if res.returncode != 0:
        return {"value": None, "unit": UNIT, "kind": "oracle, frames over a process pool", "error": res.stderr[-400:]}
    r = json.loads(res.stdout.strip().splitlines()[-1])
    return {"value": r["frames"] / r["seconds"], "unit": UNIT, "cores": r["cores"],
            "kind": "oracle, per-frame steps over a process pool (one process per core)",
            "sample": f"the same {frames}-frame video as cpu_baseline", "seconds": r["seconds"]}


def run_reference(args, spec, world, rank):
    """The oracle, timed on the host cores, on a bounded sample per step."""
    if rank != 0:
        return
    os.environ.setdefault("OPENBLAS_NUM_THREADS", "1")
    import oracle as O
    import workload as wl
    frames = REF_SAMPLE_FRAMES
    s = wl.VideoSpec(**{**spec.__dict__, "T": frames, "cuts": max(1, spec.cuts * frames // spec.T)})
    X, Q, _ = wl.make_video(s)
    x, q = X.double().numpy(), Q.double().numpy()
    for _ in range(args.warmup):
        O.condense(x, q, s.ratio)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        O.condense(x, q, s.ratio)
    dt = time.perf_counter() - t0
    value = frames * args.steps / dt
    sample = f"{frames}-frame video per step ({spec.H}x{spec.W}x{spec.D} {spec.dtype}, same recipe), fp64 oracle"
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_dict(spec, args.config),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": 1, "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


def algorithmic_bytes(spec, budgets, B, K_pad):
    """Bytes each kernel must move per launch (one video)."""
    esz = 2 if spec.dtype == "bf16" else 4
    N, D, T = spec.H * spec.W, spec.D, spec.T
    active = int((budgets > 0).sum())
    return {
        "relevance": T * N * D * esz + T * N * 4,
        "condense": active * N * D * esz + B * D * esz + B * K_pad * 4,
        # operator rows written (bf16 hi + lo) and the pooled gate of each
        # active frame read (db4: (H + 7) / 2 x (W + 7) / 2)
        "spatial": B * K_pad * 4 + active * ((spec.H + 7) // 2) * ((spec.W + 7) // 2) * 4,
        "frame_stats": None, "query_pool": None, "temporal": None,
    }


def run_ours(args, spec, world, rank, local):
    import torch
    import torch.distributed as dist

    import paper_2607_23265_gb300.build as build
    build.build()
    import paper_2607_23265_gb300.wavezip as wz
    import workload as wl

    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    X, Q, _ = wl.make_video(replica_spec(spec, rank), device=dev)
    T, H, W, D = X.shape
    B = wz.wz_budget_size(T, H, W, spec.ratio)
    K_pad = (H * W + 31) // 32 * 32
    ws = torch.empty((wz.wz_condense_workspace_size(T, H, W, D, wz._dtype_code(X), spec.ratio),),
                     dtype=torch.uint8, device=dev)
    status = torch.zeros((1,), dtype=torch.int32, device=dev)
    tokens = torch.empty((B, D), dtype=X.dtype, device=dev)
    index = torch.empty((B, 3), dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(events=None):
        return wz.wz_condense_ex(X, Q, spec.ratio, workspace=ws, out_tokens=tokens, out_index=index,
                                 device_status=status, path=args.path, kernel_events=events)

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
    # timed region: K plain steps (consecutive launches overlap through
    # programmatic dependent launch)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for k in range(args.steps):
        res = step()
    t1.record(stream)
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
    ms = max_over_ranks(t0.elapsed_time(t1) / args.steps, world, dev)
    ms_instr = max_over_ranks(t2.elapsed_time(t3) / args.steps, world, dev)
    kern_ms = {name: statistics.mean(evs[k][2 * j].elapsed_time(evs[k][2 * j + 1]) for k in range(args.steps))
               for j, name in enumerate(KERNELS)}
    if int(status.item()) != 0:
        raise RuntimeError(f"device status {int(status.item())}: a bounded wait timed out")
    budgets = res["budgets"].cpu()

    # end to end through the public API: pinned host buffers in, results out
    Xh = X.cpu().pin_memory()
    Qh = Q.cpu().pin_memory()
    tok_h = torch.empty((B, D), dtype=X.dtype).pin_memory()
    idx_h = torch.empty((B, 3), dtype=torch.int32).pin_memory()

    def e2e_step():
        # the C-ABI call on host buffers: copies in, the pass, copies out, all on the stream
        wz.wz_condense_host(Xh, Qh, spec.ratio, tok_h, idx_h, path=args.path)

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
    if args.graph_steps > 0:
        gs = torch.cuda.Stream(dev)
        gs.wait_stream(stream)
        with torch.cuda.stream(gs):
            wz.wz_condense_ex(X, Q, spec.ratio, workspace=ws, out_tokens=tokens, out_index=index,
                              device_status=status, path=args.path, stream=gs)
        torch.cuda.synchronize(dev)
        cg = torch.cuda.CUDAGraph()
        with torch.cuda.graph(cg, stream=gs):
            wz.wz_condense_ex(X, Q, spec.ratio, workspace=ws, out_tokens=tokens, out_index=index,
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
        graph = {"ms_per_step": round(gms, 5), "value": job_value(T, world, gms), "unit": UNIT,
                 "steps": args.graph_steps}
        del cg

    projector = time_projector(wz, tokens, args.projector_steps, dev) if args.projector_steps > 0 else None
    maxsim = time_maxsim(wz, X, Q, spec.ratio, ws, status, args.maxsim_steps, dev) \
        if args.maxsim_steps > 0 and X.dtype == torch.bfloat16 and D % 64 == 0 else None
    variants = time_variants(wz, X, Q, spec.ratio, ws, status, args.variant_steps, dev) \
        if args.variant_steps > 0 else None

    if rank == 0:
        peak, peak_kind = measured_peak()
        ab = algorithmic_bytes(spec, budgets, B, K_pad)
        dominant = max(KERNELS, key=lambda k: kern_ms[k])
        kern = {}
        for k in KERNELS:
            entry = {"ms": round(kern_ms[k], 5), "share": round(kern_ms[k] / sum(kern_ms.values()), 4)}
            if ab.get(k):
                entry["gb_s"] = round(ab[k] / (kern_ms[k] * 1e-3) / 1e9, 1)
            kern[k] = entry
        bytes_dom = ab.get(dominant)
        achieved = bytes_dom / (kern_ms[dominant] * 1e-3) / 1e9 if bytes_dom else None
        frames = T * world
        out = {
            "metric": METRIC, "value": job_value(T, world, ms), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": max(3, args.warmup), "ms_per_step": ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
            "data": "synthetic", "config": config_dict(spec, args.config),
            "tokens_out_per_s": B * world / (ms * 1e-3),
            "roofline": {"bound": "hbm", "kernel": dominant, "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak if achieved else None,
                         "traffic": recorded_traffic(dominant), "peak_source": peak_kind,
                         "frac_of_8000": achieved / 8000.0 if achieved else None},
            "kernels": kern,
            "ms_per_step_with_kernel_events": ms_instr,
            "active_frames": int((budgets > 0).sum()), "budget_B": B,
            "e2e": {"value": job_value(T, world, e2e_ms), "unit": UNIT,
                    "h2d_bytes_per_step": X.numel() * X.element_size() + Q.numel() * Q.element_size(),
                    "d2h_bytes_per_step": tokens.numel() * tokens.element_size() + index.numel() * 4},
            "clocks": clocks,
            "gpu_launches": len(KERNELS) * args.steps,
            "projector": projector,
            "graph": graph,
            "maxsim": maxsim,
            "variants": variants,
        }
        if world == 1 and not args.no_cpu_baseline:
            out["cpu_baseline"] = cpu_baseline(spec, CPU_SAMPLE_FRAMES)
            out["cpu_baseline_parallel"] = cpu_baseline_parallel(spec, CPU_SAMPLE_FRAMES)
        print(json.dumps(out))
    if world > 1:
        dist.destroy_process_group()


def main():
    args = parse()
    world, rank, local = dist_setup()
    import workload as wl
    spec = wl.CONFIGS[args.config]
    if args.impl == "reference":
        run_reference(args, spec, world, rank)
    else:
        run_ours(args, spec, world, rank, local)


if __name__ == "__main__":
    main()
