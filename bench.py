#!/usr/bin/env python3
"""Benchmark: batched complex64 DFT on GB300 tensor cores.

Default workload: n = 65536 (= 16^4, sqrt_m = 16), batch = 1024, N(0,1)
inputs from seed 1, forward, 3xTF32.  One "step" is one complete forward
transform of the whole batch (every stage of every pass), inputs resident in
HBM (512 MiB, larger than the 129 MB L2, so no flush is needed between
steps; a workload whose buffers are smaller than twice the L2 gets an
untimed 512 MiB write before every step, and its step time is the sum of
the steps' own events).

Prints ONE JSON line on stdout (rank 0).  Logs go to stderr.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

For N > 1 launch under torchrun: each rank transforms its own batch (weak
scaling, no collective on the data path; one all-reduce of the timings).
``--impl reference`` times the fp64 CPU oracle on the host cores on bounded
samples of the same workload.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import inputs  # noqa: E402

METRIC = ("DFT GFLOP/s (5n·log2n) & % of roofline, n=2^16 ×1024 "
          "complex64, 1×GB300")
UNIT = "GFLOP/s"


def metric_for(wl):
    """The headline metric's name, with the sizes of the workload timed
    (the default workload gives exactly the headline's name)."""
    n, batch = wl["n"], wl["batch"]
    ns = "2^%d" % (n.bit_length() - 1) if n & (n - 1) == 0 else str(n)
    return ("DFT GFLOP/s (5n·log2n) & %% of roofline, n=%s ×%d complex64, "
            "1×GB300" % (ns, batch))
# nominal dense tensor rates (PFLOP/s): ratio used to scale the measured bf16
# peak to tf32
NOMINAL_BF16 = 2.25
NOMINAL_TF32 = 1.1
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0,
                  "bf16_tflops_sustained": 1700.0}


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def dft_flops(n, batch):
    return 5.0 * n * math.log2(n) * batch


def measure_tf32_tflops(dev, size=8192, reps=10):
    """Dense TF32 tensor throughput of this GPU (TFLOP/s): the best of
    `reps` cuBLAS GEMMs of size^3 with TF32 enabled; None on any failure."""
    import torch
    prev = torch.backends.cuda.matmul.allow_tf32
    try:
        torch.backends.cuda.matmul.allow_tf32 = True
        a = torch.randn(size, size, device=dev)
        b = torch.randn(size, size, device=dev)
        c = torch.empty(size, size, device=dev)
        for _ in range(3):
            torch.matmul(a, b, out=c)
        best = None
        for _ in range(reps):
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            torch.matmul(a, b, out=c)
            e1.record()
            torch.cuda.synchronize()
            ms = e0.elapsed_time(e1)
            best = ms if best is None else min(best, ms)
        del a, b, c
        return 2.0 * size ** 3 / (best * 1e-3) / 1e12
    except Exception:
        return None
    finally:
        torch.backends.cuda.matmul.allow_tf32 = prev


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    except Exception:
        return dict(FALLBACK_PEAKS), "fallback"


class ClockSampler:
    """nvidia-smi clocks/throttle sampling during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,"
         "clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + self.Q,
                 "--format=csv,noheader,nounits", "-lms", "50"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.t.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown",
                 "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for nm, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [],
                    "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "reasons": sorted(reasons), "samples": len(sm)}


def kernel_sources_sha256():
    """sha256 over the kernel sources (csrc/*.cu, *.cuh, *.h, name order)."""
    import glob
    import hashlib
    csrc = os.path.join(ROOT, "paper_1908_06649_gb300", "csrc")
    files = sorted(glob.glob(os.path.join(csrc, "*.cu"))
                   + glob.glob(os.path.join(csrc, "*.cuh"))
                   + glob.glob(os.path.join(csrc, "*.h")))
    h = hashlib.sha256()
    for f in files:
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def profiled_traffic(batch, fused):
    """DRAM bytes per launch of the dominant kernel from the committed ncu
    summary, scaled to `batch`; None if the kernel changed since."""
    if fused:
        return None
    p = os.path.join(ROOT, "profiles", "traffic_dft_pass_kernel_n65536.txt")
    try:
        kv = {}
        with open(p) as f:
            for line in f:
                if ":" in line and not line.startswith("#"):
                    k, v = line.split(":", 1)
                    kv[k.strip()] = v.strip()
        if kv.get("sources_sha256") != kernel_sources_sha256():
            return None
        return (float(kv["dram_bytes_per_launch_b512"]) * batch
                / float(kv["profiled_batch"]))
    except Exception:
        return None


def copy_floor_ms(h_in, h_out, d_in, d_out, stream, reps=3):
    """Least time to copy h_in -> d_in and d_out -> h_out at once (one
    cudaMemcpyAsync each, on two streams): the link's floor for a step of the
    end-to-end path, which must move these bytes whatever the transform."""
    import torch
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    f0 = torch.cuda.Event(enable_timing=True)
    f1 = torch.cuda.Event(enable_timing=True)
    best = None
    for _ in range(reps):
        torch.cuda.synchronize()
        f0.record(stream)
        s_in.wait_event(f0)
        s_out.wait_event(f0)
        with torch.cuda.stream(s_in):
            d_in.copy_(h_in, non_blocking=True)
        with torch.cuda.stream(s_out):
            h_out.copy_(d_out, non_blocking=True)
        stream.wait_stream(s_in)
        stream.wait_stream(s_out)
        f1.record(stream)
        torch.cuda.synchronize()
        t = f0.elapsed_time(f1)
        best = t if best is None else min(best, t)
    return best


def rank_seed(wl, rank):
    """Each rank transforms its own batch (weak scaling): the workload's
    recipe with the seed offset by 1000 * rank."""
    return wl["seed"] + 1000 * rank


def max_over_ranks(value, dist, device):
    """Max of a float over all ranks (the slowest rank sets the job time);
    identity without a process group."""
    if dist is None:
        return float(value)
    import torch
    t = torch.tensor([float(value)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(units_per_rank, world, steps, elapsed_ms):
    """Whole-job GFLOP/s: the work of every rank over the max time."""
    return units_per_rank * world * steps / (elapsed_ms * 1e-3) / 1e9


def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def cpu_baseline(wl, seconds=10.0, sample=32, y_gpu=None, tol=None):
    """The fp64 oracle (radix-2 FFT) on a bounded sample of the workload,
    using every host core; returns the metric in GFLOP/s.  With y_gpu (the
    GPU's outputs for the same first `sample` transforms) it also returns
    their per-transform relative L2 error against the oracle's outputs."""
    import oracle
    n = wl["n"]
    x = inputs.make(wl["kind"], n, wl["batch"], wl["seed"], first=0,
                    count=sample)
    threads = oracle.default_threads()
    done, used, t0 = 0, 1, time.perf_counter()
    ref = None
    while True:
        ref, used = oracle.fft_radix2_timed(x, threads=threads)
        done += sample
        el = time.perf_counter() - t0
        if el >= seconds:
            break
    # one core on a 1/64 subset of the sample, scaled to the same unit
    x1 = x[:max(1, sample // 64)]
    done1, t1 = 0, time.perf_counter()
    while time.perf_counter() - t1 < min(3.0, seconds / 3):
        oracle.fft_radix2_timed(x1, threads=1)
        done1 += x1.shape[0]
    el1 = time.perf_counter() - t1
    direct = None
    if n <= 4096:
        # the definition itself (O(n^2) per transform), for the small workload
        nd, t2 = 0, time.perf_counter()
        while time.perf_counter() - t2 < min(3.0, seconds / 3):
            oracle.dft_direct(x, threads=threads)
            nd += sample
        el2 = time.perf_counter() - t2
        direct = {"value": dft_flops(n, nd) / el2 / 1e9, "unit": UNIT,
                  "sample": "%d transforms of n=%d by the direct O(n^2) "
                            "definition, %d threads, %.1f s" % (nd, n, threads, el2)}
    acc = None
    if y_gpu is not None:
        err = oracle.rel_l2(y_gpu.reshape(sample, n), ref)
        acc = {"max_rel_l2": float(err.max()), "median_rel_l2": float(np.median(err)),
               "transforms": sample, "tolerance": tol,
               "ok": bool(tol is None or err.max() <= tol),
               "against": "fp64 oracle outputs of the cpu_baseline sample"}
    return acc, {"value": dft_flops(n, done) / el / 1e9, "unit": UNIT,
            "cores": used, "kind": "oracle",
            "sample": "%d transforms (first %d of the workload, repeated) of "
                      "n=%d through the fp64 recursive radix-2 FFT, %.1f s "
                      "wall" % (done, sample, n, el),
            "one_core": {"value": dft_flops(n, done1) / el1 / 1e9, "unit": UNIT,
                         "sample": "%d transforms of n=%d on 1 core, %.1f s"
                                   % (done1, n, el1)},
            "direct": direct}


def run_reference(args, wl):
    world, rank, _ = dist_setup()
    if rank != 0:
        return 0
    import oracle
    n = wl["n"]
    sample = args.ref_sample
    x = inputs.make(wl["kind"], n, wl["batch"], wl["seed"], first=0,
                    count=sample)
    threads = oracle.default_threads()
    used = 1
    for _ in range(args.warmup):
        _, used = oracle.fft_radix2_timed(x, threads=threads)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        _, used = oracle.fft_radix2_timed(x, threads=threads)
    el = time.perf_counter() - t0
    value = dft_flops(n, sample) * args.steps / el / 1e9
    line = {
        "impl": "reference", "metric": metric_for(wl), "value": value, "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": el / args.steps * 1e3, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": workload_config(wl, args),
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": used,
                         "kind": "oracle",
                         "sample": "%d transforms of n=%d per step (first %d "
                                   "of the workload), fp64 recursive radix-2 "
                                   "FFT" % (sample, n, sample)},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


GRID = {
    # 2-D DFT / circular convolution of tiles the size the stencil path
    # uses, and the stencil itself (Sec. 4.6, Lemmas 1-2)
    "dft2": {"n1": 256, "n2": 256, "batch": 4096, "sqrt_m": 16, "seed": 5},
    "conv2": {"n1": 256, "n2": 256, "batch": 4096, "sqrt_m": 16, "seed": 6},
    "stencil": {"side": 4096, "steps": 16, "sqrt_m": 16, "seed": 7},
}
HEAT3 = [[0.0, 0.1, 0.0], [0.15, 0.5, 0.15], [0.0, 0.1, 0.0]]


def grid_cpu_baseline(args, g):
    """The fp64 oracle on a bounded sample of the 2-D workload (one core)."""
    from oracle import grid as ogrid
    t0 = time.perf_counter()
    if args.grid in ("dft2", "conv2"):
        n1, n2 = g["n1"], g["n2"]
        N = n1 * n2
        x = inputs.make("normal", N, 8, g["seed"]).reshape(8, n1, n2)
        done = 0
        while time.perf_counter() - t0 < args.cpu_seconds:
            y = ogrid.dft2(x)
            if args.grid == "conv2":
                ogrid.dft2(y, inverse=True)
            done += 8
        el = time.perf_counter() - t0
        per = 5.0 * N * math.log2(N) * (2 if args.grid == "conv2" else 1)
        return {"value": per * done / el / 1e9, "unit": "GFLOP/s", "cores": 1,
                "kind": "oracle",
                "sample": "%d arrays of %dx%d through the fp64 oracle 2-D DFT "
                          "(rows then columns)%s, %.1f s" % (
                              done, n1, n2, " and its inverse" if args.grid == "conv2"
                              else "", el)}
    k = g["steps"]
    side = 256
    rng = np.random.default_rng(g["seed"])
    A = rng.standard_normal((side, side))
    done = 0
    while time.perf_counter() - t0 < args.cpu_seconds:
        ogrid.stencil_direct(A, np.array(HEAT3), k)
        done += 1
    el = time.perf_counter() - t0
    return {"value": side * side * k * done / el / 1e9, "unit": "Gupdates/s", "cores": 1,
            "kind": "oracle",
            "sample": "%d runs of the fp64 oracle stencil (direct sweeps, free "
                      "plane) on a %dx%d grid for %d steps, %.1f s" % (done, side, side, k, el)}


def run_grid(args):
    """One JSON line for a 2-D workload: 2-D DFT or batched circular 2-D
    convolution of 256 x 256 arrays (GFLOP/s, 5 N log2 N per array and
    transform, N = n1 n2), or the stencil of a 4096^2 grid over 16 steps
    (grid-point updates per second).  Every pass kernel moves 16 B per
    point; the roofline line is the average pass launch of the step."""
    import torch
    from paper_1908_06649_gb300 import _build
    _build.build()
    import paper_1908_06649_gb300 as pkg
    g = GRID[args.grid]
    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    stream = torch.cuda.current_stream()
    if args.grid in ("dft2", "conv2"):
        n1, n2, batch, r = g["n1"], g["n2"], g["batch"], g["sqrt_m"]
        N = n1 * n2
        x_host = inputs.make("normal", N, batch, g["seed"])
        x = torch.from_numpy(x_host).cuda()
        y = torch.empty_like(x)
        plan = pkg.Plan2(n1, n2, batch, r, args.precision)
        if args.grid == "conv2":
            one = pkg.Plan2(n1, n2, 1, r, args.precision)
            w = torch.from_numpy(inputs.make("normal", N, 1, g["seed"] + 1)).cuda()
            spec = one.forward(w)
            one.check()
            step = lambda: plan.conv(x, spec, y)
            passes, flops = 3, 2 * 5.0 * N * math.log2(N) * batch
        else:
            step = lambda: plan.forward(x, y)
            passes, flops = 2, 5.0 * N * math.log2(N) * batch
        launches = passes
        points = N * batch
        unit, metric = "GFLOP/s", ("%s GFLOP/s (5N·log2N per array%s), %dx%d x%d "
                                   "complex64, 1xGB300" % (
                                       "2-D DFT" if args.grid == "dft2" else
                                       "circular 2-D convolution",
                                       "" if args.grid == "dft2" else " x2 transforms",
                                       n1, n2, batch))
        config = {"workload": "batched complex64 %s of %dx%d arrays x batch %d, "
                              "normal inputs seed %d, %s" % (
                                  "2-D DFT" if args.grid == "dft2" else
                                  "circular 2-D convolution with one array",
                                  n1, n2, batch, g["seed"],
                                  "3xTF32" if args.precision == 3 else "TF32"),
                  "n1": n1, "n2": n2, "batch": batch, "sqrt_m": r,
                  "l2": "inputs larger than L2 (%d MiB per buffer), no flush"
                        % (points * 8 >> 20)}
        value_of = lambda ms: flops / (ms * 1e-3) / 1e9
        bytes_min = 16.0 * points
    else:
        side, k, r = g["side"], g["steps"], g["sqrt_m"]
        rng = np.random.default_rng(g["seed"])
        A = torch.from_numpy(rng.standard_normal((side, side)).astype(np.float32)).cuda().reshape(-1)
        out = torch.empty_like(A)
        plan = pkg.StencilPlan(side, k, r, args.precision)
        step = lambda: plan.apply(A, out, w3x3=HEAT3)
        # the plan's tiling: tiles of Nt x Nt, each giving a B x B output block
        tiles, Nt, B = pkg.stencil_tiles(side, k, r)
        points = tiles * Nt * Nt
        passes = 3
        # weights: place, 2-D DFT (2), power, inverse (2); kernel W': place,
        # 2-D DFT (2); tiles: gather, convolution (3), extract
        launches = 14
        unit = "Gupdates/s"
        metric = ("linear stencil grid-point updates/s (side^2 x steps), "
                  "%d^2 grid x %d steps, 1xGB300" % (side, k))
        config = {"workload": "linear 3x3 stencil (heat update) on a %dx%d fp32 "
                              "grid for %d steps via Lemma 1 windows (%d tiles of "
                              "%dx%d, each giving a %dx%d output block) and Lemma 2 "
                              "weights, %s" % (
                                  side, side, k, tiles, Nt, Nt, B, B,
                                  "3xTF32" if args.precision == 3 else "TF32"),
                  "side": side, "steps": k, "sqrt_m": r, "tile": Nt, "block": B,
                  "l2": "grid %d MiB, but every step streams the %d MiB tile "
                        "batch through HBM three times, which evicts it; no "
                        "flush" % (side * side * 4 >> 20, points * 8 >> 20)}
        value_of = lambda ms: side * side * k / (ms * 1e-3) / 1e9
        bytes_min = 8.0 * side * side
    for _ in range(max(3, args.warmup)):
        step()
    plan.check()
    K = args.steps
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    clocks = ClockSampler(torch.cuda.current_device())
    clocks.start()
    time.sleep(0.2)
    torch.cuda.synchronize()
    t0.record(stream)
    for _ in range(K):
        step()
    t1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    plan.check()
    ms = t0.elapsed_time(t1) / K
    cpu = None if args.no_cpu_baseline else grid_cpu_baseline(args, g)
    if args.grid == "stencil":
        # whole step: the three convolution passes (16 B per tile point each),
        # the gather (tile points written, the grid read once) and the
        # extract (one tile point read and one grid point written per cell);
        # the weight and kernel-spectrum transforms are tiny
        S = float(side * side)
        step_bytes = 48.0 * points + 8.0 * points + 4.0 * S + 8.0 * S + 4.0 * S
        achieved = step_bytes / (ms * 1e-3) / 1e9
        kname = ("whole step (%d launches: weights, kernel spectrum, gather, 3 "
                 "convolution passes, extract), %.2f GB algorithmic" % (launches, step_bytes / 1e9))
    else:
        achieved = 16.0 * points / (ms / passes * 1e-3) / 1e9
        kname = "average pass launch (%d pass launches per step)" % passes
    line = {
        "metric": metric, "value": value_of(ms), "unit": unit, "n_gpus": 1,
        "steps": K, "warmup": max(3, args.warmup), "ms_per_step": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
        "dtype": "tf32x3" if args.precision == 3 else "tf32", "data": "synthetic",
        "config": config,
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm, "unit": "GB/s",
                     "frac": achieved / hbm, "traffic": None,
                     "kernel": kname, "peak_source": peak_kind},
        "roofline_step": {"hbm_bytes_min": bytes_min,
                          "t_roof_ms": bytes_min / (hbm * 1e9) * 1e3,
                          "frac": bytes_min / (hbm * 1e9) / (ms * 1e-3)},
        "cpu_baseline": cpu, "e2e": None,
        "gpu_launches": K * launches, "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    plan.destroy()
    return 0


L2_BYTES = 129 << 20           # GB300 L2
L2_FLUSH_BYTES = 512 << 20     # > 2 x L2


def needs_flush(wl):
    """Buffers smaller than twice the L2 would stay cached between steps."""
    return wl["n"] * wl["batch"] * 8 < 2 * L2_BYTES


def workload_config(wl, args):
    return {"workload": "batched complex64 forward DFT n=%d (=%d^%d) x batch "
                        "%d, %s inputs seed %d, %s" % (
                            wl["n"], wl["sqrt_m"],
                            round(math.log(wl["n"], wl["sqrt_m"])),
                            wl["batch"], wl["kind"], wl["seed"],
                            "3xTF32" if args.precision == 3 else "TF32"),
            "n": wl["n"], "batch": wl["batch"], "sqrt_m": wl["sqrt_m"],
            "precision": "3xTF32" if args.precision == 3 else "TF32",
            "l2": (("inputs larger than L2 (%d MiB per buffer), no flush"
                   % (wl["n"] * wl["batch"] * 8 >> 20))
                   if not needs_flush(wl) else
                   ("L2 flushed before every step (%d MiB write, untimed); "
                    "%d MiB per buffer" % (L2_FLUSH_BYTES >> 20,
                                           wl["n"] * wl["batch"] * 8 >> 20))),
            "parallelism": "replica/batch shard x%d" % args.gpus}


def time_exec(torch, plan, x, y, steps, direction, stream, flush, l2buf):
    """CUDA-event timing of `steps` executions of `plan` on `stream` (inputs
    resident in HBM): per pass launch and per step.  With `flush`, an
    untimed write of a buffer larger than L2 precedes every step and the
    step time is the sum of the steps' own events."""
    npass = len(plan.passes())
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(npass + 1)]
          for _ in range(steps)]
    for row in ev:
        for e in row:
            e.record(stream)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize()
    t0.record(stream)
    for i in range(steps):
        if flush:
            l2buf.fill_(float(i))
        plan.exec_timed(x, y, ev[i], direction)
    t1.record(stream)
    torch.cuda.synchronize()
    if flush:
        total = sum(ev[i][0].elapsed_time(ev[i][npass]) for i in range(steps))
    else:
        total = t0.elapsed_time(t1)
    passes = [sum(ev[i][p].elapsed_time(ev[i][p + 1]) for i in range(steps)) / steps
              for p in range(npass)]
    return total / steps, passes


def sample_rows(batch, count=8):
    """Transforms whose outputs the CPU-baseline leg checks: the first, the
    last and evenly spaced ones in between."""
    if batch <= count:
        return list(range(batch))
    return sorted(set(int(round(i * (batch - 1) / (count - 1))) for i in range(count)))


def oracle_accuracy(x_rows, y_rows, tol, inverse=False):
    """CPU-baseline leg: per-transform relative L2 of GPU outputs against the
    fp64 oracle's outputs for the same inputs."""
    import oracle
    n = x_rows.shape[1]
    sign, scale = (1, 1.0 / n) if inverse else (-1, 1.0)
    ref = oracle.fft_radix2(x_rows, sign, scale, threads=oracle.default_threads())
    err = oracle.rel_l2(y_rows, ref)
    return {"max_rel_l2": float(err.max()), "median_rel_l2": float(np.median(err)),
            "transforms": int(x_rows.shape[0]), "tolerance": tol,
            "ok": bool(err.max() <= tol), "against": "fp64 oracle (radix-2 FFT)"}


def per_workload(args, torch, pkg, dev, stream, hbm, p_tf32, skip):
    """Every other workload the method is evaluated on (the configs besides
    the headline's), each timed like the headline (warm-up, CUDA events on
    the exec stream, L2 flushed where the buffers would stay cached), with
    its step roofline, its dominant pass launch against the HBM peak and,
    in the CPU-baseline leg, its accuracy against the oracle on sampled
    transforms.  The two radix-sweep workloads add the inverse and the
    round trip."""
    out = {}
    steps = max(5, min(args.steps, 30))
    tol = 1e-5 if args.precision == 3 else 3e-3
    for name in sorted(inputs.WORKLOADS):
        if name == skip:
            continue
        wl = inputs.WORKLOADS[name]
        n, batch, r = wl["n"], wl["batch"], wl["sqrt_m"]
        t_gen = time.perf_counter()
        x_host = inputs.make(wl["kind"], n, batch, wl["seed"])
        t_gen = time.perf_counter() - t_gen
        x = torch.from_numpy(x_host).to(dev)
        y = torch.empty_like(x)
        plan = pkg.Plan(n, batch, r, args.precision)
        stages = plan.passes()
        flush = needs_flush(wl)
        l2buf = (torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
                 if flush else None)
        entry = {"n": n, "batch": batch, "sqrt_m": r, "kind": wl["kind"], "seed": wl["seed"],
                 "passes": stages, "steps": steps,
                 "l2": "flushed before every step" if flush else "inputs larger than L2"}
        dirs = [("forward", pkg.FORWARD)]
        if "inverse" in wl["dirs"]:
            dirs.append(("inverse", pkg.INVERSE))
        bytes_min = 16.0 * n * batch
        k = sum(stages)
        tensor_flops = 8.0 * r * n * batch * k * args.precision
        t_roof = max(bytes_min / (hbm * 1e9), tensor_flops / (p_tf32 * 1e12))
        ys = {}
        for dname, d in dirs:
            src = x if dname == "forward" else ys["forward"]
            dst = torch.empty_like(x)
            for _ in range(max(3, args.warmup)):
                plan.exec(src, dst, d)
            plan.check()
            ms, pms = time_exec(torch, plan, src, dst, steps, d, stream, flush, l2buf)
            plan.check()
            dom = max(range(len(pms)), key=lambda i: pms[i])
            ys[dname] = dst
            entry[dname] = {
                "ms_per_step": ms, "value": dft_flops(n, batch) / (ms * 1e-3) / 1e9,
                "unit": UNIT,
                "roofline_step": {"t_roof_ms": t_roof * 1e3, "frac": t_roof / (ms * 1e-3)},
                "dominant_launch": {"pass": dom + 1, "stages": stages[dom], "ms": pms[dom],
                                    "achieved_gbs": bytes_min / (pms[dom] * 1e-3) / 1e9,
                                    "peak_gbs": hbm,
                                    "frac": bytes_min / (pms[dom] * 1e-3) / 1e9 / hbm},
                "launch_ms": pms}
        rows = sample_rows(batch, 64 if n <= 4096 else 8)
        if "inverse" in ys:
            # round trip IDFT(DFT(x)) against x on every transform (no oracle)
            num = torch.linalg.vector_norm((ys["inverse"] - x).reshape(batch, n), dim=1)
            den = torch.linalg.vector_norm(x.reshape(batch, n), dim=1)
            entry["round_trip_max_rel_l2"] = float((num / den).max())
        if not args.no_cpu_baseline:
            acc = {}
            for dname in ys:
                src_rows = (x_host[rows] if dname == "forward"
                            else ys["forward"].reshape(batch, n)[rows].cpu().numpy())
                got = ys[dname].reshape(batch, n)[rows].cpu().numpy()
                acc[dname] = oracle_accuracy(src_rows, got, tol, inverse=dname == "inverse")
            entry["accuracy"] = acc
        entry["input_generation_s"] = t_gen
        out[name] = entry
        plan.destroy()
        del x, y, ys, l2buf
        torch.cuda.empty_cache()
        log("per-workload %s: %.4f ms forward" % (name, entry["forward"]["ms_per_step"]))
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=10)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="n65536_b1024",
                    choices=sorted(inputs.WORKLOADS))
    ap.add_argument("--precision", type=int, default=3, choices=[1, 3])
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--ref-sample", type=int, default=16)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=20)
    ap.add_argument("--fuse", action="store_true",
                    help="one fused launch with an L2-resident intermediate "
                         "instead of two pass launches")
    ap.add_argument("--one-pass", action="store_true",
                    help="both passes in one launch on cluster pairs (n = 16^4)")
    ap.add_argument("--batch", type=int, default=0,
                    help="override the workload's batch (profiling cases)")
    ap.add_argument("--no-per-workload", action="store_true",
                    help="skip the other workloads' extra fields")
    ap.add_argument("--grid", default=None, choices=sorted(GRID),
                    help="measure a 2-D workload (2-D DFT, circular 2-D "
                         "convolution or the stencil) instead of the 1-D one")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    wl = dict(inputs.WORKLOADS[args.workload])
    if args.batch > 0:
        wl["batch"] = args.batch
    if args.impl == "reference":
        return run_reference(args, wl)
    if args.grid:
        return run_grid(args)

    import torch
    world, rank, local = dist_setup()
    if world > 1:
        import torch.distributed as dist
        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    else:
        dist = None
    dev = torch.device("cuda", torch.cuda.current_device())

    from paper_1908_06649_gb300 import _build
    if rank == 0 or world == 1:
        _build.build()
    if dist is not None:
        dist.barrier()
    import paper_1908_06649_gb300 as pkg

    n, batch, r = wl["n"], wl["batch"], wl["sqrt_m"]
    log("rank %d: generating %s inputs n=%d batch=%d" % (rank, wl["kind"], n,
                                                       batch))
    x_host = inputs.make(wl["kind"], n, batch, rank_seed(wl, rank))
    x = torch.from_numpy(x_host).to(dev)
    y = torch.empty_like(x)
    plan = pkg.Plan(n, batch, r, args.precision,
                    pkg.PLAN_FUSE if args.fuse else
                    (pkg.PLAN_ONE_PASS if args.one_pass else pkg.PLAN_DEFAULT))
    npass = len(plan.passes())
    stream = torch.cuda.current_stream()

    for _ in range(args.warmup):
        plan.forward(x, y)
    plan.check()

    K = args.steps
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(npass + 1)]
          for _ in range(K)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    # torch creates the CUDA event lazily on its first record
    for row in ev:
        for e in row:
            e.record(stream)
    torch.cuda.synchronize()
    clocks = ClockSampler(torch.cuda.current_device()) if rank == 0 else None
    if clocks:
        clocks.start()
        time.sleep(0.2)
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    flush = needs_flush(wl)
    l2buf = (torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
             if flush else None)
    t_start.record(stream)
    for i in range(K):
        if flush:
            l2buf.fill_(float(i))  # untimed: outside ev[i][0] .. ev[i][npass]
        plan.exec_timed(x, y, ev[i])
    t_end.record(stream)
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    clk = clocks.stop() if clocks else None
    plan.check()
    if flush:
        # the step is its own events, first pass to last, without the flush
        elapsed_ms = sum(ev[i][0].elapsed_time(ev[i][npass]) for i in range(K))
    else:
        elapsed_ms = t_start.elapsed_time(t_end)
    pass_ms = [[ev[i][p].elapsed_time(ev[i][p + 1]) for i in range(K)]
               for p in range(npass)]
    elapsed_ms = max_over_ranks(elapsed_ms, dist, dev)

    ms_per_step = elapsed_ms / K
    value = job_rate(dft_flops(n, batch), world, K, elapsed_ms)

    peaks, peak_kind = load_peaks()
    hbm = float(peaks["hbm_gbs"])
    # per-launch algorithmic bytes: every complex64 point read once and
    # written once by each pass kernel
    bytes_launch = 16.0 * n * batch
    avg = [sum(p) / len(p) for p in pass_ms]
    stages = plan.passes()
    if plan.fused:
        # one launch runs both passes; events[1] == events[2]
        avg = [avg[0] + avg[1]]
        kname = "dft_fused_kernel (%d passes, %s stages)" % (
            npass, "+".join(map(str, stages)))
        launches = 1
    else:
        launches = npass
    dom = max(range(len(avg)), key=lambda i: avg[i])
    if not plan.fused:
        kname = "pass kernel %d of %d (%d stages)" % (dom + 1, npass, stages[dom])
    achieved = bytes_launch / (avg[dom] * 1e-3) / 1e9
    e2e = None
    if args.e2e_steps > 0:
        h_in = torch.from_numpy(x_host).pin_memory()
        h_out = torch.empty_like(h_in).pin_memory()
        work = torch.empty_like(x)
        plan.exec_host(h_in, h_out, work)
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        e0.record(stream)
        for _ in range(args.e2e_steps):
            plan.exec_host(h_in, h_out, work)
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = e0.elapsed_time(e1)
        e2e_ms = max_over_ranks(e2e_ms, dist, dev)
        floor_ms = copy_floor_ms(h_in, h_out, work, x, stream)
        e2e = {"value": job_rate(dft_flops(n, batch), world, args.e2e_steps,
                                 e2e_ms),
               "unit": UNIT, "h2d_bytes_per_step": n * batch * 8,
               "d2h_bytes_per_step": n * batch * 8,
               "steps": args.e2e_steps,
               "ms_per_step": e2e_ms / args.e2e_steps,
               # this machine's host<->device link, measured on the same pinned
               # buffers: a step's bytes both ways at once, without the DFT
               "copy_floor_ms_per_step": floor_ms,
               "frac_of_copy_floor": floor_ms / (e2e_ms / args.e2e_steps)}

    # whole-step roofline: min HBM bytes vs tensor flops at the TF32 peak,
    # measured here (cuBLAS TF32 GEMM, after every timed region) or, if that
    # fails, the measured bf16 peak times the nominal TF32/BF16 ratio
    p_tf32 = measure_tf32_tflops(dev) if rank == 0 else None
    if p_tf32:
        tf32_source = "measured in this run: cuBLAS TF32 GEMM 8192^3, best of 10"
    else:
        p_tf32 = float(peaks["bf16_tflops"]) * NOMINAL_TF32 / NOMINAL_BF16
        tf32_source = "%s bf16 x %.2f/%.2f nominal" % (peak_kind, NOMINAL_TF32,
                                                       NOMINAL_BF16)
    k = sum(stages)
    tensor_flops = 8.0 * r * n * batch * k * args.precision
    t_roof = max(bytes_launch / (hbm * 1e9), tensor_flops / (p_tf32 * 1e12))
    frac_step = t_roof / (ms_per_step * 1e-3)

    plan_fused = plan.fused
    # GPU outputs of the first transforms, for the accuracy check of the
    # CPU-baseline leg
    sample = min(32, batch)
    y_head = y.reshape(-1)[:sample * n].cpu().numpy()
    plan.destroy()
    cpu = acc = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        acc, cpu = cpu_baseline(wl, seconds=args.cpu_seconds, sample=sample,
                                y_gpu=y_head,
                                tol=1e-5 if args.precision == 3 else 3e-3)

    others = None
    if (rank == 0 and world == 1 and not args.no_per_workload and args.batch == 0
            and args.workload == "n65536_b1024"):
        others = per_workload(args, torch, pkg, dev, stream, hbm, p_tf32, args.workload)

    if rank == 0:
        line = {
            "metric": metric_for(wl), "value": value, "unit": UNIT, "n_gpus": world,
            "steps": K, "warmup": args.warmup, "ms_per_step": ms_per_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "tf32x3" if args.precision == 3 else "tf32",
            "data": "synthetic", "config": workload_config(wl, args),
            "roofline": {"bound": "hbm", "achieved": achieved, "peak": hbm,
                         "unit": "GB/s", "frac": achieved / hbm,
                         "traffic": profiled_traffic(batch, plan_fused)
                         if (n == 65536 and r == 16) else None,
                         "kernel": kname,
                         "peak_source": peak_kind,
                         "launch_ms": avg},
            "roofline_step": {"t_roof_ms": t_roof * 1e3, "frac": frac_step,
                              "hbm_bytes_min": bytes_launch,
                              "tensor_flops": tensor_flops,
                              "tf32_peak_tflops": p_tf32,
                              "tf32_peak_source": tf32_source},
            "cpu_baseline": cpu, "e2e": e2e,
            "accuracy": acc,
            "gpu": torch.cuda.get_device_name(dev),
            "gpu_launches": K * launches,
            "clocks": clk,
            "per_workload": others,
        }
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
