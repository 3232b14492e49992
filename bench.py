#!/usr/bin/env python3
"""Benchmark of the SFC bf16 GEMM on GB300.

One step = one pass of the whole hot path over the square sweep
M = N = K in {2048, 4096, 8192, 16384} (bf16 inputs uniform in [-1, 1] from
seed 0, fp32 accumulation, bf16 output, ca_c = 1, tiles ordered along the
generalized Hilbert curve).  ``value`` is the weighted harmonic mean over the
sweep, sum(2 M N K) / sum(time), in TFLOP/s, with inputs resident in HBM.

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle (the
plain fp64 triple loop) on sampled rows of the same workload instead.
"""
from __future__ import annotations

import argparse
import csv
import hashlib
import io
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "bf16 GEMM TFLOP/s & % of GB300 dense peak; weighted harmonic mean over shapes"
WORKLOAD = ("square bf16 GEMM sweep M=N=K in {2048, 4096, 8192, 16384}, uniform [-1,1] seeded inputs, "
            "fp32 accumulate, bf16 output, ca_c=1")
SIZES = (2048, 4096, 8192, 16384)
FALLBACK_PEAKS = {"bf16_tflops": 1900.0, "hbm_gbs": 6800.0}
KERNEL_SOURCES = ("paper_2601_16294_gb300/csrc/sfc_gemm_kernel.cuh", "paper_2601_16294_gb300/csrc/ptx.cuh",
                  "paper_2601_16294_gb300/csrc/sfc_curve.cuh", "paper_2601_16294_gb300/csrc/sfc_gemm.cu")
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "traffic_square_sweep.json")


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--order", choices=("sfc", "raster"), default="sfc")
    ap.add_argument("--assign", choices=("auto", "wave", "segment"), default="auto")
    ap.add_argument("--sizes", type=str, default=",".join(map(str, SIZES)),
                    help="comma-separated square sizes (default: the full sweep)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    return ap.parse_args()


def kernel_sha() -> str:
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            d = json.load(f)
        return {"bf16_tflops": float(d["bf16_tflops"]), "hbm_gbs": float(d["hbm_gbs"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except Exception:
        return dict(FALLBACK_PEAKS, bf16_tflops_sustained=1700.0, source="fallback")


# ------------------------------------------------------------------ distributed

def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if n_gpus > 0 else "gloo")
    return rank, local, world


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x, world):
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------- clocks

class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int, enabled: bool = True):
        self.proc = None
        self.index = device_index
        if not enabled:
            return
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(device_index), "--query-gpu=" + self.FIELDS,
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        rows = list(csv.reader(io.StringIO(out)))
        sm, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except ValueError:
                continue
            for name, val in zip(names, r[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ------------------------------------------------------------------- our arm

def run_ours(args, rank, local, world):
    import torch
    import paper_2601_16294_gb300 as sfc
    from paper_2601_16294_gb300 import binding, synth

    torch.cuda.set_device(local)
    sfc.load()
    stream = torch.cuda.current_stream()
    sizes = [int(s) for s in args.sizes.split(",")]
    peaks = load_peaks()

    # inputs resident in HBM before timing (seeded on the CPU, copied once)
    mats = []
    for n in sizes:
        A, B = synth.gemm_inputs(n, n, n, "uniform", seed=0)
        mats.append((n, A.cuda(), B.cuda(), torch.empty((n, n), dtype=torch.bfloat16, device="cuda"), A, B))
    torch.cuda.synchronize()

    kw = dict(ca_c=1, order=args.order, assign=args.assign, stream=stream)

    def step(events=None):
        for i, (n, A, B, C, _, _) in enumerate(mats):
            if events is not None:
                events[i][0].record(stream)
            sfc.gemm(A, B, C, **kw)
            if events is not None:
                events[i][1].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if sfc.device_status() != 0:
        raise RuntimeError("device-side timeout during warm-up")

    per_launch = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in mats] for _ in range(args.steps)]
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local, enabled=not args.no_clocks)
    time.sleep(0.2 if clocks.proc else 0)
    barrier(world)
    torch.cuda.synchronize()
    t0.record(stream)
    for k in range(args.steps):
        step(per_launch[k])
    t1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clock_info = clocks.stop()
    status = sfc.device_status()
    if status != 0:
        raise RuntimeError("device-side timeout in the timed region (status %d)" % status)

    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world)
    flops_step = sum(2.0 * n ** 3 for n, *_ in mats)
    value = world * flops_step * args.steps / (elapsed_ms * 1e-3) / 1e12
    ms_per_step = elapsed_ms / args.steps

    # per-shape kernel times (same launches, events on the launching stream)
    per_shape = []
    tot_kernel_ms = 0.0
    for i, (n, *_rest) in enumerate(mats):
        ts = [per_launch[k][i][0].elapsed_time(per_launch[k][i][1]) for k in range(args.steps)]
        mean = sum(ts) / len(ts)
        tot_kernel_ms += sum(ts)
        tf = 2.0 * n ** 3 / (mean * 1e-3) / 1e12
        per_shape.append({"M": n, "N": n, "K": n, "ms_mean": round(mean, 4), "ms_min": round(min(ts), 4),
                          "tflops": round(tf, 1), "frac_of_peak": round(tf / peaks["bf16_tflops"], 4)})

    # roofline of the dominant kernel (the GEMM kernel: every launch in the step)
    launches = args.steps * len(mats)
    achieved = flops_step * args.steps / (tot_kernel_ms * 1e-3) / 1e12
    traffic = None
    try:
        with open(TRAFFIC_FILE) as f:
            tr = json.load(f)
        if tr.get("kernel_sha") == kernel_sha() and tr.get("sizes") == sizes:
            traffic = tr["dram_bytes_per_launch"]
    except Exception:
        traffic = None
    roofline = {"bound": "tensor", "achieved": round(achieved, 1), "peak": peaks["bf16_tflops"],
                "unit": "TFLOP/s", "frac": round(achieved / peaks["bf16_tflops"], 4), "traffic": traffic,
                "kernel": "sfc_gemm_kernel<256,4,bf16>", "peak_source": peaks["source"] + " bf16 burst",
                "frac_of_sustained": round(achieved / peaks["bf16_tflops_sustained"], 4)}

    result = {
        "metric": METRIC, "value": round(value, 1), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded uniform [-1,1] bf16)",
        "config": {"workload": WORKLOAD, "sizes": sizes, "order": args.order, "assign": args.assign,
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "l2": "inputs larger than L2 between reuses: each shape's operands are re-read only "
                         "after the other shapes' GEMMs (>1.5 GB of traffic) have passed through L2",
                   "pct_of_dense_peak": round(100.0 * value / world / peaks["bf16_tflops"], 2)},
        "roofline": roofline,
        "gpu_launches": launches,
        "per_shape": per_shape,
    }
    if clock_info is not None:
        result["clocks"] = clock_info

    if not args.no_e2e:
        result["e2e"] = run_e2e(args, mats, stream, world)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = run_cpu_baseline(args, mats)
    return result


def run_e2e(args, mats, stream, world):
    """Same metric through the public API from pinned HOST buffers: every step
    copies A and B host->device, runs the GEMM, copies C device->host."""
    import torch
    import paper_2601_16294_gb300 as sfc

    host = []
    for n, A, B, C, Acpu, Bcpu in mats:
        host.append((n, Acpu.pin_memory(), Bcpu.pin_memory(),
                     torch.empty((n, n), dtype=torch.bfloat16, pin_memory=True)))
    h2d = sum(2 * 2 * n * n for n, *_ in host)
    d2h = sum(2 * n * n for n, *_ in host)

    def step():
        for n, Ah, Bh, Ch in host:
            sfc.matmul_host(Ah, Bh, Ch, out_dtype=torch.bfloat16, stream=stream)

    for _ in range(max(1, min(args.warmup, 2))):
        step()
    steps = max(1, min(args.steps, 5))
    barrier(world)
    torch.cuda.synchronize()
    t = time.perf_counter()
    for _ in range(steps):
        step()
    torch.cuda.synchronize()
    el = max_over_ranks(time.perf_counter() - t, world)
    flops = sum(2.0 * n ** 3 for n, *_ in host) * steps * world
    return {"value": round(flops / el / 1e12, 1), "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps,
            "api": "paper_2601_16294_gb300.matmul_host -> sfc_gemm_ex (C ABI)"}


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count() or 1


def oracle_sample(mats_cpu, rows):
    """Time the oracle's plain GEMM on `rows` evenly spaced rows of A for each
    shape (those rows of C); returns (flops, seconds)."""
    import numpy as np
    from oracle import oracle
    oracle.build()
    flops = 0.0
    t = 0.0
    for n, A, B in mats_cpu:
        r = np.linspace(0, n - 1, rows).astype(np.int64)
        A_rows = A[r].contiguous()
        t0 = time.perf_counter()
        oracle.gemm_f64(A_rows, B)
        t += time.perf_counter() - t0
        flops += 2.0 * rows * n * n
    return flops, t


def run_cpu_baseline(args, mats):
    """The oracle as it stands, on this host's cores, on a bounded sample of the
    workload: a 16-row probe sets the row count for about 12 s of CPU work."""
    os.environ.setdefault("OMP_NUM_THREADS", str(cpu_cores()))
    mats_cpu = [(n, Acpu, Bcpu) for n, _, _, _, Acpu, Bcpu in mats]
    f_probe, s_probe = oracle_sample(mats_cpu, 16)
    rows = int(min(1024, max(16, 16 * 12.0 / max(s_probe, 1e-3))))
    rows = max(16, rows // 16 * 16)
    flops, secs = oracle_sample(mats_cpu, rows)
    return {"value": round(flops / secs / 1e12, 6), "unit": "TFLOP/s",
            "cores": int(os.environ["OMP_NUM_THREADS"]), "kind": "oracle", "seconds": round(secs, 2),
            "sample": "%d evenly spaced rows of C for each square shape (fp64 i-k-j triple loop, "
                      "OpenMP over rows)" % rows}


# ------------------------------------------------------------- reference arm

def run_reference(args, rank, world):
    """The CPU oracle as the reference arm: each step computes sampled rows of
    every shape of the sweep (bounded so the run ends within minutes)."""
    if rank != 0:
        return None
    from paper_2601_16294_gb300 import synth
    os.environ.setdefault("OMP_NUM_THREADS", str(cpu_cores()))
    sizes = [int(s) for s in args.sizes.split(",")]
    mats_cpu = []
    for n in sizes:
        A, B = synth.gemm_inputs(n, n, n, "uniform", seed=0)
        mats_cpu.append((n, A, B))
    rows = 16
    for _ in range(args.warmup):
        oracle_sample(mats_cpu, 4)
    flops = secs = 0.0
    for _ in range(args.steps):
        f, s = oracle_sample(mats_cpu, rows)
        flops += f
        secs += s
    value = flops / secs / 1e12
    cores = int(os.environ["OMP_NUM_THREADS"])
    sample = "%d evenly spaced rows of C per square shape per step" % rows
    return {"impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * secs / args.steps, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded uniform [-1,1] bf16)",
            "config": {"workload": WORKLOAD, "sizes": sizes, "sample": sample},
            "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def main():
    args = parse_args()
    if args.impl == "reference":
        rank = int(os.environ.get("RANK", "0"))
        world = int(os.environ.get("WORLD_SIZE", "1"))
        out = run_reference(args, rank, world)
        if out is not None:
            print(json.dumps(out), flush=True)
        return
    rank, local, world = dist_setup(args.gpus)
    out = run_ours(args, rank, local, world)
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
