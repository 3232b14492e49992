#!/usr/bin/env python3
"""Benchmark of the SFC bf16 GEMM on GB300.

Default workload ("configs"): one step = one pass of the whole hot path over
the 29 shapes of the four measured configurations --
  * square: M = N = K in {2048, 4096, 8192, 16384}, uniform [-1, 1], bf16 out, ca_c = 1;
  * prefill: M in {512, 2048, 8192} x (N, K) in {(4096, 4096), (14336, 4096),
    (4096, 14336), (128256, 4096)}, activations N(0, 1), weights N(0, 0.02), bf16 out;
  * irregular: 3000x5000x7000, 1000x17000x2500, 6144x768x12288, 129x8191x4096,
    uniform, bf16 out;
  * high-K: M = N in {512, 1024, 2048} x K in {32768, 65536, 131072}, uniform, fp32 out
-- each with bf16 inputs from seed 0, fp32 accumulation and tiles ordered along
the generalized Hilbert curve.  For prefill, irregular and high-K every K-layer
count in {1, 2, 4, 8} is timed and the best is used in the step (the paper
reports the best replication factor, Sec. IV-A); the library's own choice
(ca_c = 0) is timed and reported beside it.  ``value`` is the weighted
harmonic mean over the step's shapes, sum(2 M N K) / time, in TFLOP/s, with
inputs resident in HBM.

Other workloads (``--workload``) measure one shape set alone: ``square``,
``prefill``, ``irregular``, ``highk``, ``sweep125`` (the paper's 125-shape
sweep over {512..8192}^3), ``cube512`` (the small parity case).

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
FALLBACK_PEAKS = {"bf16_tflops": 1900.0, "hbm_gbs": 6800.0, "bf16_tflops_sustained": 1700.0}
KERNEL_SOURCES = ("paper_2601_16294_gb300/csrc/sfc_gemm_kernel.cuh", "paper_2601_16294_gb300/csrc/ptx.cuh",
                  "paper_2601_16294_gb300/csrc/sfc_curve.cuh", "paper_2601_16294_gb300/csrc/sfc_gemm.cu",
                  "paper_2601_16294_gb300/csrc/sfc_gemm_pair_kernel.cuh")
# per-shape DRAM bytes of each tile's GEMM launch on a workload's shapes (one ncu capture of
# --traffic-capture), keyed by the kernel sources' hash
TRAFFIC_FILES = {"configs": os.path.join(ROOT, "profiles", "traffic_configs.json"),
                 "square": os.path.join(ROOT, "profiles", "traffic_square_sweep.json")}
# the kernel name a tile label launches (the record says which kernel each capture measured)
TILE_KERNEL = {"pair256": "sfc_gemm_pair_kernel<256", "pair128": "sfc_gemm_pair_kernel<128",
               "256": "sfc_gemm_kernel<256", "128": "sfc_gemm_kernel<128"}
CS = (1, 2, 4, 8)
HOLD_HZ = 2.07e9  # GB300's maximum SM clock: cycles per second of the hold kernel's spin


def _shape(M, N, K, kind="uniform", out="bf16", cs=(1,), shared=False):
    # shared: A (M x K) and B (K x N) are drawn per operand shape, from seeds of
    # their own, and reused by every shape of the workload that has them
    return {"M": M, "N": N, "K": K, "kind": kind, "out": out, "cs": tuple(cs), "shared": shared}


WORKLOADS = {
    "configs": {
        "desc": "configs 2-5 together (29 shapes): square M=N=K in {2048,4096,8192,16384} (ca_c=1, bf16 out); "
                "LLM prefill M in {512,2048,8192} x (N,K) in {(4096,4096),(14336,4096),(4096,14336),(128256,4096)} "
                "(activations N(0,1), weights N(0,0.02) stored KxN, bf16 out); irregular 3000x5000x7000, "
                "1000x17000x2500, 6144x768x12288, 129x8191x4096 (bf16 out); high-K M=N in {512,1024,2048} x K in "
                "{32768,65536,131072} (fp32 out); uniform [-1,1] bf16 inputs unless stated, fp32 accumulate; "
                "best ca_c in {1,2,4,8} per shape except square",
        "shapes": None,  # filled in below from the four sets
    },
    "square": {
        "desc": "square bf16 GEMM sweep M=N=K in {2048, 4096, 8192, 16384}, uniform [-1,1] seeded inputs, "
                "fp32 accumulate, bf16 output, ca_c=1",
        "shapes": [_shape(n, n, n) for n in (2048, 4096, 8192, 16384)],
    },
    "prefill": {
        "desc": "LLM-prefill-shaped bf16 GEMMs: M in {512, 2048, 8192} x (N,K) in {(4096,4096), (14336,4096), "
                "(4096,14336), (128256,4096)}, activations N(0,1), weights N(0,0.02) stored KxN, bf16 output, "
                "best ca_c in {1,2,4,8}",
        "shapes": [_shape(m, n, k, "prefill", "bf16", CS) for m in (512, 2048, 8192)
                   for (n, k) in ((4096, 4096), (14336, 4096), (4096, 14336), (128256, 4096))],
    },
    "irregular": {
        "desc": "irregular shapes 3000x5000x7000, 1000x17000x2500, 6144x768x12288, 129x8191x4096, uniform [-1,1], "
                "bf16 output, rows padded to 16 bytes, best ca_c in {1,2,4,8}",
        "shapes": [_shape(3000, 5000, 7000, cs=CS), _shape(1000, 17000, 2500, cs=CS),
                   _shape(6144, 768, 12288, cs=CS), _shape(129, 8191, 4096, cs=CS)],
    },
    "highk": {
        "desc": "communication-avoiding high-K cases M=N in {512, 1024, 2048} x K in {32768, 65536, 131072}, "
                "uniform [-1,1], fp32 output, ca_c in {1,2,4,8} each timed, best in the step",
        "shapes": [_shape(m, m, k, "uniform", "f32", CS) for m in (512, 1024, 2048)
                   for k in (32768, 65536, 131072)],
    },
    "sweep125": {
        "desc": "the paper's shape sweep: M, N, K each in {512, 1024, 2048, 4096, 8192} (125 shapes), uniform "
                "[-1,1] seeded inputs, bf16 output, best ca_c in {1,2,4,8}",
        "shapes": [_shape(m, n, k, "uniform", "bf16", CS, shared=True) for m in (512, 1024, 2048, 4096, 8192)
                   for n in (512, 1024, 2048, 4096, 8192) for k in (512, 1024, 2048, 4096, 8192)],
    },
    "cube512": {
        "desc": "single GEMM M=N=K=512, uniform [-1,1] seed 0, fp32 output, 4x4 grid of 128x128 tiles, ca_c=1",
        "shapes": [_shape(512, 512, 512, "uniform", "f32")],
    },
}


WORKLOADS["configs"]["shapes"] = (WORKLOADS["square"]["shapes"] + WORKLOADS["prefill"]["shapes"] +
                                  WORKLOADS["irregular"]["shapes"] + WORKLOADS["highk"]["shapes"])


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="configs")
    ap.add_argument("--order", choices=("sfc", "raster"), default="sfc")
    ap.add_argument("--assign", choices=("auto", "wave", "wave_static", "segment"), default="auto")
    ap.add_argument("--sizes", type=str, default=None,
                    help="square workload only: comma-separated sizes instead of the full sweep")
    ap.add_argument("--shapes", type=str, default=None,
                    help="comma-separated MxNxK shapes instead of the workload's (uniform [-1,1] inputs, output "
                         "per --out, bf16 by default; K-layer counts per --ca-c, else 1,2,4,8)")
    ap.add_argument("--ca-c", type=int, default=None, help="force one K-layer count for every shape")
    ap.add_argument("--b-layout", choices=("kn", "nk"), default="kn",
                    help="storage of B: K x N row-major (the paper's), or N x K (a linear layer's weight)")
    ap.add_argument("--ab", choices=("bf16", "e4m3", "e5m2"), default="bf16",
                    help="element type of A and B (8-bit floats use the tensor cores' 8-bit path)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--out", choices=("workload", "f32", "bf16"), default="workload",
                    help="output type of every shape (default: the workload's own)")
    ap.add_argument("--no-tune", action="store_true",
                    help="skip measuring each shape's configurations (sfc_gemm_tune) before timing; the tile then "
                         "comes from the library's time model")
    ap.add_argument("--sustained", action="store_true",
                    help="instead of the step timing: run each configuration back to back for --phase-seconds under "
                         "the power cap (ours by order / dealing / tile / K blocks, then cuBLAS) at each --sizes "
                         "(default 16384,8192), sampling SM clock and power, and print one JSON line of phases")
    ap.add_argument("--phase-seconds", type=float, default=2.5)
    ap.add_argument("--k-block-factor", type=int, default=1,
                    help="passes over each layer's K range (Listing 1's k_block_factor); 1 = one pass")
    ap.add_argument("--e2e-order", choices=("given", "largest_first"), default="largest_first",
                    help="order in which the end-to-end step issues its host-buffer calls (largest first: the "
                         "smaller calls' copies then overlap the largest call's GEMMs)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--traffic-capture", action="store_true",
                    help="the timed step runs every shape once with each tile at one K layer, for a profiler's "
                         "per-tile DRAM record (prints the launch list instead of a bench line)")
    ap.add_argument("--no-cublas", action="store_true",
                    help="skip the comparison with torch.matmul (cuBLAS) in the same power window")
    return ap.parse_args()


def workload_shapes(args):
    if getattr(args, "shapes", None):
        out = args.out if args.out != "workload" else "bf16"
        shapes = []
        for item in args.shapes.split(","):
            M, N, K = (int(x) for x in item.lower().split("x"))
            shapes.append(_shape(M, N, K, "uniform", out, CS if args.ca_c is None else (args.ca_c,)))
        return shapes
    shapes = [dict(s) for s in WORKLOADS[args.workload]["shapes"]]
    if args.sizes:
        # square shapes of the given sizes (with the default workload, or the square one)
        if args.workload not in ("square", "configs"):
            raise SystemExit("--sizes applies to the square workload only")
        shapes = [_shape(int(n), int(n), int(n)) for n in args.sizes.split(",")]
    if args.ca_c is not None:
        for s in shapes:
            s["cs"] = (args.ca_c,)
    if args.out != "workload":
        for s in shapes:
            s["out"] = args.out
    return shapes


def describe(args) -> str:
    if getattr(args, "shapes", None):
        return "shapes %s, uniform [-1,1] bf16 inputs" % args.shapes
    if args.sizes:
        return "square sweep sizes %s" % args.sizes
    return WORKLOADS[args.workload]["desc"]


def kernel_sha() -> str:
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def traffic_per_launch(record, rows, workload, sha):
    """Mean DRAM bytes per launch over the one-layer calls in `rows` (bench per-shape rows with
    M, N, K, ca_c and tile), each matched to the record's capture of the same shape and kernel;
    None when the record belongs to other kernel sources or another workload, or lacks a call."""
    if record.get("kernel_sha") != sha or record.get("workload") != workload:
        return None
    got = []
    for row in rows:
        if row["ca_c"] != 1:
            continue
        want = TILE_KERNEL.get(str(row["tile"]))
        hit = [e for e in record.get("per_shape", []) if want and (e["M"], e["N"], e["K"]) == (row["M"], row["N"], row["K"])
               and e.get("ca_c") == 1 and want in e["kernel"]]
        if not hit:
            return None
        got.append(hit[0]["dram_bytes"])
    return int(round(sum(got) / len(got))) if got else None


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return {"bf16_tflops": float(d["bf16_tflops"]), "hbm_gbs": float(d["hbm_gbs"]),
                "bf16_tflops_sustained": float(d.get("bf16_tflops_sustained", d["bf16_tflops"])),
                "source": "measured"}
    except Exception:
        return dict(FALLBACK_PEAKS, source="fallback")


F8_PEAK_RATIO = 2.0  # dense 8-bit / bf16 tensor rate, nominal (4.5 / 2.25 PFLOP/s)


def roofline_time_s(s, peaks, ab="bf16"):
    """max(compute time at the dense peak, compulsory bytes at HBM bandwidth);
    8-bit inputs: one byte per element and the bf16 peak x F8_PEAK_RATIO."""
    o = 4 if s["out"] == "f32" else 2
    ib = 2 if ab == "bf16" else 1
    flops = 2.0 * s["M"] * s["N"] * s["K"]
    bytes_min = ib * (s["M"] * s["K"] + s["K"] * s["N"]) + o * s["M"] * s["N"]
    t_tc = flops / (peaks["bf16_tflops"] * (1.0 if ab == "bf16" else F8_PEAK_RATIO) * 1e12)
    t_hbm = bytes_min / (peaks["hbm_gbs"] * 1e9)
    return max(t_tc, t_hbm), ("tensor" if t_tc >= t_hbm else "hbm")


def method_roofline_time_s(s, peaks, c, ab="bf16"):
    """roofline_time_s with the K split's own traffic counted: c > 1 fp32 copies
    of C written and read back by the final reduction (Sec. II-C, Listing 1)."""
    t, _ = roofline_time_s(s, peaks, ab)
    if c <= 1:
        return t
    o = 4 if s["out"] == "f32" else 2
    ib = 2 if ab == "bf16" else 1
    bytes_method = ib * (s["M"] * s["K"] + s["K"] * s["N"]) + o * s["M"] * s["N"] + 8.0 * c * s["M"] * s["N"]
    return max(t, bytes_method / (peaks["hbm_gbs"] * 1e9))


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
    dev = "cpu" if dist.get_backend() == "gloo" else "cuda"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
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
        sm, mx, power, reasons = [], [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in csv.reader(io.StringIO(out)):
            r = [x.strip() for x in r]
            if len(r) < 9:
                continue
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
                power.append(float(r[3]))
            except ValueError:
                continue
            for name, val in zip(names, r[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "power_w_max": max(power), "reasons": sorted(reasons)}


# ------------------------------------------------------------------- our arm

_SHARED = {}


def make_inputs(s, synth, torch, ab="bf16"):
    def dev(t):
        full = t.as_strided((t.shape[0], t.stride(0)), (t.stride(0), 1))
        return full.contiguous().cuda()[:, : t.shape[1]]

    out_dtype = torch.float32 if s["out"] == "f32" else torch.bfloat16
    # C's rows padded to 16 bytes like those of A and B (the caller's layout; unpadded rows
    # take the library's slower direct-store epilogue, which the parity tests cover)
    esz = 4 if s["out"] == "f32" else 2
    ldc = (s["N"] * esz + 15) // 16 * 16 // esz
    C = torch.empty((s["M"], ldc), dtype=out_dtype, device="cuda")[:, : s["N"]]
    if s.get("shared"):
        def operand(rows, cols, seed):
            key = (rows, cols, seed)
            if key not in _SHARED:
                t = (synth.uniform_bf16((rows, cols), seed=seed) if ab == "bf16"
                     else synth.uniform_f8((rows, cols), ab, seed=seed))
                _SHARED[key] = (t, dev(t))
            return _SHARED[key]
        A, Ad = operand(s["M"], s["K"], 1000003 * s["M"] + s["K"])
        B, Bd = operand(s["K"], s["N"], 2000003 * s["K"] + s["N"] + 7)
        return A, B, Ad, Bd, C
    if ab != "bf16":
        # 8-bit rows padded to 16 elements (16 bytes)
        A, B = synth.gemm_inputs_f8(s["M"], s["N"], s["K"], ab, s["kind"], seed=0)

        def dev16(t):
            ld = (t.shape[1] + 15) // 16 * 16
            d = torch.zeros(t.shape[0], ld, dtype=t.dtype, device="cuda")
            d[:, : t.shape[1]] = t.cuda()
            return d[:, : t.shape[1]]
        return A, B, dev16(A), dev16(B), C
    lda = synth.pad8(s["K"])
    ldb = synth.pad8(s["N"])
    A, B = synth.gemm_inputs(s["M"], s["N"], s["K"], s["kind"], seed=0, lda=lda, ldb=ldb)
    return A, B, dev(A), dev(B), C


def run_ours(args, rank, local, world):
    import torch
    import paper_2601_16294_gb300 as sfc
    from paper_2601_16294_gb300 import synth

    torch.cuda.set_device(local)
    sfc.load()
    stream = torch.cuda.current_stream()
    shapes = workload_shapes(args)
    peaks = load_peaks()

    # inputs resident in HBM before timing (seeded on the CPU, copied once)
    mats = []
    transposed = {}  # B stored N x K: one transposed device copy per B

    def as_nk(Bd):
        if id(Bd) not in transposed:
            K, N = Bd.shape
            buf = torch.zeros(N, (K + 15) // 16 * 16, dtype=Bd.dtype, device="cuda")
            buf[:, :K] = Bd.t()
            transposed[id(Bd)] = buf[:, :K]
        return transposed[id(Bd)]

    for s in shapes:
        A, B, Ad, Bd, C = make_inputs(s, synth, torch, args.ab)
        if args.b_layout == "nk":
            Bd = as_nk(Bd)
        mats.append({"s": s, "A": A, "B": B, "Ad": Ad, "Bd": Bd, "C": C, "c": s["cs"][0]})
    torch.cuda.synchronize()

    def call(m, c):
        sfc.gemm(m["Ad"], m["Bd"], m["C"], ca_c=c, order=args.order, assign=args.assign, stream=stream,
                 b_layout=args.b_layout, k_block_factor=args.k_block_factor)

    def hold(host_s):
        # a spin kernel of about twice host_s at the maximum SM clock (longer at a lower clock);
        # without torch's spin kernel the pairs may also hold gaps where the device waited
        if hasattr(torch.cuda, "_sleep"):
            torch.cuda._sleep(int(min(max(2.0 * host_s, 1e-4), 0.2) * HOLD_HZ))

    # the tensor cores' per-SM rate from resident operands (untimed), for the clock-based peak
    mma_per_clk = None
    if args.ab == "bf16":
        try:
            mma_per_clk = sfc.mma_peak(iters=2048, stream=stream)[0]
        except Exception:
            mma_per_clk = None

    # measure each shape's tiles (and layer counts where several are listed) once, untimed; the
    # timed calls below keep tile="auto", which then uses the measured choice (the tile never
    # changes the result's bits)
    tuned = {}
    if not args.no_tune and args.k_block_factor == 1:
        for i, m in enumerate(mats):
            # the configured layer counts, and the time model's own count, so that the library's
            # choice (ca_c = 0) is measured too
            model_c = sfc.plan(m["s"]["M"], m["s"]["N"], m["s"]["K"], 0, out_dtype=m["C"].dtype,
                               in_dtype=m["Ad"].dtype, b_layout=args.b_layout)[1]
            tuned[i] = sfc.tune(m["Ad"], m["Bd"], m["C"], max_layers=max(max(m["s"]["cs"]), model_c), max_kbf=1,
                                b_layout=args.b_layout, stream=stream)
        torch.cuda.synchronize()

    # pick the K-layer count per shape where several are listed (timed, warm), and time the
    # library's own choice (ca_c = 0) beside them: three interleaved rounds of 5 calls per count,
    # the minimum kept, so that neither a clock or power change during one round nor the order
    # decides
    def timed5(m, c):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(5):
            call(m, c)
        e1.record(stream)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / 5

    cs_report = {}
    for i, m in enumerate(mats):
        if len(m["s"]["cs"]) == 1:
            continue
        Kt = (m["s"]["K"] + 63) // 64
        cands = [c for c in m["s"]["cs"] if c * args.k_block_factor <= Kt] + [0]
        t_min = {c: float("inf") for c in cands}
        for r in range(3):
            # each round in another order, each count after two untimed calls of its own (the
            # previous count's partials may still be dirty in L2)
            for c in cands[r % len(cands):] + cands[:r % len(cands)]:
                for _ in range(2):
                    call(m, c)
                t_min[c] = min(t_min[c], timed5(m, c))
        configured = {c: t for c, t in t_min.items() if c != 0}
        m["c"] = min(configured, key=configured.get)
        cs_report[i] = {c: round(t, 4) for c, t in configured.items()}
        tile, c_auto = sfc.plan(m["s"]["M"], m["s"]["N"], m["s"]["K"], 0, out_dtype=m["C"].dtype,
                                in_dtype=m["Ad"].dtype, b_layout=args.b_layout)
        cs_report[i]["auto"] = {"ca_c": c_auto, "tile": str(tile), "ms": round(t_min[0], 4),
                                "vs_best_configured": round(t_min[0] / configured[m["c"]], 3)}

    capture_tiles = (128, 256, "pair128", "pair256")

    def step(events=None):
        if args.traffic_capture:
            for m in mats:
                for t in capture_tiles:
                    sfc.gemm(m["Ad"], m["Bd"], m["C"], ca_c=1, order=args.order, assign=args.assign, tile=t,
                             stream=stream, b_layout=args.b_layout)
            return
        for i, m in enumerate(mats):
            if events is not None:
                events[i][0].record(stream)
            call(m, m["c"])
            if events is not None:
                events[i][1].record(stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    # the host's time to issue one step with an event pair around every launch (the device is
    # idle meanwhile), for the hold kernel of the per-launch pass below
    pairs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in mats]
    h0 = time.perf_counter()
    step(pairs)
    issue_s = time.perf_counter() - h0
    torch.cuda.synchronize()
    if sfc.device_status() != 0:
        raise RuntimeError("device-side timeout during warm-up")

    # Pass 1, the headline: K steps back to back, one event pair around them.
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local, enabled=not args.no_clocks)
    time.sleep(0.2 if clocks.proc else 0)
    barrier(world)
    torch.cuda.synchronize()
    # an NVTX range around the timed steps lets a profiler capture exactly them
    # (ncu --nvtx --nvtx-include "sfc_timed_steps/")
    torch.cuda.nvtx.range_push("sfc_timed_steps")
    t0.record(stream)
    for k in range(args.steps):
        step()
    t1.record(stream)
    torch.cuda.nvtx.range_pop()
    torch.cuda.synchronize()
    barrier(world)
    clock_info = clocks.stop()
    status = sfc.device_status()
    if status != 0:
        raise RuntimeError("device-side timeout in the timed region (status %d)" % status)
    if args.traffic_capture:
        return {"traffic_capture": [{"M": m["s"]["M"], "N": m["s"]["N"], "K": m["s"]["K"], "ca_c": 1, "tile": str(t)}
                                    for _ in range(args.steps) for m in mats for t in capture_tiles],
                "kernel_sha": kernel_sha(), "workload": args.workload}

    elapsed_ms = max_over_ranks(t0.elapsed_time(t1), world)
    flops_step = sum(2.0 * m["s"]["M"] * m["s"]["N"] * m["s"]["K"] for m in mats)
    value = world * flops_step * args.steps / (elapsed_ms * 1e-3) / 1e12
    ms_per_step = elapsed_ms / args.steps

    # Pass 2: the same steps with an event pair around every launch (the
    # GEMM's, plus the K-layer reduction's where ca_c > 1): per-launch device
    # time of each shape, each launch started cold after the other shapes.
    per_launch = [[(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in mats] for _ in range(args.steps)]
    torch.cuda.synchronize()
    # each step is issued behind a hold kernel that keeps the stream busy for twice the host's
    # issue time, so every launch is queued before the device reaches it and each event pair
    # holds the launch's device time (started after the previous launch finished), not gaps
    # where the device waited for the host
    for k in range(args.steps):
        hold(issue_s)
        step(per_launch[k])
    torch.cuda.synchronize()

    # Pass 3: each shape alone, launches back to back, rotating over enough
    # copies of its inputs that they are re-read only after > 256 MB of other
    # inputs went through L2.
    b2b_ms = []
    for m in mats:
        s_ = m["s"]
        in_bytes = (2 if args.ab == "bf16" else 1) * (s_["M"] * s_["K"] + s_["K"] * s_["N"])
        copies = max(1, min(16, -(-(256 << 20) // in_bytes)))
        extra = [(m["Ad"], m["Bd"])]
        def clone_strided(t):  # keeps the padded row stride (16-byte aligned rows)
            return torch.empty_strided(t.size(), t.stride(), dtype=t.dtype, device=t.device).copy_(t)

        for _ in range(copies - 1):
            extra.append((clone_strided(m["Ad"]), clone_strided(m["Bd"])))
        reps = max(2 * copies, min(400, int(0.05 / max(roofline_time_s(s_, peaks, args.ab)[0], 1e-6))))
        for a, b in extra:
            sfc.gemm(a, b, m["C"], ca_c=m["c"], order=args.order, assign=args.assign, stream=stream,
                     b_layout=args.b_layout, k_block_factor=args.k_block_factor)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for r in range(reps):
            a, b = extra[r % copies]
            sfc.gemm(a, b, m["C"], ca_c=m["c"], order=args.order, assign=args.assign, stream=stream,
                     b_layout=args.b_layout, k_block_factor=args.k_block_factor)
        e1.record(stream)
        torch.cuda.synchronize()
        b2b_ms.append(e0.elapsed_time(e1) / reps)
        del extra
    torch.cuda.empty_cache()

    per_shape = []
    tot_ms = 0.0
    one_kernel_ms = 0.0     # event time of the calls that are a single GEMM launch (one layer, one pass)
    one_kernel_flops = 0.0
    for i, m in enumerate(mats):
        s = m["s"]
        ts = [per_launch[k][i][0].elapsed_time(per_launch[k][i][1]) for k in range(args.steps)]
        mean = sum(ts) / len(ts)
        tot_ms += sum(ts)
        if m["c"] == 1 and args.k_block_factor == 1:
            one_kernel_ms += sum(ts)
            one_kernel_flops += 2.0 * s["M"] * s["N"] * s["K"] * args.steps
        flops = 2.0 * s["M"] * s["N"] * s["K"]
        t_roof, bound = roofline_time_s(s, peaks, args.ab)
        row = {"M": s["M"], "N": s["N"], "K": s["K"], "out": s["out"], "ca_c": m["c"],
               "ms_mean": round(mean, 4), "ms_median": round(statistics.median(ts), 4), "ms_min": round(min(ts), 4),
               "tflops": round(flops / (mean * 1e-3) / 1e12, 1), "bound": bound,
               "frac_of_roofline": round(t_roof / (mean * 1e-3), 4),
               "ms_back_to_back": round(b2b_ms[i], 4),
               "tflops_back_to_back": round(flops / (b2b_ms[i] * 1e-3) / 1e12, 1),
               "frac_of_roofline_back_to_back": round(t_roof / (b2b_ms[i] * 1e-3), 4)}
        if i in cs_report:
            row["ms_by_ca_c"] = cs_report[i]
        tile, c_eff = sfc.plan(s["M"], s["N"], s["K"], m["c"], out_dtype=m["C"].dtype, in_dtype=m["Ad"].dtype,
                               b_layout=args.b_layout)
        row["tile"] = tile
        try:  # the library's time model for the same call on GB300's figures (no device query)
            row["model_us"] = round(sfc.binding.plan_model(s["M"], s["N"], s["K"], m["c"], out=s["out"], ab=args.ab,
                                                           b_layout=args.b_layout)[2] / 1e3, 1)
        except Exception:
            pass
        if c_eff > 1:
            # the method's roofline: the layer partials' traffic counted too
            row["frac_of_method_roofline"] = round(method_roofline_time_s(s, peaks, c_eff, args.ab) / (mean * 1e-3), 4)
        per_shape.append(row)

    # roofline of the dominant kernel, the GEMM kernel: over the calls that are one launch of it
    # (one K layer, one pass), which carry most of the step's time; the K-layer calls also hold
    # the reduction kernel in their event pairs and are reported per shape instead
    if one_kernel_ms > 0.0:
        achieved = one_kernel_flops / (one_kernel_ms * 1e-3) / 1e12
    else:
        achieved = flops_step * args.steps / (tot_ms * 1e-3) / 1e12
    traffic = None
    if not args.sizes and not args.shapes and args.workload in TRAFFIC_FILES:
        try:
            with open(TRAFFIC_FILES[args.workload]) as f:
                traffic = traffic_per_launch(json.load(f), per_shape, args.workload, kernel_sha())
        except (OSError, ValueError):
            traffic = None
    # burst peak for a short timed region, sustained (power-capped) peak for a long one;
    # 8-bit inputs: the measured bf16 peak times the nominal 8-bit / bf16 ratio
    sustained = elapsed_ms > 500.0
    ratio = 1.0 if args.ab == "bf16" else F8_PEAK_RATIO
    burst = peaks["bf16_tflops"] * ratio
    peak = (peaks["bf16_tflops_sustained"] if sustained else peaks["bf16_tflops"]) * ratio
    roofline = {"bound": "tensor", "achieved": round(achieved, 1), "peak": round(peak, 1), "unit": "TFLOP/s",
                "frac": round(achieved / peak, 4), "traffic": traffic,
                "kernel": "sfc_gemm_pair_kernel<256> (the tile AUTO picks for the dominant shapes)",
                "launches": "the calls with one K layer: %d of %d shapes, %.1f %% of the step's event time" % (
                    sum(1 for m in mats if m["c"] == 1), len(mats),
                    100.0 * (one_kernel_ms if one_kernel_ms > 0 else tot_ms) / tot_ms),
                "peak_source": "%s dense bf16 %s (timed region %.0f ms)%s" % (
                    peaks["source"], "sustained" if sustained else "burst", elapsed_ms,
                    "" if args.ab == "bf16" else " x %.1f, the nominal 8-bit / bf16 ratio" % ratio),
                "frac_of_burst_peak": round(achieved / burst, 4)}
    if mma_per_clk and clock_info is not None and clock_info.get("sm_mhz"):
        # the same kernel's ceiling at the clock the timed region actually ran at
        at_clock = world_sms(torch) * mma_per_clk * clock_info["sm_mhz"] * 1e6 / 1e12
        roofline["clock_peak"] = {"flop_per_clk_per_sm": round(mma_per_clk, 1),
                                  "source": "sfc_mma_peak: back-to-back pair MMAs from resident operands",
                                  "tflops_at_median_sm_clock": round(at_clock, 1),
                                  "frac": round(achieved / at_clock, 4)}
    def launches_per_call(m):
        # GEMM launches (one per K block) plus the reduction when partials go through the workspace
        c = m["c"] if m["c"] else sfc.plan(m["s"]["M"], m["s"]["N"], m["s"]["K"], 0, out_dtype=m["C"].dtype,
                                           in_dtype=m["Ad"].dtype, b_layout=args.b_layout)[1]
        kbf = args.k_block_factor
        return kbf + (1 if c > 1 or (kbf > 1 and m["C"].dtype != torch.float32) else 0)

    launches = args.steps * sum(launches_per_call(m) for m in mats)
    desc = describe(args)
    result = {
        "metric": METRIC, "value": round(value, 1), "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": args.ab,
        "data": "synthetic (seeded %s %s)" % (",".join(sorted({m["s"]["kind"] for m in mats})), args.ab),
        "config": {"workload": desc, "order": args.order, "assign": args.assign, "b_layout": args.b_layout,
                   "inputs": args.ab, "k_block_factor": args.k_block_factor,
                   "tile": "measured per shape before timing (sfc_gemm_tune, untimed)" if tuned
                           else "the library's time model",
                   "parallelism": "replicas" if world > 1 else "single GPU",
                   "l2": "inputs larger than L2 between reuses: one step runs every shape once, so a shape's "
                         "operands are re-read only after the other shapes' traffic has passed through L2",
                   "timing": "value: one event pair around the K steps; per_shape ms_mean: a second pass of the "
                             "same steps with an event pair around each call, each step issued behind a hold "
                             "kernel so that the pairs hold device time, not host issue; ms_back_to_back: each shape alone, "
                             "launches back to back over rotating input copies (> 256 MB between reuses)",
                   "pct_of_dense_peak": round(100.0 * value / world / burst, 2)},
        "roofline": roofline,
        "gpu_launches": launches,
        "per_shape": per_shape,
    }
    if cs_report:
        # the library's own layer count and tile (ca_c = 0) against the best configured count
        r = [(mats[i]["s"], v["auto"]["vs_best_configured"]) for i, v in cs_report.items()]
        worst = max(r, key=lambda x: x[1])
        result["library_choice"] = {
            "shapes": len(r), "within_5pct_of_best": sum(1 for _, q in r if q <= 1.05),
            "faster_than_best": sum(1 for _, q in r if q < 1.0),
            "worst": {"M": worst[0]["M"], "N": worst[0]["N"], "K": worst[0]["K"], "ratio": worst[1]},
            "timing": "min over three interleaved rounds (rotated order) of 5 back-to-back calls per count, "
                      "each after two untimed calls"}
    if clock_info is not None:
        result["clocks"] = clock_info
    if not args.no_cublas and world == 1:
        result["cublas_same_window"] = run_cublas_compare(args, mats, stream, call, hold)
    if not args.no_e2e:
        result["e2e"] = run_e2e(args, mats, stream, world)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = run_cpu_baseline(mats)
    return result


def run_cublas_compare(args, mats, stream, call, hold):
    """Comparison only: torch.matmul (cuBLAS) on the same shapes, alternating
    step by step with this library so both see the same clocks and power."""
    import torch

    one = torch.ones((), dtype=torch.float32, device="cuda")
    colmajor = {}

    def cublas(m):
        if args.ab != "bf16":
            # cuBLAS's 8-bit GEMM (torch._scaled_mm, unit scales) wants B column-major
            if id(m["Bd"]) not in colmajor:
                colmajor[id(m["Bd"])] = (m["Bd"].t().contiguous().t() if args.b_layout == "kn" else m["Bd"].t())
            out = torch._scaled_mm(m["Ad"], colmajor[id(m["Bd"])], scale_a=one, scale_b=one,
                                   out_dtype=m["C"].dtype)
            m["C"].copy_(out)
            return
        Bd = m["Bd"].t() if args.b_layout == "nk" else m["Bd"]
        if m["C"].dtype == torch.bfloat16:
            torch.matmul(m["Ad"], Bd, out=m["C"])
        else:
            m["C"].copy_(torch.matmul(m["Ad"], Bd))

    steps = max(3, min(args.steps, 50))
    t = [[0.0, 0.0] for _ in mats]
    try:
        for _ in range(2):
            for m in mats:
                cublas(m)
    except Exception as e:  # e.g. a shape cuBLAS's 8-bit GEMM does not take
        return {"unavailable": "cuBLAS comparison failed: %s" % str(e).splitlines()[0][:200]}
    arms = (lambda m: call(m, m["c"]), cublas)
    # one untimed step of each arm first, its host issue time measured (the device is busy)
    torch.cuda.synchronize()
    issue_s = []
    for arm in arms:
        h0 = time.perf_counter()
        for m in mats:
            arm(m)
        issue_s.append(time.perf_counter() - h0)
    torch.cuda.synchronize()
    # (1) an event pair around every call; each arm's step is issued behind a hold kernel of
    # twice its host issue time, so each pair holds the call's device time, started after the
    # previous call finished
    evs = []
    for k in range(steps):
        for which in (0, 1):
            hold(issue_s[which])
            ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in mats]
            for i, m in enumerate(mats):
                ev[i][0].record(stream)
                arms[which](m)
                ev[i][1].record(stream)
            evs.append((which, ev))
    torch.cuda.synchronize()
    for which, ev in evs:
        for i in range(len(mats)):
            t[i][which] += ev[i][0].elapsed_time(ev[i][1])
    # (2) one event pair around each arm's whole step, calls back to back as a caller issues them
    # (this library's launches then overlap their start with the previous launch's end)
    step_ev = []
    for k in range(steps):
        for which in (0, 1):
            hold(issue_s[which])
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for m in mats:
                arms[which](m)
            e1.record(stream)
            step_ev.append((which, e0, e1))
    torch.cuda.synchronize()
    t_step = [0.0, 0.0]
    for which, e0, e1 in step_ev:
        t_step[which] += e0.elapsed_time(e1)
    fl = [2.0 * m["s"]["M"] * m["s"]["N"] * m["s"]["K"] * steps for m in mats]
    ours, cub = sum(x[0] for x in t), sum(x[1] for x in t)
    return {"cublas_tflops": round(sum(fl) / (cub * 1e-3) / 1e12, 1),
            "ours_tflops": round(sum(fl) / (ours * 1e-3) / 1e12, 1), "steps": steps,
            "back_to_back": {"cublas_tflops": round(sum(fl) / (t_step[1] * 1e-3) / 1e12, 1),
                             "ours_tflops": round(sum(fl) / (t_step[0] * 1e-3) / 1e12, 1),
                             "timing": "one event pair around each arm's step of back-to-back calls"},
            "per_shape": [{"M": m["s"]["M"], "N": m["s"]["N"], "K": m["s"]["K"],
                           "ours": round(f / (x[0] * 1e-3) / 1e12, 1), "cublas": round(f / (x[1] * 1e-3) / 1e12, 1)}
                          for m, f, x in zip(mats, fl, t)],
            "note": "alternating steps, same stream, each step issued behind a hold kernel (one synchronisation "
                    "at the end); cublas_tflops / ours_tflops: an event pair around every call; cuBLAS output is "
                    "bf16 (fp32 rows: bf16 GEMM then cast)"}


def run_e2e(args, mats, stream, world):
    """Same metric through the public API from pinned HOST buffers: every step
    copies A and B host->device, runs the GEMM, copies C device->host (the
    library pipelines the copies against the GEMMs in slices)."""
    import torch
    import paper_2601_16294_gb300 as sfc

    pinned = {}  # operands shared between shapes are pinned once (each shape still copies them)

    def pin(t):
        if id(t) not in pinned:
            pinned[id(t)] = t.contiguous().pin_memory()
        return pinned[id(t)]

    nk = {}  # host copies of B stored N x K, one per B

    def host_b(B):
        if args.b_layout == "kn":
            return pin(B)
        if id(B) not in nk:
            nk[id(B)] = B.t().contiguous().pin_memory()
        return nk[id(B)]

    host = []
    for m in mats:
        host.append((m, pin(m["A"]), host_b(m["B"]), torch.empty(m["C"].shape, dtype=m["C"].dtype, pin_memory=True)))
    if args.e2e_order == "largest_first":
        host.sort(key=lambda h: -h[0]["s"]["M"] * h[0]["s"]["N"] * h[0]["s"]["K"])
    h2d = sum(Ah.numel() * 2 + Bh.numel() * 2 for _, Ah, Bh, _ in host)
    d2h = sum(Ch.numel() * Ch.element_size() for _, _, _, Ch in host)

    def step():
        # every shape's call is enqueued, then one synchronisation: the library
        # overlaps a call's uploads and downloads with the GEMMs
        for m, Ah, Bh, Ch in host:
            sfc.gemm_host(Ah, Bh, Ch, ca_c=m["c"], out_dtype=Ch.dtype, stream=stream, b_layout=args.b_layout)
        stream.synchronize()

    for _ in range(2):
        step()
    steps = max(1, min(args.steps, 5))
    barrier(world)
    torch.cuda.synchronize()
    t = time.perf_counter()
    for _ in range(steps):
        step()
    torch.cuda.synchronize()
    el = max_over_ranks(time.perf_counter() - t, world)
    flops = sum(2.0 * m["s"]["M"] * m["s"]["N"] * m["s"]["K"] for m in mats) * steps * world
    return {"value": round(flops / el / 1e12, 1), "unit": "TFLOP/s", "h2d_bytes_per_step": h2d,
            "d2h_bytes_per_step": d2h, "steps": steps,
            "api": "paper_2601_16294_gb300.gemm_host -> sfc_gemm_host (C ABI, host buffers)",
            "order": args.e2e_order}


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
    for A, B in mats_cpu:
        M, K = A.shape
        N = B.shape[1]
        r = np.linspace(0, M - 1, min(rows, M)).astype(np.int64)
        fmt = {"torch.float8_e4m3fn": "e4m3", "torch.float8_e5m2": "e5m2"}.get(str(A.dtype))
        if fmt:  # 8-bit tensors are sampled through their byte view
            import torch
            A_rows = A.view(torch.uint8)[r].contiguous().numpy()
            Bc = B.view(torch.uint8).contiguous().numpy()
        else:
            A_rows = A[r].contiguous()
            Bc = B.contiguous()
        t0 = time.perf_counter()
        if fmt:
            oracle.gemm_f8_f64(A_rows, Bc, fmt)
        else:
            oracle.gemm_f64(A_rows, Bc)
        t += time.perf_counter() - t0
        flops += 2.0 * r.size * N * K
    return flops, t


def run_cpu_baseline(mats, budget_s=12.0, one_core_s=4.0):
    """The oracle as it stands, on this host's cores, on a bounded sample of the
    workload: a 16-row probe sets the row count for about ``budget_s`` of CPU
    work.  Then the same oracle on one core, for about ``one_core_s``."""
    from oracle import oracle
    os.environ.setdefault("OMP_NUM_THREADS", str(cpu_cores()))
    cores = int(os.environ["OMP_NUM_THREADS"])
    oracle.set_threads(cores)
    mats_cpu = [(m["A"], m["B"]) for m in mats]
    _, s_probe = oracle_sample(mats_cpu, 16)
    rows = int(min(1024, max(16, 16 * budget_s / max(s_probe, 1e-3))))
    rows = max(16, rows // 16 * 16)
    flops, secs = oracle_sample(mats_cpu, rows)
    # one core, on fewer rows: the all-core rate times the core count predicts the time
    rows1 = int(max(2, min(rows, rows * one_core_s / max(secs * cores, 1e-6))))
    oracle.set_threads(1)
    try:
        flops1, secs1 = oracle_sample(mats_cpu, rows1)
    finally:
        oracle.set_threads(cores)
    return {"value": round(flops / secs / 1e12, 6), "unit": "TFLOP/s",
            "cores": cores, "kind": "oracle", "seconds": round(secs, 2),
            "sample": "%d evenly spaced rows of C for each shape (fp64 triple loop, OpenMP over rows)"
                      % rows,
            "one_core": {"value": round(flops1 / secs1 / 1e12, 6), "unit": "TFLOP/s", "cores": 1,
                         "seconds": round(secs1, 2),
                         "sample": "%d evenly spaced rows of C for each shape" % rows1}}


# ------------------------------------------------------------- reference arm

def run_reference(args, rank, world):
    """The CPU oracle as the reference arm: each step computes sampled rows of
    every shape of the workload (bounded so the run ends within minutes)."""
    if rank != 0:
        return None
    from paper_2601_16294_gb300 import synth
    os.environ.setdefault("OMP_NUM_THREADS", str(cpu_cores()))
    shapes = workload_shapes(args)
    mats_cpu = []
    for s in shapes:
        if args.ab == "bf16":
            A, B = synth.gemm_inputs(s["M"], s["N"], s["K"], s["kind"], seed=0)
        else:
            A, B = synth.gemm_inputs_f8(s["M"], s["N"], s["K"], args.ab, s["kind"], seed=0)
        mats_cpu.append((A, B))
    rows = 16
    for _ in range(args.warmup):
        oracle_sample(mats_cpu, 2)
    flops = secs = 0.0
    for _ in range(args.steps):
        f, s = oracle_sample(mats_cpu, rows)
        flops += f
        secs += s
    value = flops / secs / 1e12
    cores = int(os.environ["OMP_NUM_THREADS"])
    sample = "%d evenly spaced rows of C per shape per step" % rows
    desc = describe(args)
    return {"impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(1e3 * secs / args.steps, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded %s)" % args.ab, "config": {"workload": desc, "sample": sample,
                                                                  "inputs": args.ab},
            "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}


def world_sms(torch):
    return torch.cuda.get_device_properties(torch.cuda.current_device()).multi_processor_count


def run_sustained(args):
    """Sustained, power-capped phases: each configuration runs back to back for
    --phase-seconds while nvidia-smi samples the SM clock and board power every
    50 ms; medians over the second half of each phase (steady state)."""
    import torch
    import paper_2601_16294_gb300 as sfc

    torch.cuda.set_device(0)
    sfc.load()
    sizes = [int(x) for x in (args.sizes or "16384,8192").split(",")]
    phases = []

    def phase(name, n, fn):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        smi = subprocess.Popen(["nvidia-smi", "--query-gpu=clocks.sm,power.draw", "--format=csv,noheader,nounits",
                                "-lms", "50"], stdout=subprocess.PIPE, text=True)
        time.sleep(0.3)
        calls = 0
        t0 = time.time()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        while time.time() - t0 < args.phase_seconds:
            for _ in range(5):
                fn()
            calls += 5
            torch.cuda.synchronize()
        e1.record()
        torch.cuda.synchronize()
        smi.terminate()
        out = smi.communicate()[0]
        rows = [line.split(",") for line in out.strip().splitlines() if line.strip()]
        half = rows[len(rows) // 2:] or rows
        clk = statistics.median(float(r[0]) for r in half) if half else None
        pw = statistics.median(float(r[1]) for r in half) if half else None
        tf = 2.0 * n ** 3 * calls / (e0.elapsed_time(e1) * 1e-3) / 1e12
        phases.append({"phase": name, "size": n, "tflops": round(tf, 1), "sm_mhz": clk, "power_w": pw,
                       "tflops_per_ghz": round(tf / clk * 1e3, 1) if clk else None, "calls": calls})
        print(json.dumps(phases[-1]), file=sys.stderr, flush=True)

    for n in sizes:
        A = torch.empty(n, n, dtype=torch.bfloat16, device="cuda").uniform_(-1, 1)
        B = torch.empty(n, n, dtype=torch.bfloat16, device="cuda").uniform_(-1, 1)
        C = torch.empty(n, n, dtype=torch.bfloat16, device="cuda")
        ours = [("curve, dynamic dealing", dict(tile="pair256", assign="wave")),
                ("curve, static waves", dict(tile="pair256", assign="wave_static")),
                ("raster, dynamic dealing", dict(tile="pair256", assign="wave", order="raster")),
                ("curve, dynamic, k_block_factor 2", dict(tile="pair256", assign="wave", k_block_factor=2))]
        for name, kw in ours:
            phase("ours " + name, n, lambda kw=kw: sfc.gemm(A, B, C, **kw))
        phase("cuBLAS (torch.matmul)", n, lambda: torch.matmul(A, B, out=C))
        phase("ours curve, dynamic dealing (again)", n, lambda: sfc.gemm(A, B, C, tile="pair256", assign="wave"))
        del A, B, C
        torch.cuda.empty_cache()
    return {"mode": "sustained", "phase_seconds": args.phase_seconds, "out": "bf16", "inputs": "U[-1,1] bf16",
            "phases": phases}


def main():
    args = parse_args()
    if args.sustained:
        print(json.dumps(run_sustained(args)), flush=True)
        return
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
