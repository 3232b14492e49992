"""bench.py's CPU-baseline leg: the oracle timed on all of the host's cores and
on one core, over sampled rows of the workload (tiny sizes and budgets here)."""
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from oracle import oracle  # noqa: E402
from paper_2601_16294_gb300 import synth  # noqa: E402


def test_cpu_baseline_reports_all_cores_and_one_core():
    mats = []
    for (M, N, K) in [(96, 80, 64), (40, 130, 72)]:
        A, B = synth.gemm_inputs(M, N, K, "uniform", seed=3)
        mats.append({"A": A, "B": B})
    c = bench.run_cpu_baseline(mats, budget_s=0.05, one_core_s=0.02)
    assert c["kind"] == "oracle" and c["unit"] == "TFLOP/s" and c["value"] > 0
    assert c["cores"] == int(os.environ["OMP_NUM_THREADS"]) >= 1
    one = c["one_core"]
    assert one["cores"] == 1 and one["value"] > 0 and one["unit"] == "TFLOP/s"
    # the oracle's loops are back on every core afterwards
    assert oracle.max_threads() == c["cores"]


def test_roofline_times():
    peaks = {"bf16_tflops": 2000.0, "hbm_gbs": 8000.0}
    # compute-bound square: 2 n^3 flops at the peak
    sq = {"M": 4096, "N": 4096, "K": 4096, "out": "bf16"}
    t, bound = bench.roofline_time_s(sq, peaks)
    assert bound == "tensor" and abs(t - 2 * 4096 ** 3 / 2000e12) < 1e-12
    # a skinny high-K shape is bound by the compulsory bytes: 2 (MK + KN) + 4 MN
    hk = {"M": 128, "N": 128, "K": 131072, "out": "f32"}
    t, bound = bench.roofline_time_s(hk, peaks)
    want = (2 * (128 * 131072 * 2) + 4 * 128 * 128) / 8000e9
    assert bound == "hbm" and abs(t - want) < 1e-12
    # the method's roofline adds the c fp32 layer copies, written and read back
    assert bench.method_roofline_time_s(hk, peaks, 1) == t
    want8 = want + 8 * 8 * 128 * 128 / 8000e9
    assert abs(bench.method_roofline_time_s(hk, peaks, 8) - want8) < 1e-12
    # on a compute-bound shape the partials do not move the bound
    assert bench.method_roofline_time_s(sq, peaks, 2) == bench.roofline_time_s(sq, peaks)[0]
