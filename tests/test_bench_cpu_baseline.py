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
