"""bench.py's output contract on a GPU: one JSON line with the metric, the
whole-job value, the roofline of the dominant kernel, the end-to-end rate from
host buffers, the clocks seen during the timed region, the launch count and
the oracle's CPU rate (small sizes, a few steps).  The reference arm's line is
checked on CPU (test_bench_dist.py)."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run_bench(*args):
    out = subprocess.run([sys.executable, "bench.py", *args], cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [line for line in out.stdout.splitlines() if line.strip()]
    assert len(lines) == 1, out.stdout
    return json.loads(lines[0])


def test_default_line_keys():
    d = run_bench("--sizes", "2048,4096", "--steps", "3", "--warmup", "3", "--no-cublas")
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
                "vs_baseline", "dtype", "data", "config", "roofline", "gpu_launches", "e2e", "cpu_baseline",
                "clocks", "per_shape"):
        assert key in d, key
    assert d["n_gpus"] == 1 and d["steps"] == 3 and d["warmup"] == 3 and d["higher_is_better"] is True
    assert d["value"] > 0 and d["unit"] == "TFLOP/s" and d["dtype"] == "bf16"
    assert "workload" in d["config"]
    r = d["roofline"]
    assert r["bound"] == "tensor" and r["unit"] == "TFLOP/s" and r["peak"] > 0
    assert abs(r["frac"] - r["achieved"] / r["peak"]) < 1e-3
    cp = r["clock_peak"]                                    # the MMA-only ceiling at the sampled clock
    assert 2000 < cp["flop_per_clk_per_sm"] < 20000 and 0 < cp["frac"] < 1.1
    e = d["e2e"]
    assert e["value"] > 0 and e["h2d_bytes_per_step"] == 2 * 2 * (2048 ** 2 + 4096 ** 2)   # A and B, bf16
    assert e["d2h_bytes_per_step"] == 2 * (2048 ** 2 + 4096 ** 2)
    assert d["gpu_launches"] == 3 * 2                                    # one GEMM launch per shape per step
    c = d["cpu_baseline"]
    assert c["kind"] == "oracle" and c["cores"] >= 1 and c["value"] > 0
    assert c["one_core"]["cores"] == 1 and c["one_core"]["value"] > 0
    assert {"sm_mhz", "sm_max_mhz", "reasons"} <= set(d["clocks"])
    assert len(d["per_shape"]) == 2 and all(p["tile"] for p in d["per_shape"])
    assert all(p["ms_min"] <= p["ms_median"] for p in d["per_shape"])



def test_traffic_capture_runs_every_tile_of_every_shape():
    d = run_bench("--shapes", "512x512x512,256x384x128", "--traffic-capture", "--no-tune", "--ca-c", "1",
                  "--steps", "1", "--warmup", "3", "--no-cublas", "--no-e2e", "--no-cpu-baseline", "--no-clocks")
    sys.path.insert(0, ROOT)
    import bench
    assert d["kernel_sha"] == bench.kernel_sha()
    calls = d["traffic_capture"]
    assert len(calls) == 2 * 4
    assert {(c["M"], c["N"], c["K"]) for c in calls} == {(512, 512, 512), (256, 384, 128)}
    assert {c["tile"] for c in calls} == {"128", "256", "pair128", "pair256"}
    assert all(c["ca_c"] == 1 for c in calls)


def test_layer_counts_library_choice_and_both_cublas_modes():
    d = run_bench("--shapes", "512x512x8192", "--steps", "3", "--warmup", "3", "--no-e2e", "--no-cpu-baseline",
                  "--no-clocks")
    row = d["per_shape"][0]
    assert {"1", "2", "4", "8", "auto"} <= set(row["ms_by_ca_c"])
    assert row["ca_c"] in (1, 2, 4, 8)
    assert row["ms_by_ca_c"][str(row["ca_c"])] == min(v for k, v in row["ms_by_ca_c"].items() if k != "auto")
    lc = d["library_choice"]
    assert lc["shapes"] == 1 and 0 < lc["worst"]["ratio"] < 10
    c = d["cublas_same_window"]
    assert c["ours_tflops"] > 0 and c["cublas_tflops"] > 0
    assert c["back_to_back"]["ours_tflops"] > 0 and c["back_to_back"]["cublas_tflops"] > 0
