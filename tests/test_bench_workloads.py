"""bench.py's workloads are the paper's configurations: the square sweep, the
LLM-prefill projections, the irregular shapes, the communication-avoiding
high-K cases, the 125-shape sweep and the single 512^3 GEMM, each with its input
distribution, output type and set of K-layer counts (CPU only)."""
import argparse
import itertools
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402

CS = (1, 2, 4, 8)


def dims(name):
    return [(s["M"], s["N"], s["K"]) for s in bench.WORKLOADS[name]["shapes"]]


def test_square_sweep():
    assert dims("square") == [(n, n, n) for n in (2048, 4096, 8192, 16384)]
    assert all(s["out"] == "bf16" and s["cs"] == (1,) and s["kind"] == "uniform"
               for s in bench.WORKLOADS["square"]["shapes"])


def test_prefill_projections():
    want = {(m, n, k) for m in (512, 2048, 8192) for (n, k) in ((4096, 4096), (14336, 4096), (4096, 14336),
                                                               (128256, 4096))}
    assert set(dims("prefill")) == want and len(dims("prefill")) == 12
    assert all(s["kind"] == "prefill" and s["out"] == "bf16" and s["cs"] == CS
               for s in bench.WORKLOADS["prefill"]["shapes"])


def test_irregular_shapes():
    assert dims("irregular") == [(3000, 5000, 7000), (1000, 17000, 2500), (6144, 768, 12288), (129, 8191, 4096)]
    assert all(s["cs"] == CS and s["out"] == "bf16" for s in bench.WORKLOADS["irregular"]["shapes"])


def test_high_k_cases():
    assert set(dims("highk")) == {(m, m, k) for m in (512, 1024, 2048) for k in (32768, 65536, 131072)}
    assert all(s["out"] == "f32" and s["cs"] == CS for s in bench.WORKLOADS["highk"]["shapes"])


def test_sweep_of_125_shapes():
    sizes = (512, 1024, 2048, 4096, 8192)
    assert sorted(dims("sweep125")) == sorted(itertools.product(sizes, sizes, sizes))
    assert all(s["shared"] and s["cs"] == CS for s in bench.WORKLOADS["sweep125"]["shapes"])


def test_default_workload_is_configs_two_to_five():
    # the metric's weighted harmonic mean spans the square, prefill, irregular and high-K sets
    assert bench.parse_args.__defaults__ is None
    import sys as _sys
    argv = _sys.argv
    try:
        _sys.argv = ["bench.py"]
        assert bench.parse_args().workload == "configs"
    finally:
        _sys.argv = argv
    shapes = bench.WORKLOADS["configs"]["shapes"]
    assert len(shapes) == 29
    assert shapes == (bench.WORKLOADS["square"]["shapes"] + bench.WORKLOADS["prefill"]["shapes"] +
                      bench.WORKLOADS["irregular"]["shapes"] + bench.WORKLOADS["highk"]["shapes"])


def test_single_512_cube():
    assert dims("cube512") == [(512, 512, 512)]
    assert bench.WORKLOADS["cube512"]["shapes"][0]["out"] == "f32"


def args(**kw):
    base = dict(workload="square", sizes=None, ca_c=None, out="workload")
    base.update(kw)
    return argparse.Namespace(**base)


def test_overrides():
    s = bench.workload_shapes(args(sizes="256,1024"))
    assert [(x["M"], x["N"], x["K"]) for x in s] == [(256, 256, 256), (1024, 1024, 1024)]
    s = bench.workload_shapes(args(workload="highk", ca_c=4, out="bf16"))
    assert all(x["cs"] == (4,) and x["out"] == "bf16" for x in s)
    # the table itself is not modified by an override
    assert all(x["cs"] == CS and x["out"] == "f32" for x in bench.WORKLOADS["highk"]["shapes"])
    with pytest.raises(SystemExit):
        bench.workload_shapes(args(workload="prefill", sizes="256"))
