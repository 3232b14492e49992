"""bench.py's per-launch DRAM traffic: the lookup into a per-tile record, and the committed
records, which must hold one capture for every shape of their workload with every tile."""
import json
import os

import bench

ROW = {"M": 64, "N": 32, "K": 16, "ca_c": 1, "tile": "pair256"}


def record(**kw):
    r = {"kernel_sha": "abc", "workload": "configs",
         "per_shape": [{"M": 64, "N": 32, "K": 16, "ca_c": 1, "kernel": "sfc_gemm_pair_kernel<256", "dram_bytes": 100},
                       {"M": 64, "N": 32, "K": 16, "ca_c": 1, "kernel": "sfc_gemm_kernel<256", "dram_bytes": 50},
                       {"M": 8, "N": 8, "K": 8, "ca_c": 1, "kernel": "sfc_gemm_kernel<128", "dram_bytes": 10}]}
    r.update(kw)
    return r


def test_matches_shape_and_kernel_and_averages():
    rows = [ROW, dict(ROW, tile=256), {"M": 8, "N": 8, "K": 8, "ca_c": 1, "tile": 128}]
    assert bench.traffic_per_launch(record(), rows, "configs", "abc") == round((100 + 50 + 10) / 3)


def test_layered_calls_are_left_out():
    rows = [ROW, dict(ROW, ca_c=4, tile=128)]
    assert bench.traffic_per_launch(record(), rows, "configs", "abc") == 100


def test_unknown_when_any_call_lacks_a_capture_or_the_record_is_stale():
    assert bench.traffic_per_launch(record(), [ROW, dict(ROW, tile="pair128")], "configs", "abc") is None
    assert bench.traffic_per_launch(record(), [ROW], "configs", "other") is None
    assert bench.traffic_per_launch(record(), [ROW], "square", "abc") is None
    assert bench.traffic_per_launch(record(), [dict(ROW, ca_c=2)], "configs", "abc") is None


def test_committed_records_cover_every_shape_and_tile():
    class A:
        shapes = sizes = ca_c = None
        out = "workload"

    for workload, path in bench.TRAFFIC_FILES.items():
        with open(path) as f:
            rec = json.load(f)
        assert rec["workload"] == workload and len(rec["kernel_sha"]) == 16
        args = A()
        args.workload = workload
        for s in bench.workload_shapes(args):
            for tile in bench.TILE_KERNEL:
                row = {"M": s["M"], "N": s["N"], "K": s["K"], "ca_c": 1, "tile": tile}
                assert bench.traffic_per_launch(rec, [row], workload, rec["kernel_sha"]) > 0, (workload, row)
