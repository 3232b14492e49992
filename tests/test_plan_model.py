"""The library's time model on a described device (sfc_gemm_plan_desc), on
the CPU: its picks for the measured configurations and the roofline it must
respect (Sec. III-B: a BRGEMM takes max(G gamma, beta (S_A + S_B)), Eqs. 1-4).

The device is described explicitly (GB300's figures), so these tests pin the
model itself, independent of any GPU."""
import pytest

from paper_2601_16294_gb300 import binding

GB300 = dict(num_sms=152, pair_workers=76, hbm_gbs=6700.0, sm_ghz=1.9)
FLOP_PER_CLK_PER_SM = 8192.0  # dense bf16 MMA rate per SM per clock (measured by sfc_mma_peak)

SHAPES = ([(n, n, n, "bf16") for n in (2048, 4096, 8192, 16384)] +
          [(m, n, k, "bf16") for m in (512, 2048, 8192)
           for (n, k) in ((4096, 4096), (14336, 4096), (4096, 14336), (128256, 4096))] +
          [(3000, 5000, 7000, "bf16"), (1000, 17000, 2500, "bf16"), (6144, 768, 12288, "bf16"),
           (129, 8191, 4096, "bf16")] +
          [(m, m, k, "f32") for m in (512, 1024, 2048) for k in (32768, 65536, 131072)])


def roofline_ns(M, N, K, out, dev=GB300):
    peak = dev["num_sms"] * FLOP_PER_CLK_PER_SM * dev["sm_ghz"]  # flop per ns
    o = 4 if out == "f32" else 2
    return max(2.0 * M * N * K / peak, (2.0 * (M * K + K * N) + o * M * N) / dev["hbm_gbs"])


@pytest.mark.parametrize("M,N,K,out", SHAPES)
def test_prediction_respects_the_roofline(M, N, K, out):
    tile, c, ns = binding.plan_model(M, N, K, 0, out=out, device=GB300)
    assert tile in ("pair256", "pair128", 256, 128) and c >= 1
    # the tensor cores at 95 % of their rate at best, DRAM at the described bandwidth
    assert ns >= roofline_ns(M, N, K, out) * 0.999


def test_large_square_shapes_take_the_pair_tile_and_one_layer():
    for n in (2048, 4096, 8192, 16384):
        assert binding.plan_model(n, n, n, 0, device=GB300)[:2] == ("pair256", 1)


def test_dram_bound_high_k_splits_k_and_is_limited_by_dram():
    M = N = 512
    K = 131072
    tile, c, ns = binding.plan_model(M, N, K, 0, out="f32", device=GB300)
    assert 4 < c <= 20
    ab_bytes = 2.0 * (M * K + K * N)
    assert ns >= ab_bytes / GB300["hbm_gbs"]
    # one layer leaves most workers idle: far slower in the model
    assert binding.plan_model(M, N, K, 1, out="f32", device=GB300)[2] > 3 * ns
    # DRAM-bound: twice the bandwidth helps a lot, twice the clock little
    fast_mem = binding.plan_model(M, N, K, 0, out="f32", device=dict(GB300, hbm_gbs=13400.0))[2]
    fast_clk = binding.plan_model(M, N, K, 0, out="f32", device=dict(GB300, sm_ghz=3.8))[2]
    assert fast_mem < 0.8 * ns and fast_clk > 0.9 * ns


def test_tensor_bound_shape_follows_the_clock_not_the_bandwidth():
    ns = binding.plan_model(8192, 8192, 8192, 0, device=GB300)[2]
    fast_clk = binding.plan_model(8192, 8192, 8192, 0, device=dict(GB300, sm_ghz=3.8))[2]
    fast_mem = binding.plan_model(8192, 8192, 8192, 0, device=dict(GB300, hbm_gbs=13400.0))[2]
    assert fast_clk < 0.55 * ns and fast_mem == pytest.approx(ns)


def test_layer_partials_cost_dram_time():
    # the same split with c layers costs at least the c fp32 copies written and read back
    M = N = 1024
    K = 65536
    for c in (2, 4, 8):
        ns = binding.plan_model(M, N, K, c, out="f32", device=GB300)[2]
        assert ns >= 2 * 4.0 * c * M * N / GB300["hbm_gbs"]
    assert binding.plan_model(M, N, K, 8, out="f32", device=GB300)[1] == 8  # a fixed count is kept


def test_more_k_never_predicts_less_time():
    prev = 0.0
    for K in (1024, 2048, 4096, 8192, 16384, 32768, 65536, 131072):
        ns = binding.plan_model(512, 512, K, 0, out="f32", device=GB300)[2]
        assert ns >= prev
        prev = ns


def test_fewer_pairs_move_the_pick_to_one_sm_tiles():
    # a device whose pairs cannot be co-scheduled: only the one-SM tiles remain
    tile, c, ns = binding.plan_model(4096, 4096, 4096, 1, device=dict(GB300, pair_workers=0))
    assert tile in (128, 256)


@pytest.mark.parametrize("bad", [dict(num_sms=0), dict(pair_workers=-1), dict(pair_workers=77),
                                 dict(hbm_gbs=0.0), dict(sm_ghz=-1.0)])
def test_bad_device_descriptions_are_rejected(bad):
    with pytest.raises(binding.SfcError) as e:
        binding.plan_model(1024, 1024, 1024, 0, device=dict(GB300, **bad))
    assert e.value.code == binding.SFC_ERR_INVALID_ARG


def test_bad_sizes_are_rejected():
    for M, N, K, c in ((0, 8, 8, 1), (8, 8, 8, -1), (8, 8, 64, 2)):
        with pytest.raises(binding.SfcError):
            binding.plan_model(M, N, K, c, device=GB300)
