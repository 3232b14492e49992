"""Parity of the CUDA SFC GEMM (through the C ABI) with the fp64 oracle.

Sizes here finish in the oracle within seconds yet span several tiles with
ragged M / N / K tails.  Tolerances are those of ``parity.py``; integer-valued
inputs must match bit-exactly for every K-layer count, tile order, assignment
and tile width, because every fp32 partial sum is then exact.
"""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import check_bf16, check_fp32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def to_dev(A, B):
    """Copy CPU tensors (possibly padded views) to the GPU keeping row strides."""
    def dev(t):
        base = t.as_strided((t.shape[0], t.stride(0)), (t.stride(0), 1)) if t.stride(0) != t.shape[1] else t
        d = base.contiguous().cuda()
        return d[:, : t.shape[1]]
    return dev(A), dev(B)


def run(sfc, A, B, **kw):
    Ad, Bd = to_dev(A, B)
    C = sfc.gemm(Ad, Bd, **kw)
    torch.cuda.synchronize()
    assert sfc.device_status() == 0
    return C.float().cpu().numpy().astype(np.float64)


def test_config_512_cube_fp32(sfc, oracle):
    # 512^3, uniform [-1, 1] from seed 0, fp32 output, 4 x 4 grid of 128 x 128 tiles
    A, B = synth.gemm_inputs(512, 512, 512, "uniform", seed=0)
    ref = oracle.gemm_f64(A, B)
    C = run(sfc, A, B, ca_c=1, tile=128)
    check_fp32(C, ref, 512)
    C2 = run(sfc, A, B)                           # library defaults
    check_fp32(C2, ref, 512)


SHAPES = [
    (256, 384, 512),      # whole tiles
    (200, 300, 136),      # ragged M and N, K not a multiple of 64
    (129, 257, 1000),     # one extra row / column tile, K tail of 40
    (1, 1, 8),            # degenerate
    (7, 9, 64),           # tiny
    (300, 520, 8),        # K smaller than one slab
    (640, 136, 2048),     # N smaller than a 256 tile
]


TILES = [128, 256, "pair128", "pair256"]


@pytest.mark.parametrize("M,N,K", SHAPES)
@pytest.mark.parametrize("tile", TILES)
def test_shapes_fp32_and_bf16(sfc, oracle, M, N, K, tile):
    lda, ldb = synth.pad8(K), synth.pad8(N)
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=M + N + K, lda=lda, ldb=ldb)
    ref = oracle.gemm_f64(A.contiguous(), B.contiguous())
    ref_bf16 = oracle.round_bf16(ref)
    Kt = (K + 63) // 64
    for c in [c for c in (1, 2, 4) if c <= Kt]:
        C = run(sfc, A, B, ca_c=c, tile=tile)
        check_fp32(C, ref, K)
        Cb = run(sfc, A, B, ca_c=c, tile=tile, out_dtype=torch.bfloat16)
        check_bf16(Cb, ref, ref_bf16, K)


def test_integer_inputs_bit_exact_every_variant(sfc, oracle):
    M, N, K = 384, 640, 1024
    A, B = synth.gemm_inputs(M, N, K, "int", seed=11)
    ref = oracle.gemm_f64(A, B)
    ref_bits = oracle.round_bf16_bits(ref)
    Ad, Bd = to_dev(A, B)
    for c in (1, 2, 4, 8):
        for order in ("sfc", "raster"):
            for assign in ("segment", "wave"):
                for tile in TILES:
                    C = sfc.gemm(Ad, Bd, ca_c=c, order=order, assign=assign, tile=tile)
                    assert np.array_equal(C.cpu().numpy().astype(np.float64), ref), (c, order, assign, tile)
                    Cb = sfc.gemm(Ad, Bd, ca_c=c, order=order, assign=assign, tile=tile,
                                  out_dtype=torch.bfloat16)
                    got = Cb.cpu().view(torch.int16).numpy().view(np.uint16)
                    assert np.array_equal(got, ref_bits), (c, order, assign, tile)
    assert sfc.device_status() == 0


def test_order_assignment_and_tile_do_not_change_bits(sfc):
    # The per-tile K order and its accumulation chains are fixed, so curve vs
    # raster, segment vs wave and every tile shape must give bit-identical
    # results for a fixed number of K layers.
    A, B = synth.gemm_inputs(1000, 1200, 2500, "uniform", seed=5, lda=synth.pad8(2500))
    Ad, Bd = to_dev(A, B)
    for c in (1, 3):
        first = None
        for tile in TILES:
            outs = [sfc.gemm(Ad, Bd, ca_c=c, order=o, assign=a, tile=tile)
                    for o in ("sfc", "raster") for a in ("segment", "wave")]
            for other in outs[1:]:
                assert torch.equal(outs[0], other)
            again = sfc.gemm(Ad, Bd, ca_c=c, order="sfc", assign="segment", tile=tile)
            assert torch.equal(outs[0], again)                 # repeatable
            first = outs[0] if first is None else first
            assert torch.equal(first, outs[0]), tile           # the tile shape does not matter either


def test_k_layers_agree_within_tolerance(sfc, oracle):
    A, B = synth.gemm_inputs(256, 256, 8192, "uniform", seed=9)
    ref = oracle.gemm_f64(A, B)
    for c in (1, 2, 4, 8, 128):
        for tile in TILES:
            check_fp32(run(sfc, A, B, ca_c=c, tile=tile), ref, 8192)


@pytest.mark.parametrize("tile", TILES)
def test_long_k_chains_stay_accurate(sfc, oracle, tile):
    # K = 65536 in one layer: 16 accumulation chains of 4096 per tile, promoted
    # with round-to-nearest fp32 adds; the fp32 tolerance must hold at c = 1.
    A, B = synth.gemm_inputs(256, 384, 65536, "uniform", seed=12)
    ref = oracle.gemm_f64(A, B)
    check_fp32(run(sfc, A, B, ca_c=1, tile=tile), ref, 65536)


def test_unaligned_ldc_uses_scalar_stores(sfc, oracle):
    M, N, K = 300, 260, 320
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=2, ldb=264)
    ref = oracle.gemm_f64(A, B.contiguous())
    Ad, Bd = to_dev(A, B)
    for dt in (torch.float32, torch.bfloat16):
        for c, tile in ((1, 128), (2, 256), (1, "pair128"), (2, "pair256")):
            big = torch.full((M, N + 1), float("nan"), dtype=dt, device="cuda")
            C = big[:, :N]                                     # ldc = N + 1: not 16-byte rows
            sfc.gemm(Ad, Bd, C, ca_c=c, tile=tile)
            torch.cuda.synchronize()
            got = C.float().cpu().numpy().astype(np.float64)
            if dt == torch.float32:
                check_fp32(got, ref, K)
            else:
                check_bf16(got, ref, oracle.round_bf16(ref), K)
            assert torch.isnan(big[:, N]).all()                 # padding column untouched


def test_prefill_distribution(sfc, oracle):
    # activations N(0,1) x weights N(0,0.02): bound scaled by sum_k |A_ik||B_kj|
    M, N, K = 512, 1024, 4096
    A, B = synth.gemm_inputs(M, N, K, "prefill", seed=3)
    ref = oracle.gemm_f64(A, B)
    absA = A.float().abs().to(torch.bfloat16)          # |x| of a bf16 value is exact in bf16
    absB = B.float().abs().to(torch.bfloat16)
    mag = oracle.gemm_f64(absA, absB)
    for c in (1, 4):
        C = run(sfc, A, B, ca_c=c)
        check_fp32(C, ref, K, absbound=2e-6 * mag + 1e-30)


def test_caller_workspace_matches_pool(sfc):
    A, B = synth.gemm_inputs(512, 512, 4096, "uniform", seed=1)
    Ad, Bd = to_dev(A, B)
    need = sfc.workspace_size(512, 512, 4096, 4)
    ws = torch.empty(need // 4, dtype=torch.float32, device="cuda")
    C1 = sfc.gemm(Ad, Bd, ca_c=4)
    C2 = sfc.gemm(Ad, Bd, ca_c=4, workspace=ws)
    assert torch.equal(C1, C2)


def test_error_codes_on_device(sfc):
    from paper_2601_16294_gb300 import binding
    A = torch.zeros(256, 264, dtype=torch.bfloat16, device="cuda")
    B = torch.zeros(256, 256, dtype=torch.bfloat16, device="cuda")
    C = torch.empty(256, 256, dtype=torch.float32, device="cuda")
    with pytest.raises(binding.SfcError) as e:
        binding.gemm_noalloc(A[:, 1:257], B, C)                 # would need repacking: no memory to do it in
    assert e.value.code == binding.SFC_ERR_UNALIGNED
    with pytest.raises(binding.SfcError) as e:
        sfc.gemm(A[:, :256], B, ca_c=5)                         # more layers than K tiles
    assert e.value.code == binding.SFC_ERR_INVALID_ARG
    small = torch.empty(16, dtype=torch.float32, device="cuda")
    with pytest.raises(binding.SfcError) as e:
        sfc.gemm(A[:, :256], B, ca_c=2, workspace=small)
    assert e.value.code == binding.SFC_ERR_WORKSPACE


def test_bounded_wait_reports_timeout_and_context_survives(sfc, oracle):
    from paper_2601_16294_gb300 import binding
    A = torch.zeros(128, 64, dtype=torch.bfloat16, device="cuda")
    B = torch.zeros(64, 128, dtype=torch.bfloat16, device="cuda")
    C = torch.zeros(128, 128, dtype=torch.float32, device="cuda")
    assert sfc.debug_force_timeout(A, B, C, limit_ms=20) == 0
    assert sfc.device_status() == binding.SFC_ERR_TIMEOUT
    assert sfc.device_status() == 0                          # the word was cleared
    # the context is still usable
    A2, B2 = synth.gemm_inputs(256, 256, 256, "int", seed=4)
    ref = oracle.gemm_f64(A2, B2)
    assert np.array_equal(run(sfc, A2, B2), ref)


@pytest.mark.parametrize("M,N,K,off_a,off_b", [(300, 260, 1001, 1, 0), (129, 517, 2500, 0, 3), (256, 256, 130, 5, 7),
                                               (1000, 1200, 2500, 0, 0)])
def test_unaligned_operands_are_repacked(sfc, oracle, M, N, K, off_a, off_b):
    # rows of K and N bf16 values that are not multiples of 8, at bases off by a few elements
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=M + K)
    ref = oracle.gemm_f64(A, B)
    Abuf = torch.zeros(M * K + off_a, dtype=torch.bfloat16, device="cuda")
    Bbuf = torch.zeros(K * N + off_b, dtype=torch.bfloat16, device="cuda")
    Ad = Abuf[off_a:].view(M, K)
    Bd = Bbuf[off_b:].view(K, N)
    Ad.copy_(A)
    Bd.copy_(B)
    for c in (1, 3):
        for tile in ("auto", 128, "pair256"):
            C = sfc.gemm(Ad, Bd, ca_c=c, tile=tile)
            torch.cuda.synchronize()
            assert sfc.device_status() == 0
            check_fp32(C.cpu().numpy().astype(np.float64), ref, K)
    # transposed B with odd rows
    Btbuf = torch.zeros(N * K + off_b, dtype=torch.bfloat16, device="cuda")
    Btd = Btbuf[off_b:].view(N, K)
    Btd.copy_(B.t())
    C = sfc.gemm(Ad, Btd, b_layout="nk")
    check_fp32(C.cpu().numpy().astype(np.float64), ref, K)
