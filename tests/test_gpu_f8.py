"""8-bit float inputs (sfc_gemm_ex2 with SFC_AB_E4M3 / SFC_AB_E5M2) against the
oracle's exact decoding of the same bytes.  Integer-valued data makes every
product and sum exact, so those cases are compared bit for bit; uniform data
uses the fp32 tolerance of the bf16 path."""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import check_bf16, check_fp32

pytestmark = pytest.mark.gpu

FORMATS = ["e4m3", "e5m2"]
TILES = [128, 256, "pair128", "pair256"]


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def pad16(n):
    return (n + 15) // 16 * 16


def dev(t, ld):
    """CUDA copy of a CPU 8-bit matrix with row stride ld (zero padding)."""
    d = torch.zeros(t.shape[0], ld, dtype=t.dtype, device="cuda")
    d[:, : t.shape[1]] = t.cuda()
    return d[:, : t.shape[1]]


def operands(A, B, layout):
    K = A.shape[1]
    if layout == "kn":
        return dev(A, pad16(K)), dev(B, pad16(B.shape[1])), B
    Bt = B.t().contiguous()
    return dev(A, pad16(K)), dev(Bt, pad16(K)), Bt


@pytest.mark.parametrize("fmt", FORMATS)
@pytest.mark.parametrize("layout", ["kn", "nk"])
def test_integer_inputs_bit_exact(sfc, oracle, fmt, layout):
    M, N, K = 384, 640, 1000
    A, B = synth.gemm_inputs_f8(M, N, K, fmt, "int", seed=41)
    Ad, Bd, Bh = operands(A, B, layout)
    ref = oracle.gemm_f8_f64(A, Bh, fmt, b_layout=layout)
    for tile in TILES:
        for c in (1, 2, 3):
            for order in ("sfc", "raster"):
                C = sfc.gemm(Ad, Bd, b_layout=layout, ca_c=c, tile=tile, order=order)
                torch.cuda.synchronize()
                assert sfc.device_status() == 0
                assert np.array_equal(C.cpu().numpy().astype(np.float64), ref), (tile, c, order)


@pytest.mark.parametrize("M,N,K", [(200, 300, 136), (129, 257, 1000), (7, 9, 16), (640, 136, 2048), (512, 512, 8192)])
@pytest.mark.parametrize("fmt", FORMATS)
def test_uniform_inputs(sfc, oracle, M, N, K, fmt):
    A, B = synth.gemm_inputs_f8(M, N, K, fmt, "uniform", seed=M + N + K)
    for layout in ("kn", "nk"):
        Ad, Bd, Bh = operands(A, B, layout)
        ref = oracle.gemm_f8_f64(A, Bh, fmt, b_layout=layout)
        ref16 = oracle.round_bf16(ref)
        for tile in ("auto", 128, "pair256"):
            for c in (1, 2):
                if c > (K + 127) // 128:
                    continue
                C = sfc.gemm(Ad, Bd, b_layout=layout, ca_c=c, tile=tile)
                Cb = sfc.gemm(Ad, Bd, b_layout=layout, ca_c=c, tile=tile, out_dtype=torch.bfloat16)
                torch.cuda.synchronize()
                assert sfc.device_status() == 0
                check_fp32(C.cpu().numpy().astype(np.float64), ref, K)
                check_bf16(Cb.float().cpu().numpy().astype(np.float64), ref, ref16, K)


def test_long_k_chains(sfc, oracle):
    # K = 65536 in one layer: 8 accumulation chains of 8192 values of k per tile
    A, B = synth.gemm_inputs_f8(256, 384, 65536, "e4m3", "uniform", seed=12)
    ref = oracle.gemm_f8_f64(A, B, "e4m3")
    for tile in ("pair256", 256):
        C = sfc.gemm(A.cuda(), B.cuda(), ca_c=1, tile=tile)
        torch.cuda.synchronize()
        check_fp32(C.cpu().numpy().astype(np.float64), ref, 65536)


def test_order_assignment_and_layout_do_not_change_bits(sfc):
    A, B = synth.gemm_inputs_f8(1000, 1200, 2560, "e4m3", "uniform", seed=5)
    Ad, Bd = dev(A, 2560), B.cuda()
    Btd = dev(B.t().contiguous(), 2560)
    for c in (1, 3):
        outs = [sfc.gemm(Ad, Bd, ca_c=c, tile="pair256", order=o, assign=a)
                for o in ("sfc", "raster") for a in ("segment", "wave")]
        outs.append(sfc.gemm(Ad, Btd, b_layout="nk", ca_c=c, tile="pair256"))
        for other in outs[1:]:
            assert torch.equal(outs[0], other)


def test_layer_count_choice_and_beta_bias(sfc, oracle):
    M, N, K = 512, 512, 32768
    A, B = synth.gemm_inputs_f8(M, N, K, "e4m3", "int", seed=9)
    tile, c = sfc.plan(M, N, K, 0, in_dtype=A.dtype)
    assert c >= 2
    bias = torch.arange(N, dtype=torch.float32) - 100.0
    C_in = torch.ones(M, N, dtype=torch.float32) * 3.0
    ref = oracle.gemm_f8_f64(A, B, "e4m3") + 0.5 * 3.0 + bias.numpy()
    C = C_in.cuda()
    sfc.gemm(A.cuda(), B.cuda(), C, ca_c=0, beta=0.5, bias=bias.cuda())
    torch.cuda.synchronize()
    assert np.array_equal(C.cpu().numpy().astype(np.float64), ref)


def test_unaligned_rows_are_repacked(sfc, oracle):
    # 8-bit rows of 1000 and 300 values (not multiples of 16 bytes) go through the repacking copy
    M, N, K = 200, 300, 1000
    A, B = synth.gemm_inputs_f8(M, N, K, "e4m3", "int", seed=77)
    ref = oracle.gemm_f8_f64(A, B, "e4m3")
    C = sfc.gemm(A.cuda(), B.cuda(), ca_c=2)
    torch.cuda.synchronize()
    assert sfc.device_status() == 0
    assert np.array_equal(C.cpu().numpy().astype(np.float64), ref)
