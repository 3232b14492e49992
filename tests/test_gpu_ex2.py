"""The BLAS-style extension (sfc_gemm_ex2): B stored transposed (N x K, read
K-major by the kernels) and the epilogue C = A B + beta * C_in + bias, against
the oracle's independent affine GEMM.  Integer data makes every fp32 step
exact, so those cases are compared bit for bit."""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import check_bf16, check_fp32

pytestmark = pytest.mark.gpu

TILES = [128, 256, "pair128", "pair256"]


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def padded(t, ld):
    """CUDA copy of a CPU matrix with row stride ld."""
    d = torch.zeros(t.shape[0], ld, dtype=t.dtype, device="cuda")
    d[:, : t.shape[1]] = t.cuda()
    return d[:, : t.shape[1]]


@pytest.mark.parametrize("tile", TILES)
def test_transposed_b_integer_exact(sfc, oracle, tile):
    M, N, K = 384, 640, 1000
    A, B = synth.gemm_inputs(M, N, K, "int", seed=31)
    Bt = B.t().contiguous()
    ref = oracle.gemm_affine_f64(A, Bt, b_layout="nk")
    Ad, Btd = padded(A, synth.pad8(K)), padded(Bt, synth.pad8(K))
    for c in (1, 2, 3):
        for order in ("sfc", "raster"):
            C = sfc.gemm(Ad, Btd, b_layout="nk", ca_c=c, order=order, tile=tile)
            torch.cuda.synchronize()
            assert sfc.device_status() == 0
            assert np.array_equal(C.cpu().numpy().astype(np.float64), ref), (c, order)


@pytest.mark.parametrize("M,N,K", [(200, 300, 136), (129, 257, 1000), (7, 9, 64), (640, 136, 2048), (512, 512, 4096)])
@pytest.mark.parametrize("tile", ["auto", 128, "pair256"])
def test_transposed_b_uniform(sfc, oracle, M, N, K, tile):
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=M + 3 * N + K)
    Bt = B.t().contiguous()
    ref = oracle.gemm_affine_f64(A, Bt, b_layout="nk")
    ref16 = oracle.round_bf16(ref)
    Ad, Btd = padded(A, synth.pad8(K)), padded(Bt, synth.pad8(K))
    for c in (1, 2):
        if c > (K + 63) // 64:
            continue
        C = sfc.gemm(Ad, Btd, b_layout="nk", ca_c=c, tile=tile)
        Cb = sfc.gemm(Ad, Btd, b_layout="nk", ca_c=c, tile=tile, out_dtype=torch.bfloat16)
        torch.cuda.synchronize()
        assert sfc.device_status() == 0
        check_fp32(C.cpu().numpy().astype(np.float64), ref, K)
        check_bf16(Cb.float().cpu().numpy().astype(np.float64), ref, ref16, K)


def test_transposed_b_equals_row_major_b(sfc):
    # the same B in either storage gives the same bits (same products, same sums)
    A, B = synth.gemm_inputs(1000, 1200, 2500, "uniform", seed=5)
    Ad, Bd, Btd = padded(A, 2504), B.cuda(), padded(B.t().contiguous(), 2504)
    for c in (1, 3):
        for tile in ("auto", 256, "pair256"):
            assert torch.equal(sfc.gemm(Ad, Bd, ca_c=c, tile=tile),
                               sfc.gemm(Ad, Btd, b_layout="nk", ca_c=c, tile=tile)), (c, tile)


@pytest.mark.parametrize("out", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("layout", ["kn", "nk"])
def test_beta_and_bias_integer_exact(sfc, oracle, out, layout):
    M, N, K = 300, 520, 704
    A, B = synth.gemm_inputs(M, N, K, "int", seed=17)
    g = np.random.default_rng(2)
    C_in = g.integers(-60, 60, size=(M, N)).astype(np.float32)
    bias = g.integers(-20, 20, size=N).astype(np.float32)
    Bl = B if layout == "kn" else B.t().contiguous()
    ref = oracle.gemm_affine_f64(A, Bl, b_layout=layout, beta=-2.0, C_in=C_in, bias=bias)
    Ad = A.cuda()
    Bd = Bl.cuda()
    bias_d = torch.from_numpy(bias).cuda()
    for c in (1, 2, 5):
        for tile in TILES:
            C = torch.from_numpy(C_in).to(out).cuda()
            sfc.gemm(Ad, Bd, C, b_layout=layout, beta=-2.0, bias=bias_d, ca_c=c, tile=tile)
            torch.cuda.synchronize()
            assert sfc.device_status() == 0
            got = C.float().cpu().numpy().astype(np.float64)
            want = ref if out == torch.float32 else oracle.round_bf16(ref)
            assert np.array_equal(got, want), (c, tile)


def test_beta_and_bias_uniform(sfc, oracle):
    M, N, K = 520, 390, 2000
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=8)
    C_in = synth.uniform_bf16((M, N), seed=9).float().numpy()
    bias = synth.uniform_bf16((N,), seed=10).float().numpy()
    ref = oracle.gemm_affine_f64(A, B, beta=0.75, C_in=C_in, bias=bias)
    for c in (1, 4):
        C = torch.from_numpy(C_in).cuda()
        sfc.gemm(padded(A, 2000), padded(B, 392), C, beta=0.75, bias=torch.from_numpy(bias).cuda(), ca_c=c)
        torch.cuda.synchronize()
        check_fp32(C.cpu().numpy().astype(np.float64), ref, K)


def test_beta_zero_never_reads_c(sfc, oracle):
    A, B = synth.gemm_inputs(256, 256, 512, "int", seed=3)
    ref = oracle.gemm_affine_f64(A, B)
    for c in (1, 2):
        C = torch.full((256, 256), float("nan"), dtype=torch.float32, device="cuda")
        sfc.gemm(A.cuda(), B.cuda(), C, beta=0.0, ca_c=c)
        torch.cuda.synchronize()
        assert np.array_equal(C.cpu().numpy().astype(np.float64), ref)


@pytest.mark.parametrize("tile", ["auto", 128, "pair256"])
def test_accumulate_into_c(sfc, oracle, tile):
    # C += A B (beta = 1, no bias, fp32 C with 16-byte rows) adds in L2 instead of
    # reading C; it must equal the path that reads C (rows the TMA cannot store)
    # bit for bit, and the oracle exactly on integer data.
    M, N, K = 520, 392, 2000
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=81)
    C_in = synth.uniform_bf16((M, N), seed=82).float()
    Ad, Bd = padded(A, 2000), padded(B, 392)
    C = C_in.cuda()
    sfc.gemm(Ad, Bd, C, beta=1.0, tile=tile)
    big = torch.zeros(M, N + 1, dtype=torch.float32, device="cuda")
    Cr = big[:, :N]
    Cr.copy_(C_in)
    sfc.gemm(Ad, Bd, Cr, beta=1.0, tile=tile)                   # ldc = N + 1: read, add, store
    assert torch.equal(C, Cr)
    check_fp32(C.cpu().numpy().astype(np.float64),
               oracle.gemm_affine_f64(A, B, beta=1.0, C_in=C_in.numpy()), K)
    Ai, Bi = synth.gemm_inputs(M, N, K, "int", seed=83)
    Ci = torch.randint(-8, 9, (M, N), dtype=torch.float32)
    ref = oracle.gemm_affine_f64(Ai, Bi, beta=1.0, C_in=Ci.numpy())
    C = Ci.cuda()
    sfc.gemm(padded(Ai, 2000), padded(Bi, 392), C, beta=1.0, tile=tile)
    assert np.array_equal(C.cpu().numpy().astype(np.float64), ref)
