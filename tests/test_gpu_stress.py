"""Pipeline edges and failure paths.

The ring has 4, 6 or 8 stages depending on the tile shape; K-slab counts
around those depths (1, 2, stages - 1, stages, stages + 1, odd counts) with
M and N tails of one row / column exercise the producer's and the MMA
issuer's wrap-around, on integer data so the result must equal the oracle bit
for bit.  A workspace allocation that cannot succeed must come back as
SFC_ERR_CUDA with the CUDA error code, and leave the context usable.  Views
of one buffer with changing shapes and strides check that reused tensor maps
never stand in for a different operand."""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth

pytestmark = pytest.mark.gpu

TILES = [128, 256, "pair128", "pair256"]
SLABS = [1, 2, 3, 4, 5, 6, 7, 8, 9, 13, 17]


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


@pytest.mark.parametrize("tile", TILES)
def test_slab_counts_around_the_ring_depth(sfc, oracle, tile):
    for i, kt in enumerate(SLABS):
        M, N, K = 513, 257, 64 * kt - (i % 3) * 7          # tails of one row and column; ragged last slab
        A, B = synth.gemm_inputs(M, N, K, "int", seed=900 + i)
        ref = oracle.gemm_f64(A, B)
        Kp, Np = (K + 7) // 8 * 8, (N + 7) // 8 * 8
        Ad = torch.zeros(M, Kp, dtype=torch.bfloat16, device="cuda")
        Ad[:, :K] = A.cuda()
        Bd = torch.zeros(K, Np, dtype=torch.bfloat16, device="cuda")
        Bd[:, :N] = B.cuda()
        for c in sorted({1, min(2, kt)}):
            C = sfc.gemm(Ad[:, :K], Bd[:, :N], ca_c=c, tile=tile)
            torch.cuda.synchronize()
            assert np.array_equal(C.cpu().numpy().astype(np.float64), ref), (tile, kt, c)
    assert sfc.device_status() == 0


def test_workspace_allocation_failure_is_reported(sfc, oracle):
    from paper_2601_16294_gb300 import binding
    # 128 fp32 layer copies of a 32768 x 32768 C would need 550 GB
    M = N = 32768
    K = 128 * 64
    A = torch.zeros(M, K, dtype=torch.bfloat16, device="cuda")
    B = torch.zeros(K, N, dtype=torch.bfloat16, device="cuda")
    C = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(binding.SfcError) as e:
        sfc.gemm(A, B, C, ca_c=128)
    assert e.value.code == binding.SFC_ERR_CUDA
    assert e.value.cuda_error == 2                                   # cudaErrorMemoryAllocation
    del A, B, C
    torch.cuda.empty_cache()
    # nothing sticky: the next call works
    A2, B2 = synth.gemm_inputs(300, 200, 500, "int", seed=9)
    C2 = sfc.gemm(A2.cuda(), B2.cuda(), ca_c=2)                      # rows of A repacked (K = 500)
    assert np.array_equal(C2.cpu().numpy().astype(np.float64), oracle.gemm_f64(A2, B2))
    assert sfc.device_status() == 0


def test_operands_reshaped_at_one_address(sfc, oracle):
    # encoded tensor maps are reused for repeated operands: views of the same
    # buffers with other shapes and row strides, at the same addresses, must
    # still be read and written as given
    bufA = torch.zeros(300 * 520, dtype=torch.bfloat16, device="cuda")
    bufB = torch.zeros(520 * 300, dtype=torch.bfloat16, device="cuda")
    bufC = torch.zeros(300 * 300, dtype=torch.float32, device="cuda")
    shapes = [(300, 260, 520, 520, 264), (256, 300, 500, 504, 304), (300, 260, 520, 520, 264), (130, 77, 64, 64, 80)]
    for i, (M, N, K, lda, ldb) in enumerate(shapes * 2):
        A, B = synth.gemm_inputs(M, N, K, "int", seed=700 + i)
        Av = bufA[: M * lda].view(M, lda)[:, :K]
        Av.copy_(A.cuda())
        Bv = bufB[: K * ldb].view(K, ldb)[:, :N]
        Bv.copy_(B.cuda())
        Cv = bufC[: M * N].view(M, N)
        ref = oracle.gemm_f64(A, B)
        for c in [c for c in (1, 2) if c <= (K + 63) // 64]:
            Cv.fill_(-1.0)
            sfc.gemm(Av, Bv, Cv, ca_c=c)
            torch.cuda.synchronize()
            assert np.array_equal(Cv.cpu().numpy().astype(np.float64), ref), (M, N, K, c)
    assert sfc.device_status() == 0
