"""The library's choice of tile and K-layer count (ca_c = 0): the chosen call
is the explicit call with those settings, bit for bit, and agrees with the
fp64 oracle within the fp32 tolerance; a caller workspace bounds the choice."""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import check_fp32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


@pytest.mark.parametrize("M,N,K", [(512, 512, 32768), (512, 4096, 4096), (1024, 1024, 16384), (300, 520, 8),
                                   (129, 1000, 4096), (2048, 2048, 2048)])
def test_chosen_layers_equal_explicit_call(sfc, oracle, M, N, K):
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=M + K, lda=synth.pad8(K), ldb=synth.pad8(N))
    Ad = torch.empty(M, synth.pad8(K), dtype=torch.bfloat16, device="cuda")[:, :K]
    Ad.copy_(A)
    Bd = torch.empty(K, synth.pad8(N), dtype=torch.bfloat16, device="cuda")[:, :N]
    Bd.copy_(B)
    tile, c = sfc.plan(M, N, K, 0)
    assert 1 <= c <= max(1, sfc.workspace_size(M, N, K, 0) // (M * ((N + 3) // 4 * 4) * 4))
    assert sfc.plan(M, N, K, c)[1] == c
    C0 = sfc.gemm(Ad, Bd, ca_c=0)
    C1 = sfc.gemm(Ad, Bd, ca_c=c, tile=tile)
    torch.cuda.synchronize()
    assert sfc.device_status() == 0
    assert torch.equal(C0, C1)
    check_fp32(C0.cpu().numpy().astype(np.float64), oracle.gemm_f64(A.contiguous(), B.contiguous()), K)


def test_choices_follow_the_shape(sfc):
    # many tiles: one layer; few tiles and long K: several
    assert sfc.plan(16384, 16384, 16384, 0)[1] == 1
    assert sfc.plan(8192, 8192, 8192, 0)[1] == 1
    assert sfc.plan(512, 512, 131072, 0)[1] >= 8
    assert sfc.plan(1024, 1024, 65536, 0)[1] >= 2
    assert sfc.plan(2048, 2048, 2048, 0)[1] == 1
    # an explicit count is kept
    assert sfc.plan(512, 512, 131072, 3)[1] == 3


def test_caller_workspace_bounds_the_choice(sfc, oracle):
    M, N, K = 512, 512, 32768
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=7)
    Ad, Bd = A.cuda(), B.cuda()
    per_layer = M * N * 4
    ws = torch.empty(2 * per_layer // 4, dtype=torch.float32, device="cuda")   # room for 2 layers
    C = sfc.gemm(Ad, Bd, ca_c=0, workspace=ws)
    C2 = sfc.gemm(Ad, Bd, ca_c=2, workspace=ws)
    torch.cuda.synchronize()
    assert sfc.device_status() == 0
    assert torch.equal(C, C2)                 # at most 2 layers fit; 2 beats 1 here
    check_fp32(C.cpu().numpy().astype(np.float64), oracle.gemm_f64(A, B), K)


def test_release_after_pooled_workspace(sfc):
    A = torch.ones(256, 4096, dtype=torch.bfloat16, device="cuda")
    B = torch.ones(4096, 256, dtype=torch.bfloat16, device="cuda")
    C = sfc.gemm(A, B, ca_c=4)
    sfc.release()
    assert torch.equal(C, torch.full_like(C, 4096.0))
    C2 = sfc.gemm(A, B, ca_c=4)                  # the pool is usable again after trimming
    assert torch.equal(C, C2)
