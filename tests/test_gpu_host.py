"""The host-buffer entry point (sfc_gemm_host): operands and result in host
memory, copies pipelined against the GEMM along a staircase of row panels of
A and column panels of B.

Each strip of C is a GEMM over whole output tiles with the plan of the full
problem, so the result must equal sfc_gemm_ex2 on device copies (same tile,
same layer count) bit for bit, for every panel count; integer-valued inputs
must equal the oracle exactly.
"""
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


def host(t, ld=None, pinned=True):
    """Host copy of a CPU matrix with row stride ld (pinned unless asked)."""
    ld = ld or t.shape[1]
    big = torch.zeros((t.shape[0], ld), dtype=t.dtype, pin_memory=pinned)
    big[:, : t.shape[1]] = t
    return big[:, : t.shape[1]]


def device(t):
    """CUDA copy with 16-byte rows."""
    align = 16 // t.element_size()
    ld = (t.shape[1] + align - 1) // align * align
    d = torch.zeros((t.shape[0], ld), dtype=t.dtype, device="cuda")
    d[:, : t.shape[1]] = t.cuda()
    return d[:, : t.shape[1]]


def on_device(sfc, A, B, *, b_layout="kn", out_dtype=torch.float32, ca_c=0, tile="auto"):
    M, K = A.shape
    N = B.shape[1] if b_layout == "kn" else B.shape[0]
    t, c = sfc.plan(M, N, K, ca_c=ca_c, out_dtype=out_dtype, tile=tile, in_dtype=A.dtype, b_layout=b_layout)
    C = sfc.gemm(device(A), device(B), ca_c=c, tile=t, out_dtype=out_dtype, b_layout=b_layout)
    return C.cpu()


CASES = [
    # M, N, K, lda, ldb: odd K rows on the host
    (1000, 1200, 2500, 2501, 1203),
    # K not a multiple of 64, padded host rows, more row than column panels
    (3000, 700, 1001, 1001, 705),
    # several 512-row units, aligned rows (one-piece copies), one column panel
    (2600, 512, 640, 640, 512),
    # several column panels of 256 columns, one row panel
    (300, 2900, 320, 320, 2900),
    # one tile
    (100, 60, 40, 40, 60),
]


@pytest.mark.parametrize("M,N,K,lda,ldb", CASES)
@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_matches_device_call_bit_exact(sfc, M, N, K, lda, ldb, out_dtype):
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=M + N)
    A, B = A.contiguous(), B.contiguous()
    ref = on_device(sfc, A, B, out_dtype=out_dtype)
    Ah, Bh = host(A, lda), host(B, ldb)
    for panels in (0, 1, 3, 1000):
        C = sfc.matmul_host(Ah, Bh, out_dtype=out_dtype, panels=panels)
        assert torch.equal(C, ref), panels
    assert sfc.device_status() == 0


def test_layers_and_tiles(sfc):
    A, B = synth.gemm_inputs(1536, 900, 3000, "uniform", seed=3)
    Ah, Bh = host(A), host(B)
    for ca_c, tile in ((3, "auto"), (1, 128), (2, "pair128"), (1, "pair256"), (4, 256)):
        ref = on_device(sfc, A, B, ca_c=ca_c, tile=tile)
        C = sfc.matmul_host(Ah, Bh, ca_c=ca_c, tile=tile, panels=3)
        assert torch.equal(C, ref), (ca_c, tile)


def test_transposed_b_column_slices(sfc, oracle):
    M, N, K = 300, 2000, 640
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=8)
    Bt = B.t().contiguous()
    ref = on_device(sfc, A, Bt, b_layout="nk")
    C = sfc.matmul_host(host(A), host(Bt, 648), b_layout="nk", panels=4)
    assert torch.equal(C, ref)
    check_fp32(C.numpy().astype(np.float64), oracle.gemm_f64(A, B), K)


def test_integer_inputs_equal_the_oracle(sfc, oracle):
    M, N, K = 2100, 1000, 1536
    A, B = synth.gemm_inputs(M, N, K, "int", seed=21)
    ref = oracle.gemm_f64(A, B)
    for panels in (0, 2, 5):
        C = sfc.matmul_host(host(A), host(B), ca_c=2, panels=panels)
        assert np.array_equal(C.numpy().astype(np.float64), ref), panels
        Cb = sfc.matmul_host(host(A), host(B), out_dtype=torch.bfloat16, panels=panels)
        assert np.array_equal(Cb.view(torch.int16).numpy().view(np.uint16), oracle.round_bf16_bits(ref))


@pytest.mark.parametrize("fmt", ["e4m3", "e5m2"])
def test_fp8_inputs(sfc, fmt):
    A, B = synth.gemm_inputs_f8(1100, 900, 512, fmt, "uniform", seed=5)
    ref = on_device(sfc, A, B)
    C = sfc.matmul_host(host(A, 515), host(B, 903), panels=3)
    assert torch.equal(C, ref)


def test_calls_in_flight_overlap_and_stay_correct(sfc):
    # several calls enqueued back to back, one synchronisation at the end:
    # each takes its own staging slot.  The host operands are read after the
    # calls return, so they are kept alive (and unchanged) until the stream
    # has synchronised.
    shapes = [(2048, 2048, 1024), (700, 3000, 512), (4096, 1024, 2048), (512, 512, 4096)]
    jobs = []
    s = torch.cuda.current_stream()
    for i, (M, N, K) in enumerate(shapes):
        A, B = synth.gemm_inputs(M, N, K, "uniform", seed=40 + i)
        A, B = A.contiguous(), B.contiguous()
        Ch = torch.full((M, N), float("nan"), dtype=torch.bfloat16, pin_memory=True)
        jobs.append((A, B, host(A), host(B), Ch, on_device(sfc, A, B, out_dtype=torch.bfloat16)))
    for _, _, Ah, Bh, Ch, _ in jobs:
        sfc.gemm_host(Ah, Bh, Ch, stream=s)
    s.synchronize()
    for _, _, _, _, Ch, ref in jobs:
        assert torch.equal(Ch, ref)
    # the same slots serve the next round of calls
    for _, _, Ah, Bh, Ch, _ in jobs:
        Ch.fill_(float("nan"))
        sfc.gemm_host(Ah, Bh, Ch, stream=s)
    s.synchronize()
    for _, _, _, _, Ch, ref in jobs:
        assert torch.equal(Ch, ref)
    sfc.release()
    _, _, Ah, Bh, _, ref = jobs[0]
    assert torch.equal(sfc.matmul_host(Ah, Bh, out_dtype=torch.bfloat16), ref)


def test_pageable_memory_and_padded_c(sfc):
    M, N, K = 1300, 770, 900
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=6)
    A, B = A.contiguous(), B.contiguous()
    ref = on_device(sfc, A, B)
    big = torch.full((M, N + 3), float("nan"), dtype=torch.float32)        # pageable, ldc = N + 3
    C = big[:, :N]
    sfc.matmul_host(host(A, pinned=False), host(B, pinned=False), C, panels=2)
    assert torch.equal(C, ref)
    assert torch.isnan(big[:, N:]).all()                                   # padding untouched
