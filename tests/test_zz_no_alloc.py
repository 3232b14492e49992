"""The allocation-free entry point, sfc_gemm_noalloc, through the C ABI.

sfc_gemm_noalloc serves callers that cannot allocate device memory themselves:
code inside a framework that owns every device allocation, or a
latency-critical path where an allocation may block or fail.  Its K-layer
partials and its workers' item counter live in a scratch area built into the
library.  These tests check that:
  - two calls in a row (the second sees the scratch area as the first left
    it) give exactly the bits of the ordinary entry point sfc_gemm_ex with the
    same plan;
  - on integer inputs, where fp32 sums are exact in any order, the result
    equals the oracle bit for bit, for one layer, several, and the library's
    own count (ca_c = 0);
  - partials of exactly the scratch size are accepted and one layer more is
    refused with SFC_ERR_WORKSPACE, launching nothing;
  - the calls take nothing from the library's stream-ordered pools.
The file sorts last, so a run that stops at the first failure has already run
every other test; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth

pytestmark = pytest.mark.gpu

SCRATCH = 32 << 20  # SFC_NOALLOC_SCRATCH_BYTES


@pytest.fixture(scope="module")
def lib():
    from paper_2601_16294_gb300 import binding, build_lib
    build_lib.build()
    lib = binding.load()
    assert binding.NOALLOC_SCRATCH_BYTES == SCRATCH
    return lib


def _stream():
    return ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)


def _noalloc(lib, A, B, C, ca_c):
    M, K = A.shape
    N = B.shape[1]
    dtype = 0 if C.dtype == torch.float32 else 1
    return lib.sfc_gemm_noalloc(M, N, K, ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(B.data_ptr()),
                                ctypes.c_void_p(C.data_ptr()), A.stride(0), B.stride(0), C.stride(0), ca_c, dtype,
                                _stream())


def _existing(lib, A, B, C, ca_c, workspace=None):
    """sfc_gemm_ex with the same order, dealing and tile choice (SFC, AUTO, AUTO)."""
    M, K = A.shape
    N = B.shape[1]
    dtype = 0 if C.dtype == torch.float32 else 1
    ws = ctypes.c_void_p(workspace.data_ptr()) if workspace is not None else None
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    return lib.sfc_gemm_ex(M, N, K, ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(B.data_ptr()),
                           ctypes.c_void_p(C.data_ptr()), A.stride(0), B.stride(0), C.stride(0), ca_c, dtype,
                           0, 2, 0, ws, ws_bytes, _stream())


def _bits(t):
    return t.view(torch.int32 if t.dtype == torch.float32 else torch.int16).cpu()


def _pool_used_high(lib, reset):
    v = ctypes.c_size_t(0)
    assert lib.sfc_debug_pool_used_high(ctypes.byref(v), 1 if reset else 0) == 0
    return v.value


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_noalloc_matches_existing_entry_point_twice(lib, out_dtype):
    # several tiles, ragged M / N / K tails; the two calls run back to back
    cases = [(512, 512, 4096, 4, 21), (384, 640, 2048, 8, 22), (300, 200, 1000, 1, 23)]
    for M, N, K, c, seed in cases:
        A, B = synth.gemm_inputs(M, N, K, "uniform", seed=seed)
        A, B = A.cuda(), B.cuda()
        want = torch.empty((M, N), dtype=out_dtype, device="cuda")
        assert _existing(lib, A, B, want, c) == 0
        got = []
        for _ in range(2):
            g = torch.full((M, N), float("nan"), dtype=out_dtype, device="cuda")
            assert _noalloc(lib, A, B, g, c) == 0
            got.append(g)
        torch.cuda.synchronize()
        assert lib.sfc_get_device_status(None) == 0
        for g in got:
            assert torch.equal(_bits(g), _bits(want)), "noalloc result differs from sfc_gemm_ex (%dx%dx%d, c=%d)" % (
                M, N, K, c)


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
@pytest.mark.parametrize("ca_c", [0, 1, 2, 8])
def test_noalloc_integer_inputs_bit_exact_against_oracle(lib, oracle, out_dtype, ca_c):
    M, N, K = 640, 768, 3000
    A, B = synth.gemm_inputs(M, N, K, "int", seed=31)
    ref = oracle.gemm_f64(A, B)  # integers below 2^24: exact in fp32 in any summation order
    if out_dtype == torch.bfloat16:
        ref = oracle.round_bf16(ref)
    C = torch.full((M, N), float("nan"), dtype=out_dtype, device="cuda")
    assert _noalloc(lib, A.cuda(), B.cuda(), C, ca_c) == 0
    torch.cuda.synchronize()
    assert lib.sfc_get_device_status(None) == 0
    assert np.array_equal(C.double().cpu().numpy(), ref)


def test_noalloc_partials_exactly_at_the_scratch_size_and_one_layer_past(lib, oracle):
    M = N = K = 1024
    assert 8 * M * N * 4 == SCRATCH
    A, B = synth.gemm_inputs(M, N, K, "int", seed=41)
    ref = oracle.gemm_f64(A, B)
    Ad, Bd = A.cuda(), B.cuda()
    C = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    assert lib.sfc_gemm_workspace_size(M, N, K, 8) == SCRATCH
    assert _noalloc(lib, Ad, Bd, C, 8) == 0
    torch.cuda.synchronize()
    assert lib.sfc_get_device_status(None) == 0
    assert np.array_equal(C.double().cpu().numpy(), ref)
    # nine layers need one layer's partials more than the scratch holds: refused, nothing written
    C2 = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    from paper_2601_16294_gb300 import binding
    assert lib.sfc_gemm_workspace_size(M, N, K, 9) > SCRATCH
    assert _noalloc(lib, Ad, Bd, C2, 9) == binding.SFC_ERR_WORKSPACE
    torch.cuda.synchronize()
    assert torch.isnan(C2).all().item()


def test_noalloc_library_layer_count_fits_the_scratch(lib, oracle):
    # the library's unconstrained choice for this shape may take 2 layers (35.7 MB of partials);
    # ca_c = 0 then uses what fits, exactly as sfc_gemm_ex does with a caller workspace of that size
    M, N, K = 2048, 2176, 512
    assert lib.sfc_gemm_workspace_size(M, N, K, 0) > SCRATCH
    A, B = synth.gemm_inputs(M, N, K, "int", seed=51)
    Ad, Bd = A.cuda(), B.cuda()
    want = torch.empty((M, N), dtype=torch.float32, device="cuda")
    ws = torch.empty(SCRATCH, dtype=torch.uint8, device="cuda")
    assert _existing(lib, Ad, Bd, want, 0, workspace=ws) == 0
    got = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
    assert _noalloc(lib, Ad, Bd, got, 0) == 0
    torch.cuda.synchronize()
    assert lib.sfc_get_device_status(None) == 0
    assert torch.equal(_bits(got), _bits(want))
    assert np.array_equal(got.double().cpu().numpy(), oracle.gemm_f64(A, B))


def test_noalloc_takes_nothing_from_the_pools(lib):
    M, N, K = 512, 512, 8192
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=61)
    Ad, Bd = A.cuda(), B.cuda()
    C = torch.empty((M, N), dtype=torch.float32, device="cuda")
    # the ordinary entry point with 4 layers takes its workspace and counter from the pools
    assert _existing(lib, Ad, Bd, C, 4) == 0
    torch.cuda.synchronize()
    _pool_used_high(lib, reset=True)
    assert _pool_used_high(lib, reset=False) == 0
    for c in (0, 1, 4, 4):
        assert _noalloc(lib, Ad, Bd, C, c) == 0
    torch.cuda.synchronize()
    assert lib.sfc_get_device_status(None) == 0
    assert _pool_used_high(lib, reset=False) == 0
    # the mark does move for the ordinary entry point (the check above can fail)
    assert _existing(lib, Ad, Bd, C, 4) == 0
    torch.cuda.synchronize()
    assert _pool_used_high(lib, reset=False) >= 4 * M * N * 4


def test_noalloc_rejects_partials_larger_than_its_scratch(lib):
    from paper_2601_16294_gb300 import binding
    A = torch.zeros(2048, 4096, dtype=torch.bfloat16, device="cuda")
    B = torch.zeros(4096, 2048, dtype=torch.bfloat16, device="cuda")
    C = torch.zeros(2048, 2048, dtype=torch.float32, device="cuda")
    assert lib.sfc_gemm_workspace_size(2048, 2048, 4096, 8) > binding.NOALLOC_SCRATCH_BYTES
    assert _noalloc(lib, A, B, C, 8) == binding.SFC_ERR_WORKSPACE
