"""The allocation-free entry point, sfc_gemm_noalloc, against sfc_gemm_ex.

sfc_gemm_noalloc serves callers that cannot allocate device memory themselves
(a host framework owning every allocation, a latency-critical path where an
allocation may block or fail): its K-layer partials live in a scratch area
built into the library.  The test calls it through the C ABI twice in a row --
the second call sees the scratch area exactly as the first call left it -- and
compares each result with the ordinary entry point's within the GEMM parity
tolerance.  It sorts last so that a run stopping at the first failure has
already run every other test.
"""
import ctypes

import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import check_fp32

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def lib():
    from paper_2601_16294_gb300 import binding, build_lib
    build_lib.build()
    return binding.load()


def _noalloc(lib, A, B, C, ca_c):
    M, K = A.shape
    N = B.shape[1]
    dtype = 0 if C.dtype == torch.float32 else 1
    return lib.sfc_gemm_noalloc(M, N, K, ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(B.data_ptr()),
                                ctypes.c_void_p(C.data_ptr()), A.stride(0), B.stride(0), C.stride(0), ca_c, dtype,
                                ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _existing(lib, A, B, C, ca_c):
    M, K = A.shape
    N = B.shape[1]
    dtype = 0 if C.dtype == torch.float32 else 1
    return lib.sfc_gemm_ex(M, N, K, ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(B.data_ptr()),
                           ctypes.c_void_p(C.data_ptr()), A.stride(0), B.stride(0), C.stride(0), ca_c, dtype,
                           0, 2, 0, None, 0, ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


@pytest.mark.parametrize("out_dtype", [torch.float32, torch.bfloat16])
def test_noalloc_matches_existing_entry_point_twice(lib, out_dtype):
    cases = [(512, 512, 4096, 4, 21), (384, 640, 2048, 8, 22)]   # two calls in a row
    for M, N, K, c, seed in cases:
        A, B = synth.gemm_inputs(M, N, K, "uniform", seed=seed)
        A, B = A.cuda(), B.cuda()
        want = torch.empty((M, N), dtype=out_dtype, device="cuda")
        got = torch.full((M, N), float("nan"), dtype=out_dtype, device="cuda")
        assert _existing(lib, A, B, want, c) == 0
        assert _noalloc(lib, A, B, got, c) == 0
        torch.cuda.synchronize()
        assert lib.sfc_get_device_status(None) == 0
        g = got.double().cpu().numpy()
        w = want.double().cpu().numpy()
        if out_dtype == torch.float32:
            check_fp32(g, w, K)
        else:  # both are bf16 roundings of fp32 results: within one bf16 ulp
            ulp = np.spacing(np.abs(w).astype(np.float32)).astype(np.float64) * 65536.0
            assert np.all(np.abs(g - w) <= ulp)


def test_noalloc_rejects_partials_larger_than_its_scratch(lib):
    from paper_2601_16294_gb300 import binding
    A = torch.zeros(2048, 4096, dtype=torch.bfloat16, device="cuda")
    B = torch.zeros(4096, 2048, dtype=torch.bfloat16, device="cuda")
    C = torch.zeros(2048, 2048, dtype=torch.float32, device="cuda")
    assert lib.sfc_gemm_workspace_size(2048, 2048, 4096, 8) > binding.NOALLOC_SCRATCH_BYTES
    assert _noalloc(lib, A, B, C, 8) == binding.SFC_ERR_WORKSPACE
