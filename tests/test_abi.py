"""C ABI checks that need no GPU: the library builds, loads and exports every
declared entry point; its host curve decoder equals the oracle; argument
validation returns the documented codes before touching the device; without
a usable GPU the compute entry points fail loudly instead of falling back."""
import ctypes
import os
import re

import numpy as np
import pytest

import paper_2601_16294_gb300 as sfc
from paper_2601_16294_gb300 import binding, build_lib

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "sfc_gemm.h")


@pytest.fixture(scope="module")
def lib():
    build_lib.build()
    return binding.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:int|size_t|void|long long)\s+\**(sfc_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("sfc_tile_order", "sfc_gemm", "sfc_gemm_ex", "sfc_gemm_workspace_size"):
        assert required in names
    assert set(names) == set(binding.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name
        assert ctypes.cast(getattr(lib, name), ctypes.c_void_p).value


@pytest.mark.parametrize("Mt", range(1, 34))
def test_host_decoder_matches_oracle_small(lib, oracle, Mt):
    for Nt in range(1, 34):
        assert np.array_equal(sfc.tile_order(Mt, Nt), oracle.gilbert_order(Mt, Nt)), (Mt, Nt)


@pytest.mark.parametrize("Mt,Nt", [(4, 4), (128, 128), (128, 64), (64, 1002), (2, 64), (24, 40), (8, 133),
                                   (48, 6), (4, 1002), (16, 501), (1002, 64), (65, 63), (1, 1002)])
def test_host_decoder_matches_oracle_config_grids(lib, oracle, Mt, Nt):
    assert np.array_equal(sfc.tile_order(Mt, Nt), oracle.gilbert_order(Mt, Nt))


def test_tile_order_rejects_bad_arguments(lib):
    buf = np.empty(4, dtype=np.int32)
    assert lib.sfc_tile_order(0, 4, buf.ctypes.data) == binding.SFC_ERR_INVALID_ARG
    assert lib.sfc_tile_order(4, -1, buf.ctypes.data) == binding.SFC_ERR_INVALID_ARG
    assert lib.sfc_tile_order(2, 2, None) == binding.SFC_ERR_INVALID_ARG
    assert lib.sfc_tile_order(65536, 65536, buf.ctypes.data) == binding.SFC_ERR_INVALID_ARG


def test_workspace_size(lib):
    assert sfc.workspace_size(512, 512, 4096, 1) == 0
    assert sfc.workspace_size(512, 512, 4096, 4) == 4 * 512 * 512 * 4
    assert sfc.workspace_size(3, 5, 64, 2) == 2 * 3 * 8 * 4          # rows padded to 4 floats
    assert sfc.workspace_size(0, 5, 64, 2) == 0
    assert sfc.workspace_size(3, 5, 64, -1) == 0


def test_workspace_size_for_chosen_layers(lib):
    # ca_c = 0: room for the most layers the planner may pick,
    # min(64, ceil(K/64), ceil(320 / (ceil(M/128) ceil(N/128))))
    assert sfc.workspace_size(512, 512, 32768, 0) == 20 * 512 * 512 * 4      # 16 tiles -> 20 layers
    assert sfc.workspace_size(128, 128, 1 << 20, 0) == 64 * 128 * 128 * 4    # capped at 64
    assert sfc.workspace_size(128, 128, 200, 0) == 4 * 128 * 128 * 4         # Kt = 4
    assert sfc.workspace_size(4096, 4096, 4096, 0) == 0                      # 1024 tiles -> 1 layer
    assert sfc.workspace_size(3, 5, 64, 0) == 0                              # Kt = 1


# Fake, never-dereferenced device addresses: validation runs before any CUDA call.
PA, PB, PC = 0x10000, 0x20000, 0x30000


def call_ex(lib, M=256, N=256, K=256, A=PA, B=PB, C=PC, lda=None, ldb=None, ldc=None, ca_c=1, dtype=0,
            order=0, assign=2, tile=0, ws=None, ws_bytes=0):
    lda = K if lda is None else lda
    ldb = N if ldb is None else ldb
    ldc = N if ldc is None else ldc
    return lib.sfc_gemm_ex(M, N, K, ctypes.c_void_p(A), ctypes.c_void_p(B), ctypes.c_void_p(C), lda, ldb, ldc,
                           ca_c, dtype, order, assign, tile, ctypes.c_void_p(ws) if ws else None, ws_bytes, None)


def test_gemm_validation_codes(lib):
    E = binding
    assert call_ex(lib, M=0) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, N=-1) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, K=0) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, A=0) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, C=0) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, lda=128) == E.SFC_ERR_INVALID_ARG          # lda < K
    assert call_ex(lib, ldc=100) == E.SFC_ERR_INVALID_ARG          # ldc < N
    assert call_ex(lib, ca_c=-1) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, K=256, ca_c=5) == E.SFC_ERR_INVALID_ARG    # Kt = 4 < ca_c
    assert call_ex(lib, K=64 * 5000, ca_c=4097) == E.SFC_ERR_INVALID_ARG  # more than 4096 layers
    assert call_ex(lib, dtype=7) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, order=3) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, assign=9) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, tile=64) == E.SFC_ERR_INVALID_ARG
    assert call_ex(lib, A=PA + 1) == E.SFC_ERR_UNALIGNED           # A not aligned to its 2-byte elements
    assert call_ex(lib, B=PB + 3) == E.SFC_ERR_UNALIGNED
    need = sfc.workspace_size(256, 256, 256, 2)
    assert call_ex(lib, ca_c=2, ws=0x40000, ws_bytes=need - 4) == E.SFC_ERR_WORKSPACE
    assert call_ex(lib, ca_c=2, ws=0x40008, ws_bytes=need) == E.SFC_ERR_UNALIGNED
    assert lib.sfc_gemm(256, 256, 256, None, ctypes.c_void_p(PB), ctypes.c_void_p(PC), 256, 256, 256, 1,
                        None) == E.SFC_ERR_INVALID_ARG
    assert lib.sfc_debug_force_timeout(ctypes.c_void_p(PA), ctypes.c_void_p(PB), ctypes.c_void_p(PC), 0,
                                       None) == E.SFC_ERR_INVALID_ARG


def _has_gpu():
    try:
        import torch
        return torch.cuda.is_available()
    except Exception:
        return False


@pytest.mark.skipif(_has_gpu(), reason="checks the no-GPU failure path")
def test_valid_call_without_gpu_fails_loudly(lib):
    rc = call_ex(lib)
    assert rc in (binding.SFC_ERR_CUDA, binding.SFC_ERR_UNSUPPORTED)
    assert call_ex(lib, ca_c=0) in (binding.SFC_ERR_CUDA, binding.SFC_ERR_UNSUPPORTED)
    assert lib.sfc_num_workers() < 0
    assert lib.sfc_get_device_status(None) == binding.SFC_ERR_CUDA
    assert lib.sfc_release() == binding.SFC_ERR_CUDA
    t, c = ctypes.c_int(0), ctypes.c_int(0)
    assert lib.sfc_gemm_plan(512, 512, 4096, 0, 0, 0, 0, 0, ctypes.byref(t), ctypes.byref(c)) in (
        binding.SFC_ERR_CUDA, binding.SFC_ERR_UNSUPPORTED)


def test_plan_validation(lib):
    t, c = ctypes.c_int(0), ctypes.c_int(0)
    def plan(M, N, K, c_, tile=0, ab=0, layout=0, out=True):
        return lib.sfc_gemm_plan(M, N, K, c_, 0, tile, ab, layout, ctypes.byref(t) if out else None,
                                 ctypes.byref(c))
    assert plan(512, 512, 4096, 0, out=False) == binding.SFC_ERR_INVALID_ARG
    assert plan(0, 512, 4096, 0) == binding.SFC_ERR_INVALID_ARG
    assert plan(512, 512, 4096, -2) == binding.SFC_ERR_INVALID_ARG
    assert plan(512, 512, 4096, 0, tile=77) == binding.SFC_ERR_INVALID_ARG
    assert plan(512, 512, 4096, 0, ab=5) == binding.SFC_ERR_INVALID_ARG
    assert plan(512, 512, 4096, 0, layout=3) == binding.SFC_ERR_INVALID_ARG


def test_missing_library_raises(monkeypatch, tmp_path):
    monkeypatch.setattr(binding, "_lib", None)
    monkeypatch.setattr(binding, "library_path", lambda: str(tmp_path / "absent.so"))
    with pytest.raises(binding.SfcLibraryMissing):
        binding.load()


def call_ex2(lib, M=256, N=256, K=256, ldb=None, b_layout=0, beta=0.0, bias=None, ca_c=1, ab=0, lda=None):
    ldb = (N if b_layout == 0 else K) if ldb is None else ldb
    return lib.sfc_gemm_ex2(M, N, K, ctypes.c_void_p(PA), ctypes.c_void_p(PB), ctypes.c_void_p(PC), lda or K, ldb,
                            N, ab, b_layout, beta, ctypes.c_void_p(bias) if bias else None, ca_c, 0, 0, 2, 0, None,
                            0, None)


def test_gemm_ex2_validation_codes(lib):
    E = binding
    assert call_ex2(lib, b_layout=2) == E.SFC_ERR_INVALID_ARG
    assert call_ex2(lib, N=512, K=256, b_layout=1, ldb=200) == E.SFC_ERR_INVALID_ARG    # B^T rows shorter than K
    assert call_ex2(lib, N=512, K=256, b_layout=0, ldb=256) == E.SFC_ERR_INVALID_ARG    # B rows shorter than N
    assert call_ex2(lib, bias=0x50002) == E.SFC_ERR_UNALIGNED                           # bias not 4-byte aligned
    assert call_ex2(lib, ab=3) == E.SFC_ERR_INVALID_ARG                                 # unknown input type
    assert call_ex2(lib, ab=1, K=256 * 129, ca_c=259) == E.SFC_ERR_INVALID_ARG          # 258 slabs of 128 k


def call_host(lib, M=256, N=256, K=256, lda=None, ldb=None, ldc=None, ab=0, b_layout=0, c_dtype=0, panels=0,
              a=0x10000, b=0x20000, c=0x30000):
    ldb = (N if b_layout == 0 else K) if ldb is None else ldb
    return lib.sfc_gemm_host(M, N, K, ctypes.c_void_p(a), ctypes.c_void_p(b), ctypes.c_void_p(c), lda or K, ldb,
                             ldc or N, ab, b_layout, 1, c_dtype, 0, panels, None)


def test_gemm_host_validation_codes(lib):
    # every case fails on the host before any staging memory or stream is touched
    E = binding
    assert call_host(lib, M=0) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, K=-1) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, a=0) == E.SFC_ERR_INVALID_ARG                       # null host pointer
    assert call_host(lib, c=0) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, lda=255) == E.SFC_ERR_INVALID_ARG                   # rows of A shorter than K
    assert call_host(lib, N=512, ldb=256) == E.SFC_ERR_INVALID_ARG            # rows of B shorter than N
    assert call_host(lib, N=512, K=256, b_layout=1, ldb=200) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, ldc=100) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, ab=7) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, b_layout=3) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, c_dtype=5) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, panels=-1) == E.SFC_ERR_INVALID_ARG
    assert call_host(lib, a=0x10001) == E.SFC_ERR_UNALIGNED                   # bf16 at an odd address
    assert call_host(lib, c=0x30002) == E.SFC_ERR_UNALIGNED                   # fp32 C at a 2-byte offset


def test_workspace_size_with_k_blocks(lib):
    import torch
    ws = sfc.workspace_size
    assert ws(512, 512, 4096, 1, k_block_factor=4) == 0                                  # fp32 C: in place
    assert ws(512, 512, 4096, 1, k_block_factor=4, out_dtype=torch.bfloat16) == 512 * 512 * 4   # one fp32 copy
    assert ws(512, 512, 4096, 1, k_block_factor=1, out_dtype=torch.bfloat16) == 0
    assert ws(512, 512, 4096, 3, k_block_factor=2) == 3 * 512 * 512 * 4
    # ca_c = 0: the planner's bound, at most ceil(K/64) / k_block_factor layers
    assert ws(512, 512, 32768, 0, k_block_factor=1) == 20 * 512 * 512 * 4
    assert ws(512, 512, 1024, 0, k_block_factor=4) == 4 * 512 * 512 * 4                 # 16 slabs / 4
    assert ws(512, 512, 4096, 1, k_block_factor=0) == 0                                  # invalid
    assert ws(512, 512, 4096, 1, k_block_factor=65) == 0


def call_ex3(lib, M=256, N=256, K=1024, ca_c=1, kbf=2, ab=0):
    return lib.sfc_gemm_ex3(M, N, K, ctypes.c_void_p(PA), ctypes.c_void_p(PB), ctypes.c_void_p(PC), K, N, N, ab, 0,
                            0.0, None, ca_c, kbf, 0, 0, 2, 0, None, 0, None)


def test_gemm_ex3_validation_codes(lib):
    # every case is rejected on the host, before the device is touched
    E = binding
    assert call_ex3(lib, kbf=0) == E.SFC_ERR_INVALID_ARG
    assert call_ex3(lib, kbf=65) == E.SFC_ERR_INVALID_ARG
    assert call_ex3(lib, K=256, kbf=5) == E.SFC_ERR_INVALID_ARG                # 4 slabs of 64
    assert call_ex3(lib, K=1024, ca_c=4, kbf=5) == E.SFC_ERR_INVALID_ARG       # 16 slabs: 4 per layer < 5
    assert call_ex3(lib, K=1024, ab=1, ca_c=2, kbf=5) == E.SFC_ERR_INVALID_ARG  # 8 slabs of 128: 4 per layer
    assert call_ex3(lib, M=0) == E.SFC_ERR_INVALID_ARG


def test_gemm_tune_validation_codes(lib):
    # rejected on the host before the device is touched
    E = binding
    t, c, k = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_int(0)

    def tune(M=256, N=256, K=256, max_layers=8, max_kbf=4, outs=True):
        args = (ctypes.byref(t), ctypes.byref(c), ctypes.byref(k)) if outs else (None, None, None)
        return lib.sfc_gemm_tune(M, N, K, ctypes.c_void_p(PA), ctypes.c_void_p(PB), ctypes.c_void_p(PC), K, N, N,
                                 0, 0, 0, max_layers, max_kbf, None, *args)
    assert tune(outs=False) == E.SFC_ERR_INVALID_ARG
    assert tune(max_layers=0) == E.SFC_ERR_INVALID_ARG
    assert tune(max_layers=65) == E.SFC_ERR_INVALID_ARG
    assert tune(max_kbf=0) == E.SFC_ERR_INVALID_ARG
    assert tune(max_kbf=65) == E.SFC_ERR_INVALID_ARG
    assert tune(M=0) == E.SFC_ERR_INVALID_ARG


def test_tune_lookup_modes(lib):
    assert lib.sfc_gemm_tune_lookup(3) == binding.SFC_ERR_INVALID_ARG
    assert lib.sfc_gemm_tune_lookup(0) == binding.SFC_ERR_INVALID_ARG
    assert lib.sfc_gemm_tune_lookup(2) == binding.SFC_OK
    assert lib.sfc_gemm_tune_lookup(1) == binding.SFC_OK


def test_mma_peak_validation(lib):
    f, t = ctypes.c_double(0.0), ctypes.c_double(0.0)
    assert lib.sfc_mma_peak(0, ctypes.byref(f), ctypes.byref(t), None) == binding.SFC_ERR_INVALID_ARG
    assert lib.sfc_mma_peak((1 << 20) + 1, ctypes.byref(f), ctypes.byref(t), None) == binding.SFC_ERR_INVALID_ARG
    assert lib.sfc_mma_peak(16, None, ctypes.byref(t), None) == binding.SFC_ERR_INVALID_ARG
