"""The Python binding's own argument checks (CPU only).  Every malformed call
must raise before anything reaches the C library, so the library here is a fake
that fails the test if called; one well-formed call checks what the binding
passes through (strides, type codes, the stream)."""
import pytest
import torch

from paper_2601_16294_gb300 import binding


class FakeLib:
    def __init__(self, allow=False):
        self.allow = allow
        self.calls = []

    def sfc_gemm_ex3(self, *args):
        if not self.allow:
            raise AssertionError("a malformed call reached the library")
        self.calls.append(args)
        return binding.SFC_OK


class FakeStream:
    cuda_stream = 0x1234


@pytest.fixture
def fake(monkeypatch):
    lib = FakeLib()
    monkeypatch.setattr(binding, "_lib", lib)
    return lib


def bf(*shape):
    return torch.zeros(*shape, dtype=torch.bfloat16)


@pytest.mark.parametrize("case", [
    "A_3d", "layout", "inner", "dtype_mix", "dtype_f16", "beta_no_C", "C_dtype", "C_shape",
    "bias_dtype", "bias_len", "bias_strided", "A_col_stride", "B_col_stride"])
def test_malformed_calls_raise_before_the_library(fake, case):
    A, B, C = bf(64, 32), bf(32, 48), torch.zeros(64, 48)
    kw = {"stream": FakeStream()}
    err = ValueError
    if case == "A_3d":
        A = bf(2, 64, 32)
    elif case == "layout":
        kw["b_layout"] = "kk"
    elif case == "inner":
        B = bf(31, 48)
    elif case == "dtype_mix":
        B = torch.zeros(32, 48, dtype=torch.float32)
        err = TypeError
    elif case == "dtype_f16":
        A, B = A.half(), B.half()
        err = TypeError
    elif case == "beta_no_C":
        C = None
        kw["beta"] = 1.0
    elif case == "C_dtype":
        C = C.half()
    elif case == "C_shape":
        C = torch.zeros(48, 64)
    elif case == "bias_dtype":
        kw["bias"] = torch.zeros(48, dtype=torch.float64)
    elif case == "bias_len":
        kw["bias"] = torch.zeros(47)
    elif case == "bias_strided":
        kw["bias"] = torch.zeros(96)[::2]
    elif case == "A_col_stride":
        A = bf(32, 64).t()
    elif case == "B_col_stride":
        B = bf(48, 32).t()
    with pytest.raises(err):
        binding.gemm(A, B, C, **kw)
    assert fake.calls == []


def test_well_formed_call_passes_strides_codes_and_stream(monkeypatch):
    lib = FakeLib(allow=True)
    monkeypatch.setattr(binding, "_lib", lib)
    A = bf(64, 40)[:, :32]                       # padded rows: lda 40
    B = bf(32, 56)[:, :48]                       # ldb 56
    Cb = torch.zeros(64, 52, dtype=torch.bfloat16)
    C = Cb[:, :48]                               # ldc 52
    bias = torch.zeros(48)
    out = binding.gemm(A, B, C, ca_c=2, k_block_factor=1, order="raster", assign="segment", tile="pair256",
                       beta=0.5, bias=bias, stream=FakeStream())
    assert out is C and len(lib.calls) == 1
    (M, N, K, a, b, c, lda, ldb, ldc, ab, layout, beta, bias_ptr, ca_c, kbf, c_code, order, assign, tile,
     ws, ws_bytes, stream) = lib.calls[0]
    assert (M, N, K) == (64, 48, 32) and (lda, ldb, ldc) == (40, 56, 52)
    assert (a, b, c) == (A.data_ptr(), B.data_ptr(), C.data_ptr()) and bias_ptr == bias.data_ptr()
    assert ab == 0 and layout == binding.B_LAYOUTS["kn"] and c_code == binding.SFC_BF16
    assert (ca_c, kbf, beta) == (2, 1, 0.5)
    assert order == binding.ORDERS["raster"] and assign == binding.ASSIGNS["segment"]
    assert tile == binding.TILES["pair256"] and ws is None and ws_bytes == 0 and stream == 0x1234
    # B given as N x K
    lib.calls.clear()
    Bt = bf(48, 32)
    binding.gemm(A, Bt, torch.zeros(64, 48), b_layout="nk", stream=FakeStream())
    (M, N, K, *_rest) = lib.calls[0]
    assert (M, N, K) == (64, 48, 32) and lib.calls[0][10] == binding.B_LAYOUTS["nk"]
    assert lib.calls[0][15] == binding.SFC_F32


def test_library_errors_become_sfc_errors(monkeypatch):
    class Failing(FakeLib):
        def sfc_gemm_ex3(self, *args):
            return binding.SFC_ERR_UNALIGNED
    monkeypatch.setattr(binding, "_lib", Failing())
    with pytest.raises(binding.SfcError) as e:
        binding.gemm(bf(8, 8), bf(8, 8), torch.zeros(8, 8), stream=FakeStream())
    assert e.value.code == binding.SFC_ERR_UNALIGNED


class FakeNoAlloc:
    def __init__(self):
        self.calls = []

    def sfc_gemm_noalloc(self, *args):
        self.calls.append(args)
        return binding.SFC_OK


@pytest.mark.parametrize("case", ["A_3d", "inner", "A_f32", "B_f16", "C_dtype", "C_shape", "A_col_stride"])
def test_malformed_noalloc_calls_raise_before_the_library(monkeypatch, case):
    # the allocation-free entry point's tensor maps take their extents from M, N and K,
    # so a mis-shaped C or B would be read or written past its end: the binding refuses it
    lib = FakeNoAlloc()
    monkeypatch.setattr(binding, "_lib", lib)
    A, B, C = bf(64, 32), bf(32, 48), torch.zeros(64, 48)
    err = ValueError
    if case == "A_3d":
        A = bf(2, 64, 32)
    elif case == "inner":
        B = bf(40, 48)
    elif case == "A_f32":
        A = torch.zeros(64, 32)
        err = TypeError
    elif case == "B_f16":
        B = B.half()
        err = TypeError
    elif case == "C_dtype":
        C = C.half()
    elif case == "C_shape":
        C = torch.zeros(64, 40)
    elif case == "A_col_stride":
        A = bf(32, 64).t()
    with pytest.raises(err):
        binding.gemm_noalloc(A, B, C, ca_c=2, stream=FakeStream())
    assert lib.calls == []


def test_noalloc_passes_sizes_strides_and_codes(monkeypatch):
    lib = FakeNoAlloc()
    monkeypatch.setattr(binding, "_lib", lib)
    A = bf(64, 40)[:, :32]
    B = bf(32, 56)[:, :48]
    C = torch.zeros(64, 52, dtype=torch.bfloat16)[:, :48]
    assert binding.gemm_noalloc(A, B, C, ca_c=0, stream=FakeStream()) is C
    (M, N, K, a, b, c, lda, ldb, ldc, ca_c, c_code, stream) = lib.calls[0]
    assert (M, N, K, lda, ldb, ldc, ca_c) == (64, 48, 32, 40, 56, 52, 0)
    assert (a.value, b.value, c.value) == (A.data_ptr(), B.data_ptr(), C.data_ptr())
    assert c_code == binding.SFC_BF16 and stream == 0x1234
