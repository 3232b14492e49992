"""ctypes binding of ``libsfcgemm.so`` (C ABI declared in ``include/sfc_gemm.h``).

Argument marshalling only: every step of the GEMM runs in the library's CUDA
kernels.  PyTorch provides device memory and streams.  If the library is
missing, every call raises :class:`SfcLibraryMissing` -- there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

from . import build_lib

SFC_OK = 0
SFC_ERR_INVALID_ARG = -1
SFC_ERR_UNALIGNED = -2
SFC_ERR_WORKSPACE = -3
SFC_ERR_CUDA = -4
SFC_ERR_TIMEOUT = -5
SFC_ERR_UNSUPPORTED = -6
_NAMES = {0: "SFC_OK", -1: "SFC_ERR_INVALID_ARG", -2: "SFC_ERR_UNALIGNED", -3: "SFC_ERR_WORKSPACE",
          -4: "SFC_ERR_CUDA", -5: "SFC_ERR_TIMEOUT", -6: "SFC_ERR_UNSUPPORTED"}

SFC_F32, SFC_BF16 = 0, 1
ORDERS = {"sfc": 0, "raster": 1}
ASSIGNS = {"segment": 0, "wave": 1, "auto": 2, "wave_static": 3}
TILES = {0: 0, "auto": 0, 128: 128, 256: 256, "pair128": 1128, "pair256": 1256}
B_LAYOUTS = {"kn": 0, "nk": 1}


_AB_CODES = None
_torch = None


def _import_torch():
    """torch, imported on first use (the curve functions work without it)."""
    global _torch
    import torch
    _torch = torch
    return torch


def _ab_code(dtype) -> int:
    """sfc_ab_t of a torch dtype of A and B."""
    global _AB_CODES
    if _AB_CODES is None:
        import torch
        codes = {torch.bfloat16: 0}
        for name, code in (("float8_e4m3fn", 1), ("float8_e5m2", 2)):
            if hasattr(torch, name):
                codes[getattr(torch, name)] = code
        _AB_CODES = codes
    code = _AB_CODES.get(dtype)
    if code is None:
        raise TypeError("A and B must be bfloat16, float8_e4m3fn or float8_e5m2 (got %s)" % dtype)
    return code

EXPORTS = ("sfc_tile_order", "sfc_tile_order_device", "sfc_gemm_workspace_size", "sfc_gemm", "sfc_gemm_ex",
           "sfc_get_device_status", "sfc_last_cuda_error", "sfc_num_workers", "sfc_debug_force_timeout",
           "sfc_gemm_noalloc", "sfc_gemm_plan", "sfc_release", "sfc_gemm_ex2", "sfc_gemm_host", "sfc_gemm_ex3",
           "sfc_gemm_workspace_size2", "sfc_gemm_tune", "sfc_gemm_tune_forget",
           "sfc_gemm_tune_lookup", "sfc_mma_peak", "sfc_debug_pool_used_high", "sfc_gemm_plan_desc")
NOALLOC_SCRATCH_BYTES = 32 << 20


class SfcLibraryMissing(RuntimeError):
    pass


class SfcError(RuntimeError):
    def __init__(self, code: int, what: str, cuda_error: int = 0):
        self.code = code
        self.cuda_error = cuda_error
        msg = "%s failed: %s" % (what, _NAMES.get(code, str(code)))
        if code == SFC_ERR_CUDA:
            msg += " (CUDA error %d)" % cuda_error
        super().__init__(msg)


_lock = threading.Lock()
_lib = None


def library_path() -> str:
    return build_lib.LIB


def load():
    """Load the library (once).  Raises SfcLibraryMissing if it was not built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = library_path()
        if not os.path.exists(path):
            raise SfcLibraryMissing("libsfcgemm.so is not built (%s); run "
                                    "`python -m paper_2601_16294_gb300.build_lib`" % path)
        lib = ctypes.CDLL(path)
        i64, i32, vp, sz = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t
        lib.sfc_tile_order.argtypes = [i32, i32, vp]
        lib.sfc_tile_order_device.argtypes = [i32, i32, vp, vp]
        lib.sfc_gemm_workspace_size.argtypes = [i64, i64, i64, i32]
        lib.sfc_gemm_workspace_size.restype = sz
        lib.sfc_gemm.argtypes = [i64, i64, i64, vp, vp, vp, i64, i64, i64, i32, vp]
        lib.sfc_gemm_ex.argtypes = [i64, i64, i64, vp, vp, vp, i64, i64, i64, i32, i32, i32, i32, i32, vp, sz, vp]
        lib.sfc_get_device_status.argtypes = [vp]
        lib.sfc_last_cuda_error.argtypes = []
        lib.sfc_num_workers.argtypes = []
        lib.sfc_debug_force_timeout.argtypes = [vp, vp, vp, i32, vp]
        lib.sfc_gemm_noalloc.argtypes = [i64, i64, i64, vp, vp, vp, i64, i64, i64, i32, i32, vp]
        lib.sfc_gemm_plan.argtypes = [i64, i64, i64, i32, i32, i32, i32, i32, vp, vp]
        lib.sfc_gemm_ex2.argtypes = [i64, i64, i64, vp, vp, vp, i64, i64, i64, i32, i32, ctypes.c_float, vp, i32,
                                     i32, i32, i32, i32, vp, sz, vp]
        lib.sfc_release.argtypes = []
        lib.sfc_gemm_host.argtypes = [i64, i64, i64, vp, vp, vp, i64, i64, i64, i32, i32, i32, i32, i32, i32, vp]
        lib.sfc_gemm_ex3.argtypes = [i64, i64, i64, vp, vp, vp, i64, i64, i64, i32, i32, ctypes.c_float, vp, i32,
                                     i32, i32, i32, i32, i32, vp, sz, vp]
        lib.sfc_gemm_workspace_size2.argtypes = [i64, i64, i64, i32, i32, i32]
        lib.sfc_gemm_tune.argtypes = [i64, i64, i64, vp, vp, vp, i64, i64, i64, i32, i32, i32, i32, i32, vp, vp, vp, vp]
        lib.sfc_gemm_tune_forget.argtypes = []
        lib.sfc_gemm_tune_lookup.argtypes = [i32]
        lib.sfc_mma_peak.argtypes = [i32, vp, vp, vp]
        lib.sfc_debug_pool_used_high.argtypes = [vp, i32]
        lib.sfc_gemm_plan_desc.argtypes = [vp, i64, i64, i64, i32, i32, i32, i32, vp, vp, vp]

        lib.sfc_gemm_workspace_size2.restype = sz
        for name in EXPORTS:
            if name not in ("sfc_gemm_workspace_size", "sfc_gemm_workspace_size2"):
                getattr(lib, name).restype = ctypes.c_int
        _lib = lib
        return lib


def _check(rc: int, what: str):
    if rc != SFC_OK:
        raise SfcError(rc, what, load().sfc_last_cuda_error() if rc == SFC_ERR_CUDA else 0)


def _stream_ptr(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


# ------------------------------------------------------------------ curve

def tile_order(Mt: int, Nt: int) -> np.ndarray:
    """Curve permutation from the library's host decoder: out[s] = tm*Nt + tn."""
    out = np.empty(int(Mt) * int(Nt), dtype=np.int32)
    _check(load().sfc_tile_order(int(Mt), int(Nt), out.ctypes.data), "sfc_tile_order")
    return out


def tile_order_device(Mt: int, Nt: int, stream=None):
    """Curve permutation from the GPU decoder the GEMM kernel uses (int32 CUDA tensor)."""
    import torch
    out = torch.empty(int(Mt) * int(Nt), dtype=torch.int32, device="cuda")
    _check(load().sfc_tile_order_device(int(Mt), int(Nt), ctypes.c_void_p(out.data_ptr()),
                                        _stream_ptr(stream)), "sfc_tile_order_device")
    return out


# ------------------------------------------------------------------- GEMM

def workspace_size(M: int, N: int, K: int, ca_c: int, k_block_factor: int = 1, out_dtype=None) -> int:
    """Bytes of workspace a call needs (``sfc_gemm_workspace_size2``)."""
    import torch
    dt = SFC_BF16 if out_dtype == torch.bfloat16 else SFC_F32
    return int(load().sfc_gemm_workspace_size2(int(M), int(N), int(K), int(ca_c), int(k_block_factor), dt))


def plan(M: int, N: int, K: int, ca_c: int = 0, out_dtype=None, tile="auto", in_dtype=None,
         b_layout: str = "kn"):
    """(tile, ca_c) the library would use for this call on the current device;
    tile is a key of TILES other than "auto".  in_dtype: the dtype of A and B
    (bfloat16 when None)."""
    import torch
    t = ctypes.c_int(0)
    c = ctypes.c_int(0)
    dt = SFC_BF16 if out_dtype == torch.bfloat16 else SFC_F32
    ab = _ab_code(in_dtype or torch.bfloat16)
    _check(load().sfc_gemm_plan(int(M), int(N), int(K), int(ca_c), dt, TILES[tile], ab, B_LAYOUTS[b_layout],
                                ctypes.byref(t), ctypes.byref(c)), "sfc_gemm_plan")
    name = {v: k for k, v in TILES.items() if k not in (0, "auto")}[t.value]
    return name, c.value


class DeviceDesc(ctypes.Structure):
    """``sfc_device_desc_t``: a device as the library's time model sees it."""
    _fields_ = [("num_sms", ctypes.c_int), ("pair_workers", ctypes.c_int), ("hbm_gbs", ctypes.c_double),
                ("sm_ghz", ctypes.c_double)]


GB300 = dict(num_sms=152, pair_workers=76, hbm_gbs=6700.0, sm_ghz=1.9)


def plan_model(M: int, N: int, K: int, ca_c: int = 0, *, out: str = "bf16", ab: str = "bf16",
               b_layout: str = "kn", device: dict | None = None):
    """The time model alone (``sfc_gemm_plan_desc``, no GPU): ``(tile, ca_c,
    predicted_ns)`` for a described device (default: GB300's figures)."""
    d = DeviceDesc(**(device or GB300))
    t, c, ns = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_double(0.0)
    ab_code = {"bf16": 0, "e4m3": 1, "e5m2": 2}[ab]
    _check(load().sfc_gemm_plan_desc(ctypes.byref(d), int(M), int(N), int(K), int(ca_c),
                                     SFC_F32 if out == "f32" else SFC_BF16, ab_code, B_LAYOUTS[b_layout],
                                     ctypes.byref(t), ctypes.byref(c), ctypes.byref(ns)), "sfc_gemm_plan_desc")
    name = {v: k for k, v in TILES.items() if k not in (0, "auto")}[t.value]
    return name, c.value, ns.value


def tune(A, B, C=None, *, out_dtype=None, b_layout: str = "kn", max_layers: int = 8, max_kbf: int = 4,
         stream=None):
    """Measure the configurations of this shape (``sfc_gemm_tune``) and remember
    the fastest for later calls with ``tile="auto"``.  A, B: CUDA tensors as
    for :func:`gemm`; C is overwritten (allocated if not given).  Returns
    ``(tile, ca_c, k_block_factor)`` of the fastest configuration."""
    import torch
    M, K = A.shape
    N = B.shape[1] if b_layout == "kn" else B.shape[0]
    if C is None:
        C = torch.empty((M, N), dtype=out_dtype or torch.float32, device=A.device)
    t, c, kbf = ctypes.c_int(0), ctypes.c_int(0), ctypes.c_int(0)
    rc = load().sfc_gemm_tune(M, N, K, ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(B.data_ptr()),
                              ctypes.c_void_p(C.data_ptr()), _row_major_2d(A, "A"), _row_major_2d(B, "B"),
                              _row_major_2d(C, "C"), _ab_code(A.dtype), B_LAYOUTS[b_layout],
                              SFC_F32 if C.dtype == torch.float32 else SFC_BF16, int(max_layers), int(max_kbf),
                              _stream_ptr(stream), ctypes.byref(t), ctypes.byref(c), ctypes.byref(kbf))
    _check(rc, "sfc_gemm_tune")
    name = {v: k for k, v in TILES.items() if k not in (0, "auto")}[t.value]
    return name, c.value, kbf.value


def tune_lookup(nearest: bool) -> None:
    """AUTO calls use tuned shapes exactly (False, the default) or also the
    nearest tuned shape (True; ``sfc_gemm_tune_lookup``)."""
    _check(load().sfc_gemm_tune_lookup(2 if nearest else 1), "sfc_gemm_tune_lookup")


def tune_forget() -> None:
    """Forget every tuned shape on the current device."""
    _check(load().sfc_gemm_tune_forget(), "sfc_gemm_tune_forget")


def mma_peak(iters: int = 4096, stream=None):
    """``(flop_per_clk_per_sm, tflops)``: the tensor cores' attainable rate
    from resident operands (``sfc_mma_peak``)."""
    f, t = ctypes.c_double(0.0), ctypes.c_double(0.0)
    _check(load().sfc_mma_peak(int(iters), ctypes.byref(f), ctypes.byref(t), _stream_ptr(stream)), "sfc_mma_peak")
    return f.value, t.value


def release() -> None:
    """Give the device memory the library keeps between calls (host-entry staging
    slots, its workspace pool) back to the driver."""
    _check(load().sfc_release(), "sfc_release")


def num_workers() -> int:
    n = load().sfc_num_workers()
    if n < 0:
        _check(n, "sfc_num_workers")
    return n


def _row_major_2d(t, name):
    st = t.stride()
    if len(st) != 2 or st[1] != 1:
        raise ValueError("%s must be a 2-D row-major (unit column stride) tensor" % name)
    return st[0]


def gemm(A, B, C=None, *, ca_c: int = 1, out_dtype=None, order: str = "sfc", assign: str = "auto",
         tile=0, workspace=None, stream=None, b_layout: str = "kn", beta: float = 0.0, bias=None,
         k_block_factor: int = 1):
    """C = A @ B (+ beta * C + bias) on the GPU.  A: (M, K) CUDA tensor, bf16
    or an 8-bit float (float8_e4m3fn, float8_e5m2), row-major (row stride may
    be padded).  B: the same dtype, (K, N) for ``b_layout="kn"`` or its
    transpose (N, K) for ``"nk"`` (a linear layer's weight).  C: (M, N)
    fp32 or bf16 CUDA tensor, allocated if not given (then ``beta`` must be 0).
    ``bias``: optional fp32 CUDA tensor of N values.  ``ca_c``: K layers (0: the
    library chooses).  ``k_block_factor``: passes over each layer's K range,
    summed into C (or the layer copies) in place.  ``workspace``: optional CUDA
    tensor of at least ``workspace_size(M, N, K, ca_c, k_block_factor,
    out_dtype)`` bytes."""
    lib = _lib or load()
    torch = _torch or _import_torch()
    M, K = A.shape
    if b_layout == "kn":
        K2, N = B.shape
    elif b_layout == "nk":
        N, K2 = B.shape
    else:
        raise ValueError("b_layout must be 'kn' or 'nk'")
    if K != K2:
        raise ValueError("inner dimensions differ: %d vs %d" % (K, K2))
    a_dtype = A.dtype
    if a_dtype != B.dtype:
        raise TypeError("A and B must have the same dtype")
    ab = _ab_code(a_dtype)
    if C is None:
        if beta != 0.0:
            raise ValueError("beta != 0 needs an input C")
        C = torch.empty((M, N), dtype=out_dtype or torch.float32, device=A.device)
    c_dtype = C.dtype
    if c_dtype == torch.float32:
        c_code = SFC_F32
    elif c_dtype == torch.bfloat16:
        c_code = SFC_BF16
    else:
        c_code = -1
    if c_code < 0 or C.shape != (M, N):
        raise ValueError("C must be (M, N) float32 or bfloat16")
    bias_ptr = None
    if bias is not None:
        if bias.dtype != torch.float32 or bias.numel() != N or not bias.is_contiguous():
            raise ValueError("bias must be a contiguous float32 tensor of N values")
        bias_ptr = bias.data_ptr()
    lda = _row_major_2d(A, "A")
    ldb = _row_major_2d(B, "B")
    ldc = _row_major_2d(C, "C")
    ws_ptr, ws_bytes = None, 0
    if workspace is not None:
        ws_ptr, ws_bytes = workspace.data_ptr(), workspace.numel() * workspace.element_size()
    rc = lib.sfc_gemm_ex3(M, N, K, A.data_ptr(), B.data_ptr(), C.data_ptr(), lda, ldb, ldc, ab,
                          B_LAYOUTS[b_layout], beta, bias_ptr, ca_c, k_block_factor, c_code, ORDERS[order],
                          ASSIGNS[assign], TILES[tile], ws_ptr, ws_bytes,
                          (stream if stream is not None else torch.cuda.current_stream()).cuda_stream)
    if rc != SFC_OK:
        _check(rc, "sfc_gemm_ex3")
    return C


def gemm_noalloc(A, B, C, *, ca_c: int = 1, stream=None):
    """C = A @ B through ``sfc_gemm_noalloc``, for callers that cannot allocate
    device memory: the K-layer partials and the workers' item counter use the
    library's built-in scratch area, so the call allocates nothing.  A: (M, K)
    bf16, B: (K, N) bf16, both CUDA tensors with 16-byte-aligned rows (nothing
    is repacked); C: preallocated (M, N) fp32 or bf16 CUDA tensor.  Raises
    SfcError(SFC_ERR_WORKSPACE) when ca_c >= 2 layers' partials would not fit in
    ``NOALLOC_SCRATCH_BYTES`` (ca_c = 0 picks a count that fits)."""
    torch = _torch or _import_torch()
    if A.dim() != 2 or B.dim() != 2 or C.dim() != 2:
        raise ValueError("A, B and C must be 2-D")
    M, K = A.shape
    K2, N = B.shape
    if K != K2:
        raise ValueError("inner dimensions differ: %d vs %d" % (K, K2))
    if A.dtype != torch.bfloat16 or B.dtype != torch.bfloat16:
        raise TypeError("A and B must be bfloat16")
    if C.dtype not in (torch.float32, torch.bfloat16) or tuple(C.shape) != (M, N):
        raise ValueError("C must be (M, N) float32 or bfloat16")
    rc = load().sfc_gemm_noalloc(M, N, K, ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(B.data_ptr()),
                                 ctypes.c_void_p(C.data_ptr()), _row_major_2d(A, "A"), _row_major_2d(B, "B"),
                                 _row_major_2d(C, "C"), int(ca_c),
                                 SFC_F32 if C.dtype == torch.float32 else SFC_BF16, _stream_ptr(stream))
    _check(rc, "sfc_gemm_noalloc")
    return C


def pool_used_high(reset: bool = False) -> int:
    """High-water mark in bytes of the memory in use from the library's
    stream-ordered pools on the current device since the last reset
    (``sfc_debug_pool_used_high``); ``reset=True`` starts a new count."""
    v = ctypes.c_size_t(0)
    _check(load().sfc_debug_pool_used_high(ctypes.byref(v), 1 if reset else 0), "sfc_debug_pool_used_high")
    return int(v.value)


def gemm_raw(M, N, K, A_ptr, B_ptr, C_ptr, lda, ldb, ldc, ca_c=1, stream_ptr=None) -> int:
    """Direct call of ``sfc_gemm`` with raw device pointers; returns the status code."""
    return load().sfc_gemm(int(M), int(N), int(K), ctypes.c_void_p(A_ptr), ctypes.c_void_p(B_ptr),
                           ctypes.c_void_p(C_ptr), int(lda), int(ldb), int(ldc), int(ca_c),
                           ctypes.c_void_p(stream_ptr))


def device_status(stream=None) -> int:
    """Synchronise the stream and return (and clear) the kernels' error word."""
    return load().sfc_get_device_status(_stream_ptr(stream))


def debug_force_timeout(A, B, C, limit_ms: int = 20, stream=None) -> int:
    return load().sfc_debug_force_timeout(ctypes.c_void_p(A.data_ptr()), ctypes.c_void_p(B.data_ptr()),
                                          ctypes.c_void_p(C.data_ptr()), int(limit_ms), _stream_ptr(stream))


def gemm_host(A_host, B_host, C_host=None, *, ca_c: int = 0, out_dtype=None, tile=0, b_layout: str = "kn",
              panels: int = 0, stream=None):
    """C = A @ B from HOST tensors through ``sfc_gemm_host``: the library
    uploads A and B, runs the GEMM and downloads C, overlapping the copies
    with the contraction (slices of ``panels`` rows or columns; 0 = automatic).
    A, B: CPU tensors (bf16 or an 8-bit float), row-major with any row stride,
    ideally pinned; B is (K, N) for ``b_layout="kn"`` or (N, K) for ``"nk"``.
    C_host: (M, N) fp32 or bf16 CPU tensor, allocated pinned if not given.
    Asynchronous on ``stream``: C_host is complete once the stream has been
    synchronised, and A and B are read until then, so the caller keeps all
    three tensors alive and A and B unchanged until it synchronises (a
    temporary passed here could be freed and its memory reused too early)."""
    import torch
    M, K = A_host.shape
    if b_layout == "kn":
        K2, N = B_host.shape
    elif b_layout == "nk":
        N, K2 = B_host.shape
    else:
        raise ValueError("b_layout must be 'kn' or 'nk'")
    if K != K2:
        raise ValueError("inner dimensions differ: %d vs %d" % (K, K2))
    if A_host.dtype != B_host.dtype:
        raise TypeError("A and B must have the same dtype")
    for name, t in (("A", A_host), ("B", B_host)):
        if t.device.type != "cpu":
            raise ValueError("%s must be a host (CPU) tensor" % name)
    if C_host is None:
        C_host = torch.empty((M, N), dtype=out_dtype or torch.float32, pin_memory=True)
    if C_host.device.type != "cpu" or C_host.dtype not in (torch.float32, torch.bfloat16) or \
            tuple(C_host.shape) != (M, N):
        raise ValueError("C_host must be an (M, N) float32 or bfloat16 CPU tensor")
    rc = load().sfc_gemm_host(M, N, K, ctypes.c_void_p(A_host.data_ptr()), ctypes.c_void_p(B_host.data_ptr()),
                              ctypes.c_void_p(C_host.data_ptr()), _row_major_2d(A_host, "A"),
                              _row_major_2d(B_host, "B"), _row_major_2d(C_host, "C"), _ab_code(A_host.dtype),
                              B_LAYOUTS[b_layout], int(ca_c), SFC_F32 if C_host.dtype == torch.float32 else SFC_BF16,
                              TILES[tile], int(panels), _stream_ptr(stream))
    _check(rc, "sfc_gemm_host")
    return C_host


def matmul_host(A_host, B_host, C_host=None, *, ca_c: int = 0, out_dtype=None, stream=None, **kw):
    """End-to-end call from HOST tensors: :func:`gemm_host`, then a
    synchronisation of the stream.  Returns C_host, complete."""
    import torch
    s = stream or torch.cuda.current_stream()
    C_host = gemm_host(A_host, B_host, C_host, ca_c=ca_c, out_dtype=out_dtype, stream=s, **kw)
    s.synchronize()
    return C_host
