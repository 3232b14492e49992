"""Python access to the plain CPU oracle (``oracle.c``).

TEST INFRASTRUCTURE ONLY.  Only the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this module.  The product path (the
CUDA library and its binding) never touches it.

What the oracle computes, and the passage each part follows:

* ``gilbert_order(Mt, Nt)`` -- the generalized Hilbert curve over the Mt x Nt
  output-tile grid (Sec. II-B, Fig. 2; ``create_sfc_map`` / ``map_sfc_index``
  of Listing 1).  ``out[s] = tm * Nt + tn``.
* ``gemm_f64(A, B)`` -- C = A * B by definition, fp64 accumulation over the
  bf16 inputs widened exactly (Sec. II-A, Listing 1).
* ``gemm_sub_f64(A, B, rows, cols, k0, k1)`` -- selected rows/columns, optionally
  one K range (one layer's partial product of the K split, Sec. II-C/D).
* ``round_bf16(x)`` -- one-step round-to-nearest-even of doubles to bf16.
* ``set_threads(n)`` / ``max_threads()`` -- the OpenMP thread count of the loops
  (for timing on a chosen number of host cores; no arithmetic).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``oracle.c`` into ``liboracle.so`` beside it (gcc, OpenMP)."""
    if not force and os.path.exists(_LIB) and os.path.getmtime(_LIB) >= os.path.getmtime(_SRC):
        return _LIB
    tmp = _LIB + ".tmp%d" % os.getpid()
    cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
           "-ffp-contract=off", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        i32p = ctypes.POINTER(ctypes.c_int32)
        u16p = ctypes.c_void_p
        i64 = ctypes.c_int64
        lib.oracle_gilbert_order.argtypes = [ctypes.c_int, ctypes.c_int, i32p]
        lib.oracle_gilbert_order.restype = ctypes.c_int
        lib.oracle_gemm_f64.argtypes = [i64, i64, i64, u16p, i64, u16p, i64, ctypes.c_void_p, i64]
        lib.oracle_gemm_f64.restype = None
        lib.oracle_gemm_sub_f64.argtypes = [ctypes.c_void_p, i64, ctypes.c_void_p, i64, i64, i64,
                                            u16p, i64, u16p, i64, ctypes.c_void_p]
        lib.oracle_gemm_sub_f64.restype = None
        lib.oracle_gemm_affine_f64.argtypes = [i64, i64, i64, u16p, i64, u16p, i64, ctypes.c_int,
                                               ctypes.c_double, ctypes.c_void_p, i64, ctypes.c_void_p,
                                               ctypes.c_void_p, i64]
        lib.oracle_gemm_affine_f64.restype = None
        lib.oracle_decode_f8.argtypes = [ctypes.c_uint8, ctypes.c_int]
        lib.oracle_decode_f8.restype = ctypes.c_double
        lib.oracle_gemm_f8_f64.argtypes = [i64, i64, i64, ctypes.c_void_p, i64, ctypes.c_void_p, i64, ctypes.c_int,
                                           ctypes.c_int, ctypes.c_void_p, i64]
        lib.oracle_gemm_f8_f64.restype = None
        lib.oracle_round_bf16.argtypes = [ctypes.c_double]
        lib.oracle_round_bf16.restype = ctypes.c_uint16
        lib.oracle_round_bf16_array.argtypes = [ctypes.c_void_p, i64, ctypes.c_void_p]
        lib.oracle_round_bf16_array.restype = None
        lib.oracle_set_threads.argtypes = [ctypes.c_int]
        lib.oracle_set_threads.restype = None
        lib.oracle_max_threads.argtypes = []
        lib.oracle_max_threads.restype = ctypes.c_int
        _lib = lib
        return lib


def gilbert_order(Mt: int, Nt: int) -> np.ndarray:
    """Curve permutation: ``out[s] = tm * Nt + tn`` (int32, length Mt*Nt)."""
    out = np.empty(Mt * Nt, dtype=np.int32)
    rc = _load().oracle_gilbert_order(int(Mt), int(Nt),
                                      out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)))
    if rc != 0:
        raise RuntimeError("oracle_gilbert_order(%d, %d) failed with %d" % (Mt, Nt, rc))
    return out


def _bf16_bits(x) -> np.ndarray:
    """Accept a torch bf16 tensor or a uint16 array of bf16 bit patterns."""
    if hasattr(x, "dtype") and str(x.dtype) == "torch.bfloat16":
        import torch
        return x.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)
    arr = np.ascontiguousarray(x)
    if arr.dtype != np.uint16:
        raise TypeError("expected bf16 bit patterns (uint16) or a torch.bfloat16 tensor")
    return arr


def gemm_f64(A, B) -> np.ndarray:
    """C = A @ B in fp64 over bf16 inputs (row-major, dense)."""
    a = _bf16_bits(A)
    b = _bf16_bits(B)
    M, K = a.shape
    K2, N = b.shape
    if K != K2:
        raise ValueError("inner dimensions differ")
    C = np.empty((M, N), dtype=np.float64)
    _load().oracle_gemm_f64(M, N, K, a.ctypes.data, K, b.ctypes.data, N, C.ctypes.data, N)
    return C


def gemm_sub_f64(A, B, rows=None, cols=None, k0: int = 0, k1: int | None = None) -> np.ndarray:
    """Rows ``rows`` x columns ``cols`` of A[:, k0:k1] @ B[k0:k1, :] in fp64."""
    a = _bf16_bits(A)
    b = _bf16_bits(B)
    M, K = a.shape
    N = b.shape[1]
    rows = np.arange(M, dtype=np.int64) if rows is None else np.ascontiguousarray(rows, dtype=np.int64)
    cols = np.arange(N, dtype=np.int64) if cols is None else np.ascontiguousarray(cols, dtype=np.int64)
    if k1 is None:
        k1 = K
    if not (0 <= k0 <= k1 <= K):
        raise ValueError("bad k range")
    if rows.size and (rows.min() < 0 or rows.max() >= M):
        raise ValueError("row index out of range")
    if cols.size and (cols.min() < 0 or cols.max() >= N):
        raise ValueError("column index out of range")
    out = np.empty((rows.size, cols.size), dtype=np.float64)
    _load().oracle_gemm_sub_f64(rows.ctypes.data, rows.size, cols.ctypes.data, cols.size,
                                int(k0), int(k1), a.ctypes.data, K, b.ctypes.data, N,
                                out.ctypes.data)
    return out


def gemm_affine_f64(A, B, *, b_layout: str = "kn", beta: float = 0.0, C_in=None, bias=None) -> np.ndarray:
    """C = A @ B + beta * C_in + bias (broadcast over rows) in fp64 -- an
    extension beyond the paper.  B is K x N (``b_layout="kn"``) or its
    transpose N x K (``"nk"``).  C_in (M x N) and bias (N) are float arrays;
    either may be None (term left out)."""
    a = _bf16_bits(A)
    b = _bf16_bits(B)
    M, K = a.shape
    if b_layout == "kn":
        K2, N = b.shape
        nk = 0
    elif b_layout == "nk":
        N, K2 = b.shape
        nk = 1
    else:
        raise ValueError("b_layout must be 'kn' or 'nk'")
    if K != K2:
        raise ValueError("inner dimensions differ")
    cin = None if C_in is None else np.ascontiguousarray(C_in, dtype=np.float64)
    if cin is not None and cin.shape != (M, N):
        raise ValueError("C_in must be M x N")
    bv = None if bias is None else np.ascontiguousarray(bias, dtype=np.float64)
    if bv is not None and bv.shape != (N,):
        raise ValueError("bias must have N entries")
    C = np.empty((M, N), dtype=np.float64)
    _load().oracle_gemm_affine_f64(M, N, K, a.ctypes.data, K, b.ctypes.data, b.shape[1], nk, float(beta),
                                   None if cin is None else cin.ctypes.data, N,
                                   None if bv is None else bv.ctypes.data, C.ctypes.data, N)
    return C


F8_FORMATS = {"e4m3": 1, "e5m2": 2}


def decode_f8(code: int, fmt: str) -> float:
    """Exact value of one 8-bit float code (0..255) of format "e4m3" or "e5m2"."""
    return float(_load().oracle_decode_f8(int(code), F8_FORMATS[fmt]))


def _f8_bytes(x) -> np.ndarray:
    """Accept a torch float8 tensor or a uint8 array of codes."""
    if hasattr(x, "dtype") and str(x.dtype).startswith("torch.float8"):
        import torch
        return x.detach().cpu().contiguous().view(torch.uint8).numpy()
    arr = np.ascontiguousarray(x)
    if arr.dtype != np.uint8:
        raise TypeError("expected 8-bit float codes (uint8) or a torch float8 tensor")
    return arr


def gemm_f8_f64(A, B, fmt: str, *, b_layout: str = "kn") -> np.ndarray:
    """C = A @ B in fp64 over 8-bit float inputs of format ``fmt`` ("e4m3" or
    "e5m2"); B is K x N (``"kn"``) or its transpose N x K (``"nk"``)."""
    a = _f8_bytes(A)
    b = _f8_bytes(B)
    M, K = a.shape
    if b_layout == "kn":
        K2, N = b.shape
    elif b_layout == "nk":
        N, K2 = b.shape
    else:
        raise ValueError("b_layout must be 'kn' or 'nk'")
    if K != K2:
        raise ValueError("inner dimensions differ")
    C = np.empty((M, N), dtype=np.float64)
    _load().oracle_gemm_f8_f64(M, N, K, a.ctypes.data, K, b.ctypes.data, b.shape[1], 1 if b_layout == "nk" else 0,
                               F8_FORMATS[fmt], C.ctypes.data, N)
    return C


def round_bf16_bits(x) -> np.ndarray:
    """Round doubles to bf16 (nearest, ties to even); uint16 bit patterns."""
    flat = np.ascontiguousarray(np.asarray(x, dtype=np.float64).ravel())
    bits = np.empty(flat.size, dtype=np.uint16)
    _load().oracle_round_bf16_array(flat.ctypes.data, flat.size, bits.ctypes.data)
    return bits.reshape(np.shape(x))


def round_bf16(x) -> np.ndarray:
    """Round doubles to bf16 (nearest, ties to even), returned as float64 values."""
    bits = round_bf16_bits(x)
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def set_threads(n: int) -> None:
    """Run the oracle's parallel loops on ``n`` host threads from now on."""
    _load().oracle_set_threads(int(n))


def max_threads() -> int:
    """Threads the oracle's next parallel loop will use."""
    return int(_load().oracle_max_threads())
