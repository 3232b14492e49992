"""The oracle's pins catch plausible mistakes.

Each case plants one mistake in a private copy of ``oracle/oracle.c`` (on the
CPU, in a temporary directory), builds it, and checks that the same kinds of
pin the real oracle passes (adjacency, bijection, the classical Hilbert curve,
identity / permutation / exact-integer products) now fail.
"""
import ctypes
import os
import subprocess

import numpy as np
import pytest

SRC = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "oracle", "oracle.c")

MUTATIONS = {
    "no_parity_rule": ("if ((longer % 2) == 1 && (shorter % 2) == 0) x_major = !x_major;", ""),
    "no_even_split_long": ("if ((length_of(a_first) % 2) == 1 && la > 2) a_first = add(a_first, ua);", ""),
    "no_even_split_minor": ("if ((length_of(b_first) % 2) == 1 && lb > 2) b_first = add(b_first, ub);", ""),
    "far_corner_off_by_one": ("add(add(o, sub(a, ua)), sub(b_first, ub))", "add(add(o, a), sub(b_first, ub))"),
    "corner_axes_not_exchanged": ("walk_region(st, o, b_first, a_first);", "walk_region(st, o, a_first, b_first);"),
    "return_not_negated": ("walk_region(st, far, neg(b_first), neg(a_rest));",
                           "walk_region(st, far, b_first, neg(a_rest));"),
    "gemm_drops_first_k": ("for (int64_t k = 0; k < K; ++k) {\n            double a = widen_bf16(A[i * lda + k]);",
                           "for (int64_t k = 1; k < K; ++k) {\n            double a = widen_bf16(A[i * lda + k]);"),
    "gemm_transposed_b": ("c[j] += a * widen_bf16(b[j]);", "c[j] += a * widen_bf16(B[j * ldb + k]);"),
    "gemm_not_zeroed": ("for (int64_t j = 0; j < N; ++j) c[j] = 0.0;", ""),
    "gemm_wrong_sign": ("c[j] += a * widen_bf16(b[j]);", "c[j] -= a * widen_bf16(b[j]);"),
}


def _build_mutant(tmp_path, name):
    text = open(SRC).read()
    if name in MUTATIONS:
        old, new = MUTATIONS[name]
        assert text.count(old) == 1, "mutation anchor for %s not found exactly once" % name
        text = text.replace(old, new)
    src = tmp_path / ("%s.c" % name)
    src.write_text(text)
    so = tmp_path / ("%s.so" % name)
    subprocess.run(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-ffp-contract=off", "-o", str(so),
                    str(src), "-lm"], check=True)
    lib = ctypes.CDLL(str(so))
    lib.oracle_gilbert_order.argtypes = [ctypes.c_int, ctypes.c_int, ctypes.c_void_p]
    lib.oracle_gilbert_order.restype = ctypes.c_int
    i64 = ctypes.c_int64
    lib.oracle_gemm_f64.argtypes = [i64, i64, i64, ctypes.c_void_p, i64, ctypes.c_void_p, i64,
                                    ctypes.c_void_p, i64]
    return lib


def _curve_pins_pass(lib):
    def order(Mt, Nt):
        out = np.full(Mt * Nt, -1, dtype=np.int32)
        rc = lib.oracle_gilbert_order(Mt, Nt, out.ctypes.data)
        return rc, out

    for Mt in range(1, 20):
        for Nt in range(1, 20):
            rc, o = order(Mt, Nt)
            if rc != 0 or not np.array_equal(np.sort(o), np.arange(Mt * Nt)):
                return False
            tm, tn = o // Nt, o % Nt
            if tm[0] != 0 or tn[0] != 0:
                return False
            if np.any(np.abs(np.diff(tm)) + np.abs(np.diff(tn)) != 1):
                return False
    return True


def _gemm_pins_pass(lib):
    rng = np.random.default_rng(0)

    def gemm(a, b):
        a16 = (np.asarray(a, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)
        b16 = (np.asarray(b, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)
        M, K = a.shape
        N = b.shape[1]
        C = np.full((M, N), 123.0)
        lib.oracle_gemm_f64(M, N, K, a16.ctypes.data, K, b16.ctypes.data, N, C.ctypes.data, N)
        return C

    I = np.eye(8)
    X = rng.integers(-2, 3, size=(8, 11)).astype(np.float64)
    perm = rng.permutation(8)
    P = np.zeros((8, 8))
    P[np.arange(8), perm] = 1
    Y = rng.integers(-2, 3, size=(11, 5)).astype(np.float64)
    return (np.array_equal(gemm(I, X), X) and np.array_equal(gemm(P, X), X[perm])
            and np.array_equal(gemm(X, Y), X @ Y))


def test_unmutated_copy_passes(tmp_path):
    lib = _build_mutant(tmp_path, "unmutated")
    assert _curve_pins_pass(lib) and _gemm_pins_pass(lib)


@pytest.mark.parametrize("name", sorted(k for k in MUTATIONS if not k.startswith("gemm")))
def test_curve_mutation_caught(tmp_path, name):
    assert not _curve_pins_pass(_build_mutant(tmp_path, name))


@pytest.mark.parametrize("name", sorted(k for k in MUTATIONS if k.startswith("gemm")))
def test_gemm_mutation_caught(tmp_path, name):
    assert not _gemm_pins_pass(_build_mutant(tmp_path, name))
