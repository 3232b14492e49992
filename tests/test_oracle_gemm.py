"""Pins for the oracle GEMM (Sec. II-A, Listing 1: C = A * B, C zeroed first).

Each check has an answer fixed by mathematics, not by re-running the oracle:
identity and permutation matrices, a rank-1 closed form, exact integer
products, brute force in exact rational arithmetic, and K-range additivity (the
K split of the communication-avoiding scheme, Sec. II-C/D, only regroups the
sum).
"""
from fractions import Fraction

import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth


def bf16_bits(t):
    return t.contiguous().view(torch.int16).numpy().view(np.uint16)


def bf16_values(t):
    return t.float().numpy().astype(np.float64)


def test_identity_left_and_right(oracle):
    B = synth.uniform_bf16((48, 40), seed=3)
    I48 = torch.eye(48, dtype=torch.bfloat16)
    I40 = torch.eye(40, dtype=torch.bfloat16)
    assert np.array_equal(oracle.gemm_f64(I48, B), bf16_values(B))      # I * B = B
    assert np.array_equal(oracle.gemm_f64(B, I40), bf16_values(B))      # B * I = B


def test_permutation_matrices(oracle):
    g = np.random.default_rng(7)
    X = synth.uniform_bf16((24, 36), seed=5)
    prow = g.permutation(24)
    pcol = g.permutation(36)
    P = torch.zeros(24, 24, dtype=torch.bfloat16)
    P[np.arange(24), prow] = 1              # (P X)[i] = X[prow[i]]
    Q = torch.zeros(36, 36, dtype=torch.bfloat16)
    Q[pcol, np.arange(36)] = 1              # (X Q)[:, j] = X[:, pcol[j]]
    xv = bf16_values(X)
    assert np.array_equal(oracle.gemm_f64(P, X), xv[prow, :])
    assert np.array_equal(oracle.gemm_f64(X, Q), xv[:, pcol])


def test_rank_one_closed_form(oracle):
    # A[i][k] = x_i, B[k][j] = y_j  =>  C[i][j] = K x_i y_j exactly.
    M, N, K = 9, 13, 777
    x = np.array([(i - 4) * 0.25 for i in range(M)])
    y = np.array([(j - 6) * 0.125 for j in range(N)])
    A = torch.tensor(np.repeat(x[:, None], K, axis=1), dtype=torch.bfloat16)
    B = torch.tensor(np.repeat(y[None, :], K, axis=0), dtype=torch.bfloat16)
    assert np.array_equal(oracle.gemm_f64(A, B), K * np.outer(x, y))


def test_small_integers_exact(oracle):
    # Entries in {-2..2}: every partial sum is an integer of magnitude <= 4K,
    # so the fp64 result must equal the exact integer product.
    A = synth.small_int_bf16((70, 130), seed=1)
    B = synth.small_int_bf16((130, 50), seed=2)
    ai = A.float().numpy().astype(np.int64)
    bi = B.float().numpy().astype(np.int64)
    exact = ai @ bi
    assert np.array_equal(oracle.gemm_f64(A, B), exact.astype(np.float64))


def test_brute_force_4x4x4_exact_rationals(oracle):
    # Brute force with exact rational arithmetic (j-k-i order, no floats).
    for seed in range(5):
        A = synth.uniform_bf16((4, 4), seed=10 + seed)
        B = synth.uniform_bf16((4, 4), seed=20 + seed)
        a = [[Fraction(float(v)) for v in row] for row in bf16_values(A)]
        b = [[Fraction(float(v)) for v in row] for row in bf16_values(B)]
        C = oracle.gemm_f64(A, B)
        for j in range(4):
            for i in range(4):
                exact = Fraction(0)
                mag = Fraction(0)
                for k in range(4):
                    exact += a[i][k] * b[k][j]
                    mag += abs(a[i][k] * b[k][j])
                # fp64 sum of 4 exact products: error <= 4 * 2^-53 * sum|terms|
                assert abs(Fraction(C[i, j]) - exact) <= 4 * Fraction(1, 2 ** 53) * mag


def test_accumulates_in_double(oracle):
    # 2^24 + 1 - 2^24 = 1 needs more than fp32's 24 significant bits.
    A = torch.tensor([[2.0 ** 24, 1.0, -(2.0 ** 24)]], dtype=torch.bfloat16)
    B = torch.ones(3, 1, dtype=torch.bfloat16)
    assert oracle.gemm_f64(A, B)[0, 0] == 1.0


def test_sub_rows_cols_and_k_ranges(oracle):
    A = synth.small_int_bf16((33, 200), seed=4)
    B = synth.small_int_bf16((200, 29), seed=5)
    full = oracle.gemm_f64(A, B)
    rows = np.array([0, 5, 32, 17])
    cols = np.array([28, 0, 3])
    assert np.array_equal(oracle.gemm_sub_f64(A, B, rows, cols), full[np.ix_(rows, cols)])
    # K split into c layers (balanced ranges) sums back to the full product.
    for c in (2, 3, 8):
        bounds = [(l * 200) // c for l in range(c + 1)]
        parts = [oracle.gemm_sub_f64(A, B, None, None, bounds[l], bounds[l + 1]) for l in range(c)]
        assert np.array_equal(sum(parts), full)


def test_round_bf16_single_step(oracle):
    one = 1.0
    ulp = 2.0 ** -7                      # bf16 spacing in [1, 2)
    cases = {
        1.0: 1.0,
        one + ulp / 2: 1.0,              # tie -> even (1.0)
        one + 3 * ulp / 2: one + 2 * ulp,  # tie -> even (1 + 2 ulp)
        one + ulp / 2 + 2.0 ** -40: one + ulp,  # above the tie: a two-step
                                         # double->fp32->bf16 rounding gets 1.0
        -(one + ulp / 2 + 2.0 ** -40): -(one + ulp),
        0.0: 0.0,
        3.4e38: float("inf"),            # beyond max bf16 + half an ulp -> inf
        2.0 ** 127 * (2 - 2.0 ** -7): 2.0 ** 127 * (2 - 2.0 ** -7),  # largest finite bf16
    }
    for v, want in cases.items():
        assert oracle.round_bf16(np.array([v]))[0] == want, v
    # Where fp32 is exact, it agrees with torch's round-to-nearest-even cast.
    vals = torch.randn(5000, generator=torch.Generator().manual_seed(0), dtype=torch.float32) * 100
    ref = vals.to(torch.bfloat16).float().numpy().astype(np.float64)
    assert np.array_equal(oracle.round_bf16(vals.numpy().astype(np.float64)), ref)


# --- the BLAS-style extension: transposed B, beta * C_in, bias (no paper counterpart)

def test_affine_without_terms_is_the_plain_product(oracle):
    A, B = synth.gemm_inputs(37, 29, 53, "uniform", seed=3)
    plain = oracle.gemm_f64(A, B)
    assert np.array_equal(oracle.gemm_affine_f64(A, B), plain)
    # the transposed storage of the same B gives the same sums in the same order
    assert np.array_equal(oracle.gemm_affine_f64(A, B.t().contiguous(), b_layout="nk"), plain)


def test_affine_closed_forms(oracle):
    M, N, K = 12, 20, 12
    Bt = synth.uniform_bf16((N, K), seed=9)              # B stored transposed
    C_in = np.arange(M * N, dtype=np.float64).reshape(M, N) / 8.0
    bias = np.linspace(-3.0, 3.0, N)
    I = torch.eye(M, dtype=torch.bfloat16)
    # A = I: C = B = Bt^T exactly, then + bias
    assert np.array_equal(oracle.gemm_affine_f64(I, Bt, b_layout="nk"), bf16_values(Bt).T)
    assert np.array_equal(oracle.gemm_affine_f64(I, Bt, b_layout="nk", bias=bias), bf16_values(Bt).T + bias)
    # A = 0: only the affine terms remain
    Z = torch.zeros(M, K, dtype=torch.bfloat16)
    got = oracle.gemm_affine_f64(Z, Bt, b_layout="nk", beta=-2.5, C_in=C_in, bias=bias)
    assert np.array_equal(got, -2.5 * C_in + bias)


def test_affine_small_integers_exact(oracle):
    M, N, K = 33, 18, 70
    A, B = synth.gemm_inputs(M, N, K, "int", seed=21)
    g = np.random.default_rng(4)
    C_in = g.integers(-50, 50, size=(M, N)).astype(np.float64)
    bias = g.integers(-9, 9, size=N).astype(np.float64)
    ai = bf16_values(A).astype(np.int64)
    bi = bf16_values(B).astype(np.int64)
    want = (ai @ bi) + 3 * C_in.astype(np.int64) + bias.astype(np.int64)
    for layout, b in (("kn", B), ("nk", B.t().contiguous())):
        got = oracle.gemm_affine_f64(A, b, b_layout=layout, beta=3.0, C_in=C_in, bias=bias)
        assert np.array_equal(got, want.astype(np.float64)), layout


# --- 8-bit float inputs (the method is independent of the data type, Sec. III)

@pytest.mark.parametrize("fmt,tdtype", [("e4m3", "float8_e4m3fn"), ("e5m2", "float8_e5m2")])
def test_f8_decode_matches_the_library_format_for_every_code(oracle, fmt, tdtype):
    # torch's float8 -> float32 conversion is an independent implementation of the formats
    codes = torch.arange(256, dtype=torch.int32).to(torch.uint8)
    ref = codes.view(getattr(torch, tdtype)).float().numpy().astype(np.float64)
    got = np.array([oracle.decode_f8(c, fmt) for c in range(256)])
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.array_equal(got[~nan], ref[~nan])


def test_f8_decode_fixed_points(oracle):
    # values the format definitions fix
    assert oracle.decode_f8(0x38, "e4m3") == 1.0
    assert oracle.decode_f8(0xC0, "e4m3") == -2.0
    assert oracle.decode_f8(0x7E, "e4m3") == 448.0           # largest finite e4m3
    assert oracle.decode_f8(0x01, "e4m3") == 2.0 ** -9       # smallest subnormal
    assert np.isnan(oracle.decode_f8(0x7F, "e4m3"))
    assert oracle.decode_f8(0x3C, "e5m2") == 1.0
    assert oracle.decode_f8(0x7B, "e5m2") == 57344.0         # largest finite e5m2
    assert oracle.decode_f8(0x01, "e5m2") == 2.0 ** -16
    assert oracle.decode_f8(0x7C, "e5m2") == float("inf")


@pytest.mark.parametrize("fmt", ["e4m3", "e5m2"])
def test_f8_gemm_small_integers_exact(oracle, fmt):
    M, N, K = 21, 34, 90
    A, B = synth.gemm_inputs_f8(M, N, K, fmt, "int", seed=6)
    ai = A.float().numpy().astype(np.int64)
    bi = B.float().numpy().astype(np.int64)
    assert set(np.unique(ai)) <= {-2, -1, 0, 1, 2}
    want = (ai @ bi).astype(np.float64)
    assert np.array_equal(oracle.gemm_f8_f64(A, B, fmt), want)
    assert np.array_equal(oracle.gemm_f8_f64(A, B.t().contiguous(), fmt, b_layout="nk"), want)


def test_f8_gemm_equals_bf16_gemm_of_the_same_values(oracle):
    # every e4m3 value is a bf16 value, so the bf16 oracle on the widened inputs gives the same sums
    A, B = synth.gemm_inputs_f8(17, 23, 61, "e4m3", "uniform", seed=2)
    assert np.array_equal(oracle.gemm_f8_f64(A, B, "e4m3"),
                          oracle.gemm_f64(A.float().to(torch.bfloat16), B.float().to(torch.bfloat16)))
