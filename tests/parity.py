"""Tolerances for comparing the CUDA GEMM with the fp64 oracle.

fp32 output, entries uniform in [-1, 1]:
    ||C - C_ref||_F / ||C_ref||_F <= 1e-5   and   max |C - C_ref| <= 2e-6 * K.
bf16 output: every entry within one bf16 ulp of RNE_bf16(C_ref); entries where
cancellation makes |C_ref| tiny may instead be within the fp32 bound 2e-6 * K
of C_ref.
Other value distributions (the prefill recipe): the relative Frobenius bound
and max |C - C_ref| <= 2e-6 * sum_k |A_ik| |B_kj|, checked as
<= 2e-6 * (|A| @ |B|) computed in fp64 by the oracle.
"""
import numpy as np


def rel_frobenius(C, ref):
    ref = np.asarray(ref, dtype=np.float64)
    num = np.linalg.norm(np.asarray(C, dtype=np.float64) - ref)
    den = np.linalg.norm(ref)
    return num / den if den > 0 else num


def check_fp32(C, ref, K, absbound=None):
    C = np.asarray(C, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    assert C.shape == ref.shape
    assert np.all(np.isfinite(C)), "non-finite output"
    rf = rel_frobenius(C, ref)
    bound = 2e-6 * K if absbound is None else absbound
    err = np.abs(C - ref)
    worst = float(err.max()) if err.size else 0.0
    assert rf <= 1e-5, "relative Frobenius error %.3e > 1e-5" % rf
    assert np.all(err <= bound), "max |C - C_ref| = %.3e exceeds bound (max bound %.3e)" % (
        worst, float(np.max(bound)))
    return rf, worst


def bf16_ulp(v):
    """Spacing of bf16 numbers at |v| (v already a bf16 value)."""
    a = np.abs(np.asarray(v, dtype=np.float32))
    a = np.where(a < np.float32(2.0 ** -126), np.float32(2.0 ** -126), a)
    return np.spacing(a).astype(np.float64) * 65536.0


def check_bf16(C_bf16_values, ref, ref_rounded, K):
    """C_bf16_values: GPU output widened to float64; ref: fp64 C_ref;
    ref_rounded: RNE_bf16(C_ref) as float64 (from the oracle)."""
    C = np.asarray(C_bf16_values, dtype=np.float64)
    within_ulp = np.abs(C - ref_rounded) <= bf16_ulp(ref_rounded)
    within_abs = np.abs(C - ref) <= 2e-6 * K
    ok = within_ulp | within_abs
    assert np.all(ok), "%d bf16 entries off by more than 1 ulp (worst %.3e)" % (
        int((~ok).sum()), float(np.abs(C - ref_rounded)[~ok].max()))
    return int(within_ulp.sum()), int((~within_ulp & within_abs).sum())
