"""Full-size parity: every shape of the five benchmark configurations, run the
way bench.py runs it (curve order, automatic assignment and tile width), checked
on sampled rows and columns the oracle computes one by one.

Sampled rows / columns always include the first and last, both sides of a
tile boundary and the ragged tail, plus seeded random ones.  Tolerances are
those of parity.py (R8 / R9 readings for bf16 output and the prefill
distribution).
"""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import bf16_ulp, rel_frobenius

pytestmark = pytest.mark.gpu

CONFIGS = {
    "square": [(n, n, n, "uniform", "bf16", (1,)) for n in (2048, 4096, 8192, 16384)],
    "prefill": [(m, n, k, "prefill", "bf16", (1, 4)) for m in (512, 2048, 8192)
                for (n, k) in ((4096, 4096), (14336, 4096), (4096, 14336), (128256, 4096))],
    "irregular": [(3000, 5000, 7000, "uniform", "bf16", (1, 4)), (1000, 17000, 2500, "uniform", "bf16", (1, 4)),
                  (6144, 768, 12288, "uniform", "bf16", (1, 4)), (129, 8191, 4096, "uniform", "bf16", (1, 4))],
    "highk": [(m, m, k, "uniform", "f32", (1, 2, 4, 8)) for m in (512, 1024, 2048)
              for k in (32768, 65536, 131072)],
}
CASES = [(name, shape) for name, shapes in CONFIGS.items() for shape in shapes]


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def sample_indices(n, seed, extra=4):
    idx = {0, n - 1, min(127, n - 1), min(128, n - 1), min(255, n - 1), min(256, n - 1), (n // 2)}
    g = np.random.default_rng(seed)
    idx.update(int(x) for x in g.integers(0, n, size=extra))
    return np.array(sorted(idx), dtype=np.int64)


def dev(t):
    full = t.as_strided((t.shape[0], t.stride(0)), (t.stride(0), 1))
    return full.contiguous().cuda()[:, : t.shape[1]]


def check_samples(oracle, got, ref, ref_mag, K, out):
    """got / ref / ref_mag: the same sampled entries (got widened to fp64)."""
    bound = 2e-6 * ref_mag if ref_mag is not None else 2e-6 * K
    if out == "f32":
        assert rel_frobenius(got, ref) <= 1e-5
        assert np.all(np.abs(got - ref) <= bound)
    else:
        rounded = oracle.round_bf16(ref)
        ok = (np.abs(got - rounded) <= bf16_ulp(rounded)) | (np.abs(got - ref) <= bound)
        assert np.all(ok), "%d sampled bf16 entries off by more than 1 ulp" % int((~ok).sum())


@pytest.mark.parametrize("name,shape", CASES, ids=["%s-%dx%dx%d" % (n, s[0], s[1], s[2]) for n, s in CASES])
def test_full_size_sampled(sfc, oracle, name, shape):
    M, N, K, kind, out, cs = shape
    lda, ldb = synth.pad8(K), synth.pad8(N)
    A, B = synth.gemm_inputs(M, N, K, kind, seed=0, lda=lda, ldb=ldb)
    rows = sample_indices(M, seed=M + K)
    cols = sample_indices(N, seed=N + K)
    Ac, Bc = A.contiguous(), B.contiguous()
    ref_rows = oracle.gemm_sub_f64(Ac, Bc, rows, None)
    ref_cols = oracle.gemm_sub_f64(Ac, Bc, None, cols)
    mag_rows = mag_cols = None
    if kind == "prefill":
        absA = Ac.float().abs().to(torch.bfloat16)
        absB = Bc.float().abs().to(torch.bfloat16)
        mag_rows = oracle.gemm_sub_f64(absA, absB, rows, None)
        mag_cols = oracle.gemm_sub_f64(absA, absB, None, cols)
    Ad, Bd = dev(A), dev(B)
    del A, B, Ac, Bc
    out_dtype = torch.float32 if out == "f32" else torch.bfloat16
    C = torch.empty((M, N), dtype=out_dtype, device="cuda")
    Kt = (K + 63) // 64
    rows_t = torch.from_numpy(rows).cuda()
    cols_t = torch.from_numpy(cols).cuda()
    for c in [c for c in cs if c <= Kt]:
        C.fill_(float("nan"))
        sfc.gemm(Ad, Bd, C, ca_c=c)
        torch.cuda.synchronize()
        assert sfc.device_status() == 0
        got_rows = C.index_select(0, rows_t).double().cpu().numpy()
        got_cols = C.index_select(1, cols_t).double().cpu().numpy()
        check_samples(oracle, got_rows, ref_rows, mag_rows, K, out)
        check_samples(oracle, got_cols, ref_cols, mag_cols, K, out)
        # whole output written, nothing non-finite
        assert torch.isfinite(C).all().item()
