"""Full-size parity: every shape of the four measured configurations (square,
prefill, irregular, high-K), run the way bench.py runs them (curve order,
automatic dealing and tile), against the fp64 oracle.

Where 2 M N K <= 1.2e12 the whole of C is compared with the oracle's whole C,
element by element.  Larger shapes (16384^3, 2048 x 128256 x 4096 and
8192 x 128256 x 4096) are compared on at least 256 full rows and 256 full
columns of C: the first and last, both sides of every multiple of 256 (and so
of 512) -- the tile edges of every tile shape, including the ragged tail --
and seeded random ones up to 256.  C is filled with NaN before each call and
must come back finite everywhere, so an unwritten tile fails even where no
sample falls.

Tolerances are those of parity.py: fp32 output within the relative Frobenius
and 2e-6 K bounds, bf16 output within one bf16 ulp of RNE(C_ref) (or the fp32
bound where cancellation makes C_ref tiny), and for the prefill distribution
the bound 2e-6 sum_k |A_ik| |B_kj| from the oracle's |A| @ |B|.
"""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import bf16_ulp, rel_frobenius

pytestmark = pytest.mark.gpu

FULL_FLOP_LIMIT = 1.2e12  # 2 M N K up to which the whole of C is checked
EDGE = 256                # tile edges: every tile's rows and columns are multiples of 128 or 256

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


def is_full(M, N, K):
    return 2.0 * M * N * K <= FULL_FLOP_LIMIT


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def sample_indices(n, seed, want=256):
    """Sorted indices into 0..n-1: first, last, both sides of every multiple of
    EDGE, then seeded random ones until there are at least `want` (or n)."""
    idx = {0, n - 1}
    for e in range(EDGE, n, EDGE):
        idx.update((e - 1, e))
    g = np.random.default_rng(seed)
    while len(idx) < min(want, n):
        idx.add(int(g.integers(0, n)))
    return np.array(sorted(idx), dtype=np.int64)


def test_sample_indices_cover_edges_and_count():
    r = sample_indices(16384, seed=1)
    assert r.size >= 256 and r[0] == 0 and r[-1] == 16383
    for e in range(256, 16384, 256):
        assert e - 1 in r and e in r
    c = sample_indices(128256, seed=2)
    assert 128255 in c and 128000 in c and 127999 in c and c.size >= 256
    assert sample_indices(129, seed=3).size == 129  # fewer than 256: every index


def dev(t):
    full = t.as_strided((t.shape[0], t.stride(0)), (t.stride(0), 1))
    return full.contiguous().cuda()[:, : t.shape[1]]


def check(oracle, got, ref, ref_mag, K, out):
    """got / ref / ref_mag: the same entries of C (got widened to fp64)."""
    bound = 2e-6 * ref_mag if ref_mag is not None else 2e-6 * K
    if out == "f32":
        rf = rel_frobenius(got, ref)
        assert rf <= 1e-5, "relative Frobenius error %.3e" % rf
        bad = np.abs(got - ref) > bound
        assert not bad.any(), "%d entries beyond the bound (worst %.3e)" % (
            int(bad.sum()), float(np.abs(got - ref).max()))
    else:
        rounded = oracle.round_bf16(ref)
        ok = (np.abs(got - rounded) <= bf16_ulp(rounded)) | (np.abs(got - ref) <= bound)
        assert ok.all(), "%d bf16 entries off by more than 1 ulp" % int((~ok).sum())


@pytest.mark.parametrize("name,shape", CASES, ids=["%s-%dx%dx%d" % (n, s[0], s[1], s[2]) for n, s in CASES])
def test_full_size(sfc, oracle, name, shape):
    M, N, K, kind, out, cs = shape
    lda, ldb = synth.pad8(K), synth.pad8(N)
    A, B = synth.gemm_inputs(M, N, K, kind, seed=0, lda=lda, ldb=ldb)
    Ac, Bc = A.contiguous(), B.contiguous()
    absA = absB = None
    if kind == "prefill":
        absA = Ac.float().abs().to(torch.bfloat16)  # exact: |x| of a bf16 value is a bf16 value
        absB = Bc.float().abs().to(torch.bfloat16)
    full = is_full(M, N, K)
    if full:
        refs = [(None, None, oracle.gemm_f64(Ac, Bc), oracle.gemm_f64(absA, absB) if absA is not None else None)]
    else:
        rows = sample_indices(M, seed=M + K)
        cols = sample_indices(N, seed=N + K)
        refs = [(rows, None, oracle.gemm_sub_f64(Ac, Bc, rows, None),
                 oracle.gemm_sub_f64(absA, absB, rows, None) if absA is not None else None),
                (None, cols, oracle.gemm_sub_f64(Ac, Bc, None, cols),
                 oracle.gemm_sub_f64(absA, absB, None, cols) if absA is not None else None)]
    Ad, Bd = dev(A), dev(B)
    del A, B, Ac, Bc, absA, absB
    out_dtype = torch.float32 if out == "f32" else torch.bfloat16
    C = torch.empty((M, N), dtype=out_dtype, device="cuda")
    Kt = (K + 63) // 64
    for c in [c for c in cs if c <= Kt]:
        C.fill_(float("nan"))
        sfc.gemm(Ad, Bd, C, ca_c=c)
        torch.cuda.synchronize()
        assert sfc.device_status() == 0
        assert torch.isfinite(C).all().item(), "unwritten or non-finite entries (ca_c=%d)" % c
        for rows, cols, ref, mag in refs:
            if rows is None and cols is None:
                got = C.double().cpu().numpy()
            elif rows is not None:
                got = C.index_select(0, torch.from_numpy(rows).cuda()).double().cpu().numpy()
            else:
                got = C.index_select(1, torch.from_numpy(cols).cuda()).double().cpu().numpy()
            check(oracle, got, ref, mag, K, out)
