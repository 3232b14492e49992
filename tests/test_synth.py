"""The seeded input generator shared by the tests and the benchmark: the same
seed gives the same bits, each 2^22-element block of an operand comes from its
own generator seeded as the module states (so the bits do not depend on the
number of threads), and each recipe has the distribution the workloads state
(CPU only)."""
import pytest
import torch

from paper_2601_16294_gb300 import synth


def test_same_seed_same_bits_other_seed_other_bits():
    A1, B1 = synth.gemm_inputs(64, 48, 32, "uniform", seed=5)
    A2, B2 = synth.gemm_inputs(64, 48, 32, "uniform", seed=5)
    A3, _ = synth.gemm_inputs(64, 48, 32, "uniform", seed=6)
    assert torch.equal(A1.view(torch.int16), A2.view(torch.int16)) and torch.equal(B1.view(torch.int16),
                                                                                  B2.view(torch.int16))
    assert not torch.equal(A1, A3)


def test_blocks_follow_the_stated_seeds():
    # A (operand 0) spans two blocks and a ragged third; B is operand 1
    M, K, N = 3000, 3000, 24
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=11)
    flat = A.reshape(-1)
    n = M * K
    assert n > 2 * synth.BLOCK
    for b in range(3):
        g = torch.Generator().manual_seed(((11 * 1000003 + 0) * 1000003 + b) % (1 << 63))
        lo, hi = b * synth.BLOCK, min(n, (b + 1) * synth.BLOCK)
        want = (torch.rand(hi - lo, generator=g) * 2 - 1).to(torch.bfloat16)
        assert torch.equal(flat[lo:hi], want)
    g = torch.Generator().manual_seed((11 * 1000003 + 1) * 1000003)
    assert torch.equal(B.reshape(-1), (torch.rand(K * N, generator=g) * 2 - 1).to(torch.bfloat16))
    # the prefill weights: N(0, 1) draws times 0.02, rounded once
    _, Bp = synth.gemm_inputs(8, 16, 32, "prefill", seed=3)
    g = torch.Generator().manual_seed((3 * 1000003 + 1) * 1000003)
    assert torch.equal(Bp.reshape(-1), (torch.randn(32 * 16, generator=g) * 0.02).to(torch.bfloat16))


def test_bits_do_not_depend_on_threads():
    one = synth.draw((2100, 4100), 9, 1, "normal", 0.02, threads=1)
    many = synth.draw((2100, 4100), 9, 1, "normal", 0.02, threads=7)
    assert torch.equal(one.view(torch.int16), many.view(torch.int16))


def test_uniform_recipe():
    A, B = synth.gemm_inputs(512, 512, 512, "uniform", seed=1)
    for t in (A.float(), B.float()):
        assert t.min() >= -1.0 and t.max() <= 1.0
        assert abs(t.mean().item()) < 0.01
        assert abs(t.std().item() - 3 ** -0.5) < 0.01          # U[-1, 1]: sd 1/sqrt(3)


def test_prefill_recipe():
    A, B = synth.gemm_inputs(512, 512, 1024, "prefill", seed=2)
    assert abs(A.float().std().item() - 1.0) < 0.02 and abs(A.float().mean().item()) < 0.01
    assert abs(B.float().std().item() - 0.02) < 0.0005 and abs(B.float().mean().item()) < 0.0005


def test_integer_recipe():
    A, B = synth.gemm_inputs(300, 200, 100, "int", seed=3)
    for t in (A.float(), B.float()):
        vals = set(torch.unique(t).tolist())
        assert vals == {-2.0, -1.0, 0.0, 1.0, 2.0}


def test_padded_rows_hold_the_same_values():
    A0, B0 = synth.gemm_inputs(30, 21, 13, "uniform", seed=4)
    A, B = synth.gemm_inputs(30, 21, 13, "uniform", seed=4, lda=16, ldb=24)
    assert A.stride() == (16, 1) and B.stride() == (24, 1)
    assert torch.equal(A, A0) and torch.equal(B, B0)
    assert torch.count_nonzero(A.as_strided((30, 16), (16, 1))[:, 13:]) == 0


@pytest.mark.parametrize("fmt", ["e4m3", "e5m2"])
def test_eight_bit_inputs(fmt):
    A, B = synth.gemm_inputs_f8(64, 32, 128, fmt, "int", seed=7)
    assert A.dtype == synth.f8_dtype(fmt) and B.dtype == synth.f8_dtype(fmt)
    assert set(torch.unique(A.float()).tolist()) <= {-2.0, -1.0, 0.0, 1.0, 2.0}
    U, _ = synth.gemm_inputs_f8(64, 32, 128, fmt, "uniform", seed=7)
    assert U.float().abs().max() <= 1.0


def test_unknown_kind_and_pad8():
    with pytest.raises(ValueError):
        synth.gemm_inputs(4, 4, 4, "cauchy")
    assert [synth.pad8(n) for n in (1, 8, 9, 4096, 4097)] == [8, 8, 16, 4096, 4104]
