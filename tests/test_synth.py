"""The seeded input generator shared by the tests and the benchmark: the same
seed gives the same bits, A is drawn before B from one generator, and each
recipe has the distribution the workloads state (CPU only)."""
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


def test_a_is_drawn_before_b_from_one_generator():
    g = torch.Generator().manual_seed(11)
    A_ref = (torch.rand((40, 24), generator=g) * 2 - 1).to(torch.bfloat16)
    B_ref = (torch.rand((24, 56), generator=g) * 2 - 1).to(torch.bfloat16)
    A, B = synth.gemm_inputs(40, 56, 24, "uniform", seed=11)
    assert torch.equal(A, A_ref) and torch.equal(B, B_ref)


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
