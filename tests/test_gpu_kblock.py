"""K blocks (sfc_gemm_ex3, Listing 1's outer loop over ik with k_block_factor
passes): each pass contracts one block of every layer's K slabs and adds it
into that layer's copy of C in place.

The sum is the plain GEMM, so the oracle's definition is the reference
(tolerance for uniform data, bit for bit for integer data); the pass structure
itself is pinned by composing the same result from separate calls over the
K blocks, and the invariances of the method (curve == raster, every deal,
repeatable) hold for each (ca_c, k_block_factor).
"""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth
from parity import check_bf16, check_fp32

pytestmark = pytest.mark.gpu

TILES = [128, 256, "pair128", "pair256"]


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def padded(t, ld):
    """CUDA copy of a CPU matrix with row stride ld."""
    d = torch.zeros(t.shape[0], ld, dtype=t.dtype, device="cuda")
    d[:, : t.shape[1]] = t.cuda()
    return d[:, : t.shape[1]]


@pytest.mark.parametrize("tile", TILES)
def test_integer_inputs_bit_exact(sfc, oracle, tile):
    M, N, K = 384, 640, 1500                       # 24 slabs, tail of 28
    A, B = synth.gemm_inputs(M, N, K, "int", seed=51)
    ref = oracle.gemm_f64(A, B)
    bits = oracle.round_bf16_bits(ref)
    Ad, Bd = padded(A, synth.pad8(K)), padded(B, N)
    for c, kbf in ((1, 2), (1, 3), (2, 2), (3, 4), (1, 24), (4, 6)):
        C = sfc.gemm(Ad, Bd, ca_c=c, k_block_factor=kbf, tile=tile)
        Cb = sfc.gemm(Ad, Bd, ca_c=c, k_block_factor=kbf, tile=tile, out_dtype=torch.bfloat16)
        torch.cuda.synchronize()
        assert sfc.device_status() == 0
        assert np.array_equal(C.cpu().numpy().astype(np.float64), ref), (c, kbf)
        assert np.array_equal(Cb.cpu().view(torch.int16).numpy().view(np.uint16), bits), (c, kbf)


@pytest.mark.parametrize("M,N,K", [(200, 300, 1000), (129, 257, 4100), (640, 136, 2048), (1, 1, 200)])
def test_uniform_inputs_within_tolerance(sfc, oracle, M, N, K):
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=M + N + K)
    ref = oracle.gemm_f64(A, B)
    ref16 = oracle.round_bf16(ref)
    Ad, Bd = padded(A, synth.pad8(K)), padded(B, synth.pad8(N))
    Kt = (K + 63) // 64
    for c, kbf in ((1, 2), (2, 2), (1, 3), (3, 1)):
        if c * kbf > Kt:
            continue
        C = sfc.gemm(Ad, Bd, ca_c=c, k_block_factor=kbf)
        Cb = sfc.gemm(Ad, Bd, ca_c=c, k_block_factor=kbf, out_dtype=torch.bfloat16)
        check_fp32(C.cpu().numpy().astype(np.float64), ref, K)
        check_bf16(Cb.float().cpu().numpy().astype(np.float64), ref, ref16, K)


def test_passes_compose_from_separate_calls(sfc):
    # one layer, fp32 C, k_block_factor 3 on 20 slabs: blocks of 6, 7, 7 slabs
    # (floor(ik * 20 / 3)).  The same result comes from three calls over the
    # blocks, the later ones adding into C (beta = 1): pass ik adds its block
    # into C exactly like a beta = 1 call over that block.
    M, N, K = 500, 700, 1280
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=61)
    Ad, Bd = padded(A, K), padded(B, synth.pad8(N))
    edges = [64 * (ik * 20 // 3) for ik in range(4)]
    for tile in (128, "pair256"):
        got = sfc.gemm(Ad, Bd, ca_c=1, k_block_factor=3, tile=tile)
        C = torch.empty(M, N, dtype=torch.float32, device="cuda")
        for ik in range(3):
            k0, k1 = edges[ik], edges[ik + 1]
            sfc.gemm(Ad[:, k0:k1], Bd[k0:k1], C, ca_c=1, tile=tile, beta=0.0 if ik == 0 else 1.0)
        assert torch.equal(got, C), tile


def test_layers_compose_from_separate_calls(sfc):
    # two layers of 8 slabs, two blocks each: the layer copies are the K-block
    # sums of each layer, and C is their sum in layer order
    M, N, K = 256, 384, 1024
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=62)
    Ad, Bd = padded(A, K), padded(B, N)
    got = sfc.gemm(Ad, Bd, ca_c=2, k_block_factor=2, tile="pair256")
    layers = []
    for l in range(2):
        P = torch.empty(M, N, dtype=torch.float32, device="cuda")
        for ik in range(2):
            k0 = 512 * l + 256 * ik
            sfc.gemm(Ad[:, k0:k0 + 256], Bd[k0:k0 + 256], P, ca_c=1, tile="pair256", beta=0.0 if ik == 0 else 1.0)
        layers.append(P)
    assert torch.equal(got, layers[0] + layers[1])


def test_order_and_assignment_do_not_change_bits(sfc):
    A, B = synth.gemm_inputs(1000, 1200, 2500, "uniform", seed=63, lda=synth.pad8(2500))
    Ad, Bd = padded(A.contiguous(), synth.pad8(2500)), padded(B, 1200)
    for c, kbf in ((1, 3), (2, 2)):
        for tile in ("pair256", 128):
            outs = [sfc.gemm(Ad, Bd, ca_c=c, k_block_factor=kbf, order=o, assign=a, tile=tile)
                    for o in ("sfc", "raster") for a in ("segment", "wave", "wave_static")]
            for other in outs[1:]:
                assert torch.equal(outs[0], other), (c, kbf, tile)
            assert torch.equal(outs[0], sfc.gemm(Ad, Bd, ca_c=c, k_block_factor=kbf, tile=tile))


def test_beta_bias_transposed_b_and_8bit(sfc, oracle):
    M, N, K = 300, 392, 1000
    A, B = synth.gemm_inputs(M, N, K, "int", seed=64)
    C0 = torch.randint(-4, 5, (M, N), dtype=torch.float32)
    bias = torch.randint(-3, 4, (N,), dtype=torch.float32)
    ref = oracle.gemm_affine_f64(A, B, beta=2.0, C_in=C0.numpy(), bias=bias.numpy())
    Ad, Bd = padded(A, synth.pad8(K)), padded(B, N)
    for c, kbf in ((1, 2), (2, 3)):
        for dt in (torch.float32, torch.bfloat16):
            C = C0.to(dt).cuda()
            sfc.gemm(Ad, Bd, C, ca_c=c, k_block_factor=kbf, beta=2.0, bias=bias.cuda())
            want = ref if dt == torch.float32 else oracle.round_bf16(ref)
            assert np.array_equal(C.float().cpu().numpy().astype(np.float64), want), (c, kbf, dt)
        Bt = padded(B.t().contiguous(), synth.pad8(K))
        Ct = sfc.gemm(Ad, Bt, b_layout="nk", ca_c=c, k_block_factor=kbf)
        assert np.array_equal(Ct.cpu().numpy().astype(np.float64), oracle.gemm_f64(A, B)), (c, kbf)
    if hasattr(torch, "float8_e4m3fn"):
        A8, B8 = synth.gemm_inputs_f8(256, 512, 2048, "e4m3", "int", seed=65)
        ref8 = oracle.gemm_f8_f64(A8, B8, "e4m3")
        C8 = sfc.gemm(A8.cuda(), B8.cuda(), ca_c=2, k_block_factor=4)      # 16 slabs of 128
        assert np.array_equal(C8.cpu().numpy().astype(np.float64), ref8)


def test_workspace_and_library_choice(sfc, oracle):
    from paper_2601_16294_gb300 import binding
    M, N, K = 512, 512, 1024
    A, B = synth.gemm_inputs(M, N, K, "int", seed=66)
    ref = oracle.gemm_f64(A, B)
    Ad, Bd = A.cuda(), B.cuda()
    need = sfc.workspace_size(M, N, K, 1, k_block_factor=4, out_dtype=torch.bfloat16)
    assert need == M * N * 4
    ws = torch.empty(need // 4, dtype=torch.float32, device="cuda")
    Cb = sfc.gemm(Ad, Bd, ca_c=1, k_block_factor=4, out_dtype=torch.bfloat16, workspace=ws)
    assert np.array_equal(Cb.cpu().view(torch.int16).numpy().view(np.uint16), oracle.round_bf16_bits(ref))
    with pytest.raises(binding.SfcError) as e:
        sfc.gemm(Ad, Bd, ca_c=1, k_block_factor=4, out_dtype=torch.bfloat16, workspace=ws[: need // 8])
    assert e.value.code == binding.SFC_ERR_WORKSPACE
    # ca_c = 0: the planner keeps every layer at least k_block_factor slabs deep
    C = sfc.gemm(Ad, Bd, ca_c=0, k_block_factor=4)
    assert np.array_equal(C.cpu().numpy().astype(np.float64), ref)
    with pytest.raises(binding.SfcError) as e:
        sfc.gemm(Ad, Bd, ca_c=8, k_block_factor=4)                         # 16 slabs: 2 per layer
    assert e.value.code == binding.SFC_ERR_INVALID_ARG


def test_unaligned_c_reads_the_partial_sum(sfc, oracle):
    # rows of C that the TMA cannot store: later passes read C and add instead
    # of adding in L2; the result is the same
    M, N, K = 300, 260, 1024
    A, B = synth.gemm_inputs(M, N, K, "int", seed=67)
    ref = oracle.gemm_f64(A, B)
    Ad, Bd = padded(A, K), padded(B, 264)
    big = torch.full((M, N + 1), float("nan"), dtype=torch.float32, device="cuda")
    C = big[:, :N]                                                        # ldc = N + 1
    sfc.gemm(Ad, Bd, C, ca_c=1, k_block_factor=4)
    assert np.array_equal(C.cpu().numpy().astype(np.float64), ref)
    assert torch.isnan(big[:, N]).all()
    aligned = sfc.gemm(Ad, Bd, ca_c=1, k_block_factor=4)
    assert torch.equal(aligned, C)
