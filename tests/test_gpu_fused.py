"""K layers summed inside the GEMM launch (2..4 layers, one item per worker).

The option is off by default (measured slower than the reduction kernel); these
tests switch it on.  Each 32 x 128 region of a tile is summed by one of the
tile's layer workers from the other layers' fp32 partials, in layer order
0, 1, ..., c-1, which is the order of the reduction kernel, so the output must
have the same bits as the two-kernel path (forced with ``set_fused(False)``),
and integer-valued inputs (every partial sum exact) must give the oracle's
result bit for bit.  Outputs are allocated with 16-byte rows, the layout the
in-launch sum needs; an unaligned C takes the reduction kernel instead.
"""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


@pytest.fixture(autouse=True)
def fused_default(sfc):
    previous = sfc.binding.set_fused(True)
    yield
    sfc.binding.set_fused(previous)


def dev(t):
    """CPU tensor (possibly a padded view) -> CUDA tensor with the same row stride."""
    base = t.as_strided((t.shape[0], t.stride(0)), (t.stride(0), 1)) if t.stride(0) != t.shape[1] else t
    return base.contiguous().cuda()[:, : t.shape[1]]


def out_like(M, N, dtype, aligned=True):
    esz = 4 if dtype == torch.float32 else 2
    ld = (N * esz + 15) // 16 * 16 // esz if aligned else N
    return torch.full((M, ld), float("nan"), dtype=dtype, device="cuda")[:, :N]


def bits(C):
    return C.contiguous().view(torch.int32 if C.dtype == torch.float32 else torch.int16).cpu()


def both(sfc, Ad, Bd, dtype, **kw):
    """(in-launch sum, reduction kernel) outputs of the same call."""
    M, N = Ad.shape[0], (Bd.shape[1] if kw.get("b_layout", "kn") == "kn" else Bd.shape[0])
    outs = []
    for fused in (True, False):
        sfc.binding.set_fused(fused)
        C = out_like(M, N, dtype)
        sfc.gemm(Ad, Bd, C, **kw)
        outs.append(C)
    torch.cuda.synchronize()
    assert sfc.device_status() == 0
    return outs


# (M, N, K, tile, layers): one wave of items for the tile (pairs: 76 workers, one SM: 152)
CASES = [
    (512, 1024, 4096, "pair256", 2),
    (512, 4096, 4096, "pair256", 2),
    (300, 520, 1000, "pair256", 3),
    (129, 8191, 512, "pair256", 2),
    (512, 512, 8192, "pair256", 4),
    (256, 1024, 2048, "pair128", 4),
    (384, 640, 1000, 128, 3),
    (129, 1000, 2500, 256, 2),
    (1024, 1024, 4096, "pair256", 4),
]


@pytest.mark.parametrize("M,N,K,tile,c", CASES)
@pytest.mark.parametrize("dtype", [torch.float32, torch.bfloat16])
def test_same_bits_as_reduction_kernel(sfc, M, N, K, tile, c, dtype):
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=M * 3 + N + K, lda=synth.pad8(K), ldb=synth.pad8(N))
    Ad, Bd = dev(A), dev(B)
    fused, plain = both(sfc, Ad, Bd, dtype, ca_c=c, tile=tile)
    assert torch.isfinite(fused.float()).all()
    assert torch.equal(bits(fused), bits(plain)), (M, N, K, tile, c)


def test_integer_inputs_match_oracle_bit_for_bit(sfc, oracle):
    M, N, K = 384, 1000, 3000
    A, B = synth.gemm_inputs(M, N, K, "int", seed=21, lda=synth.pad8(K), ldb=synth.pad8(N))
    ref = oracle.gemm_f64(A.contiguous(), B.contiguous())
    ref_bits = oracle.round_bf16_bits(ref)
    Ad, Bd = dev(A), dev(B)
    sfc.binding.set_fused(True)
    for c in (2, 3, 4):
        for tile in (128, 256, "pair128", "pair256"):
            for order in ("sfc", "raster"):
                for assign in ("segment", "wave", "auto"):
                    C = out_like(M, N, torch.float32)
                    sfc.gemm(Ad, Bd, C, ca_c=c, tile=tile, order=order, assign=assign)
                    got = C.cpu().numpy().astype(np.float64)
                    assert np.array_equal(got, ref), (c, tile, order, assign)
                    Cb = out_like(M, N, torch.bfloat16)
                    sfc.gemm(Ad, Bd, Cb, ca_c=c, tile=tile, order=order, assign=assign)
                    got_b = Cb.cpu().view(torch.int16).numpy().view(np.uint16)
                    assert np.array_equal(got_b, ref_bits), (c, tile, order, assign)
    assert sfc.device_status() == 0


def test_beta_and_bias_same_bits(sfc):
    M, N, K = 512, 1024, 3000
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=3, lda=synth.pad8(K))
    Ad, Bd = dev(A), dev(B)
    bias = torch.linspace(-1.0, 1.0, N, device="cuda", dtype=torch.float32)
    for dtype in (torch.float32, torch.bfloat16):
        C0 = torch.randn(M, N, device="cuda").to(dtype)
        outs = []
        for fused in (True, False):
            sfc.binding.set_fused(fused)
            C = out_like(M, N, dtype)
            C.copy_(C0)
            sfc.gemm(Ad, Bd, C, ca_c=2, tile="pair256", beta=0.5, bias=bias)
            outs.append(C)
        assert torch.equal(bits(outs[0]), bits(outs[1])), dtype
    assert sfc.device_status() == 0


def test_transposed_b_and_8bit_inputs_same_bits(sfc):
    M, N, K = 512, 2048, 4096
    A, B = synth.gemm_inputs(M, N, K, "prefill", seed=8)
    Ad = A.cuda()
    Bt = B.t().contiguous().cuda()  # N x K
    fused, plain = both(sfc, Ad, Bt, torch.bfloat16, ca_c=2, tile="pair256", b_layout="nk")
    assert torch.equal(bits(fused), bits(plain))
    A8, B8 = synth.gemm_inputs_f8(M, N, K, "e4m3", "uniform", seed=9)
    fused, plain = both(sfc, A8.cuda(), B8.t().contiguous().cuda(), torch.float32, ca_c=3, tile="pair256",
                        b_layout="nk")
    assert torch.equal(bits(fused), bits(plain))


def test_repeated_runs_identical(sfc):
    M, N, K = 512, 4096, 4096
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=4)
    Ad, Bd = A.cuda(), B.cuda()
    sfc.binding.set_fused(True)
    first = None
    for _ in range(10):
        C = out_like(M, N, torch.bfloat16)
        sfc.gemm(Ad, Bd, C, ca_c=2, tile="pair256")
        if first is None:
            first = bits(C)
        else:
            assert torch.equal(bits(C), first)
    assert sfc.device_status() == 0


def test_unaligned_output_takes_the_reduction_kernel(sfc, oracle):
    # bf16 C with 300-element rows (600 bytes) cannot be stored by the TMA: the call sums its
    # layers with the reduction kernel, with the same result
    M, N, K = 256, 300, 2048
    A, B = synth.gemm_inputs(M, N, K, "int", seed=5, ldb=synth.pad8(N))
    ref_bits = oracle.round_bf16_bits(oracle.gemm_f64(A.contiguous(), B.contiguous()))
    Ad, Bd = dev(A), dev(B)
    sfc.binding.set_fused(True)
    C = out_like(M, N, torch.bfloat16, aligned=False)
    sfc.gemm(Ad, Bd, C, ca_c=2, tile="pair256")
    got = C.cpu().view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(got, ref_bits)
    assert sfc.device_status() == 0


def test_graph_replays(sfc):
    # a captured call keeps its epoch: every replay must still wait for its own partials
    M, N, K = 512, 4096, 4096
    Ad = torch.empty(M, K, dtype=torch.bfloat16, device="cuda")
    Bd = torch.empty(K, N, dtype=torch.bfloat16, device="cuda")
    C = out_like(M, N, torch.bfloat16)
    sfc.binding.set_fused(True)
    inputs = [synth.gemm_inputs(M, N, K, "uniform", seed=s) for s in (30, 31, 32)]
    Ad.copy_(inputs[0][0].cuda())
    Bd.copy_(inputs[0][1].cuda())
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        sfc.gemm(Ad, Bd, C, ca_c=2, tile="pair256")
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            sfc.gemm(Ad, Bd, C, ca_c=2, tile="pair256")
    torch.cuda.synchronize()
    for A, B in inputs + inputs:
        Ad.copy_(A.cuda())
        Bd.copy_(B.cuda())
        C.fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        E = out_like(M, N, torch.bfloat16)
        sfc.gemm(Ad, Bd, E, ca_c=2, tile="pair256")
        torch.cuda.synchronize()
        assert torch.equal(bits(C), bits(E))
    assert sfc.device_status() == 0


def test_two_streams_at_once(sfc, oracle):
    # launches whose blocks wait for one another, on two streams at the same time: each grid is
    # resident as a whole (cooperative launch), so neither waits on blocks the other holds back
    shapes = [(512, 4096, 4096), (1024, 1024, 8192)]
    data = []
    for i, (M, N, K) in enumerate(shapes):
        A, B = synth.gemm_inputs(M, N, K, "int", seed=40 + i)
        data.append((A.cuda(), B.cuda(), oracle.gemm_f64(A, B)))
    sfc.binding.set_fused(True)
    streams = [torch.cuda.Stream(), torch.cuda.Stream()]
    outs = [[], []]
    for rep in range(20):
        for i, st in enumerate(streams):
            Ad, Bd, _ = data[i]
            with torch.cuda.stream(st):
                C = out_like(Ad.shape[0], Bd.shape[1], torch.float32)
                sfc.gemm(Ad, Bd, C, ca_c=2 if i == 0 else 4, tile="pair256", stream=st)
                outs[i].append(C)
    torch.cuda.synchronize()
    assert sfc.device_status() == 0
    for i in range(2):
        for C in outs[i]:
            assert np.array_equal(C.cpu().numpy().astype(np.float64), data[i][2])


def test_which_reduction_ran(sfc):
    # a call that fits one wave sums in the launch; with the switch off, or with too many layers
    # for it, the reduction kernel runs instead
    M, N, K = 512, 4096, 4096
    Ad = torch.randn(M, K, device="cuda").to(torch.bfloat16)
    Bd = torch.randn(K, N, device="cuda").to(torch.bfloat16)
    C = out_like(M, N, torch.bfloat16)
    cases = [(True, 2, 1), (False, 2, 0), (True, 8, 0)]
    for fused, c, expect in cases:
        sfc.binding.set_fused(fused)
        before = sfc.binding.fused_launches()
        sfc.gemm(Ad, Bd, C, ca_c=c, tile="pair256")
        torch.cuda.synchronize()
        assert sfc.binding.fused_launches() - before == expect, (fused, c)
    assert sfc.device_status() == 0
