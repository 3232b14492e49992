"""Per-shape tuning (sfc_gemm_tune, the paper's a-priori autotuning of a
shape's knobs): the measured choice is a valid configuration, C holds its
result, later automatic calls use it, and the tile it picks never changes the
result's bits."""
import pytest
import torch

from paper_2601_16294_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    s.tune_forget()
    yield s
    s.tune_forget()


def inputs(M, N, K, seed):
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=seed)
    return A.cuda(), B.cuda()


@pytest.mark.parametrize("M,N,K", [(3000, 5000, 7000), (512, 512, 8192), (1000, 1200, 2500)])
def test_tuned_choice_is_used_and_keeps_bits(sfc, M, N, K):
    A, B = inputs(M, N, K, M + N)
    before = sfc.gemm(A, B, ca_c=1, out_dtype=torch.bfloat16)        # time model's tile
    C = torch.empty(M, N, dtype=torch.bfloat16, device="cuda")
    tile, c, kbf = sfc.tune(A, B, C, max_layers=8, max_kbf=4)
    assert tile in ("128", 128, 256, "pair128", "pair256")
    assert 1 <= c <= 8 and kbf in (1, 2, 4)
    # C holds the chosen configuration's result
    assert torch.equal(C, sfc.gemm(A, B, ca_c=c, tile=tile, k_block_factor=kbf, out_dtype=torch.bfloat16))
    # the library's own choice is now the tuned one
    assert sfc.plan(M, N, K, ca_c=0, out_dtype=torch.bfloat16) == (tile, c)
    assert torch.equal(sfc.gemm(A, B, ca_c=0, out_dtype=torch.bfloat16),
                       sfc.gemm(A, B, ca_c=c, tile=tile, out_dtype=torch.bfloat16))
    # with the layer count fixed only the tile can change, and the tile never changes the bits
    assert torch.equal(sfc.gemm(A, B, ca_c=1, out_dtype=torch.bfloat16), before)
    assert sfc.device_status() == 0


def test_forget_and_tile_only(sfc):
    M, N, K = 1536, 2048, 3072
    A, B = inputs(M, N, K, 7)
    model = sfc.plan(M, N, K, ca_c=1)
    tile, c, kbf = sfc.tune(A, B, max_layers=1, max_kbf=1)              # tile only
    assert c == 1 and kbf == 1
    assert sfc.plan(M, N, K, ca_c=1) == (tile, 1)
    sfc.tune_forget()
    assert sfc.plan(M, N, K, ca_c=1) == model


@pytest.mark.filterwarnings("ignore:The CUDA Graph is empty")
def test_tuning_is_refused_during_capture(sfc):
    from paper_2601_16294_gb300 import binding
    A, B = inputs(512, 512, 512, 9)
    C = torch.empty(512, 512, dtype=torch.float32, device="cuda")
    sfc.gemm(A, B, C)                                                   # set-up before the capture
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with pytest.raises(binding.SfcError) as e:
        with torch.cuda.graph(g, stream=s):
            sfc.tune(A, B, C, stream=s)
    assert e.value.code == binding.SFC_ERR_UNSUPPORTED


def test_nearest_tuned_shape(sfc):
    sfc.tune_forget()
    M, N, K = 3000, 5000, 7000
    A, B = inputs(M, N, K, 11)
    tile, c, _ = sfc.tune(A, B, out_dtype=torch.bfloat16, max_layers=1, max_kbf=1)
    near = (3100, 4900, 7000)                                          # never tuned
    model = sfc.plan(*near, ca_c=1, out_dtype=torch.bfloat16)
    try:
        sfc.tune_lookup(True)
        assert sfc.plan(*near, ca_c=1, out_dtype=torch.bfloat16) == (tile, 1)
        # other output types are other tables
        f32 = sfc.plan(*near, ca_c=1)
        sfc.tune_lookup(False)
        assert sfc.plan(*near, ca_c=1) == f32
        Anear, Bnear = inputs(*near, 12)
        sfc.tune_lookup(True)
        got = sfc.gemm(Anear, Bnear, ca_c=1, out_dtype=torch.bfloat16)
        sfc.tune_lookup(False)
        assert torch.equal(got, sfc.gemm(Anear, Bnear, ca_c=1, out_dtype=torch.bfloat16))   # the tile keeps the bits
    finally:
        sfc.tune_lookup(False)
    assert sfc.plan(*near, ca_c=1, out_dtype=torch.bfloat16) == model   # exact lookup again
    sfc.tune_forget()
