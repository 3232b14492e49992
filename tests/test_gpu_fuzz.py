"""Seeded random configurations against the oracle: random shapes (ragged in
every dimension), input type, B layout, tile, layer count, K blocks, order,
dealing, output type, beta and bias, on integer data, where every fp32 step is
exact, so the result must equal the oracle bit for bit; and random host-buffer
calls (shape, layout, output type, panel count, host row padding), which must
equal the device call with the same plan bit for bit."""
import numpy as np
import pytest
import torch

from paper_2601_16294_gb300 import synth

pytestmark = pytest.mark.gpu

CASES = 48
TILES = ["auto", 128, 256, "pair128", "pair256"]


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def padded(t, ld):
    d = torch.zeros(t.shape[0], ld, dtype=t.dtype, device="cuda")
    d[:, : t.shape[1]] = t.cuda()
    return d[:, : t.shape[1]]


def config(i):
    rng = np.random.default_rng(1000 + i)
    M = int(rng.integers(1, 1100))
    N = int(rng.integers(1, 1100))
    K = int(rng.integers(1, 3000))
    f8 = bool(rng.random() < 0.25) and hasattr(torch, "float8_e4m3fn")
    slab = 128 if f8 else 64
    Kt = (K + slab - 1) // slab
    c = int(rng.choice([c for c in (1, 2, 3, 5, 8) if c <= Kt]))
    kbf = int(rng.choice([k for k in (1, 1, 2, 3) if c * k <= Kt]))
    return dict(M=M, N=N, K=K, f8=f8, c=c, kbf=kbf, tile=TILES[int(rng.integers(len(TILES)))],
                layout=str(rng.choice(["kn", "nk"])), order=str(rng.choice(["sfc", "raster"])),
                assign=str(rng.choice(["auto", "wave", "wave_static", "segment"])),
                out=torch.float32 if rng.random() < 0.5 else torch.bfloat16,
                beta=float(rng.choice([0.0, 0.0, 1.0, -2.0])), bias=bool(rng.random() < 0.3), seed=int(rng.integers(1 << 30)))


@pytest.mark.parametrize("i", range(CASES))
def test_random_configuration(sfc, oracle, i):
    cfg = config(i)
    M, N, K = cfg["M"], cfg["N"], cfg["K"]
    if cfg["f8"]:
        A, B = synth.gemm_inputs_f8(M, N, K, "e4m3", "int", seed=cfg["seed"])
        align = 16
    else:
        A, B = synth.gemm_inputs(M, N, K, "int", seed=cfg["seed"])
        align = 8
    gen = torch.Generator().manual_seed(cfg["seed"])
    C0 = torch.randint(-4, 5, (M, N), generator=gen).float()
    bias = torch.randint(-3, 4, (N,), generator=gen).float() if cfg["bias"] else None
    Bl = B if cfg["layout"] == "kn" else B.t().contiguous()
    if cfg["f8"]:
        ref = oracle.gemm_f8_f64(A, B, "e4m3")
        ref = ref + cfg["beta"] * C0.numpy().astype(np.float64) + (0 if bias is None else bias.numpy())
    else:
        ref = oracle.gemm_affine_f64(A, Bl, b_layout=cfg["layout"], beta=cfg["beta"], C_in=C0.numpy(),
                                     bias=None if bias is None else bias.numpy())
    pad = lambda n: (n + align - 1) // align * align
    Ad = padded(A, pad(K))
    Bd = padded(Bl, pad(Bl.shape[1]))
    C = C0.to(cfg["out"]).cuda()
    sfc.gemm(Ad, Bd, C, ca_c=cfg["c"], k_block_factor=cfg["kbf"], tile=cfg["tile"], order=cfg["order"],
             assign=cfg["assign"], b_layout=cfg["layout"], beta=cfg["beta"],
             bias=None if bias is None else bias.cuda())
    torch.cuda.synchronize()
    assert sfc.device_status() == 0, cfg
    got = C.float().cpu().numpy().astype(np.float64)
    want = ref if cfg["out"] == torch.float32 else oracle.round_bf16(ref)
    assert np.array_equal(got, want), cfg


@pytest.mark.parametrize("i", range(16))
def test_random_host_configuration(sfc, i):
    # the host-buffer path against the device call with the same plan: bit-identical
    rng = np.random.default_rng(5000 + i)
    M, N, K = (int(rng.integers(1, 3000)) for _ in range(3))
    layout = str(rng.choice(["kn", "nk"]))
    out = torch.float32 if rng.random() < 0.5 else torch.bfloat16
    panels = int(rng.choice([0, 1, 2, 3, 7]))
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=int(rng.integers(1 << 30)))
    Bl = B if layout == "kn" else B.t().contiguous()

    def host(t):
        ld = t.shape[1] + int(rng.integers(0, 5))
        h = torch.zeros(t.shape[0], ld, dtype=t.dtype, pin_memory=True)
        h[:, : t.shape[1]] = t
        return h[:, : t.shape[1]]
    tile, c = sfc.plan(M, N, K, ca_c=0, out_dtype=out, b_layout=layout)
    ref = sfc.gemm(padded(A, (K + 7) // 8 * 8), padded(Bl, (Bl.shape[1] + 7) // 8 * 8), ca_c=c, tile=tile,
                   out_dtype=out, b_layout=layout).cpu()
    got = sfc.matmul_host(host(A), host(Bl), ca_c=0, out_dtype=out, b_layout=layout, panels=panels)
    assert torch.equal(got, ref), (M, N, K, layout, out, panels)
