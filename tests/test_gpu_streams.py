"""Streams, graphs and threads: the GEMM is an ordinary stream-ordered call,
so it must give the same bits when captured in a CUDA graph and replayed, and
when issued from several host threads onto several streams at once (each
launch takes its own dynamic-dealing counter)."""
import threading

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


def inputs(M, N, K, seed):
    A, B = synth.gemm_inputs(M, N, K, "uniform", seed=seed)
    return A.cuda(), B.cuda()


def test_graph_capture_and_replay(sfc):
    A, B = inputs(1000, 1200, 2500, 71)
    A2, B2 = inputs(512, 512, 8192, 72)
    s = torch.cuda.Stream()
    C1 = torch.empty(1000, 1200, dtype=torch.bfloat16, device="cuda")
    C2 = torch.empty(512, 512, dtype=torch.float32, device="cuda")
    C3 = torch.empty(512, 512, dtype=torch.float32, device="cuda")
    with torch.cuda.stream(s):
        # eager results (and the one-time per-device set-up, which must precede capture)
        ref1 = sfc.gemm(A, B, out_dtype=torch.bfloat16, ca_c=1, stream=s).clone()
        ref2 = sfc.gemm(A2, B2, ca_c=4, stream=s).clone()          # layer workspace from the pool
        ref3 = sfc.gemm(A2, B2, ca_c=1, k_block_factor=2, stream=s).clone()
    s.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        sfc.gemm(A, B, C1, ca_c=1, stream=s)
        sfc.gemm(A2, B2, C2, ca_c=4, stream=s)
        sfc.gemm(A2, B2, C3, ca_c=1, k_block_factor=2, stream=s)
    for _ in range(3):
        C1.zero_()
        C2.zero_()
        C3.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(C1, ref1)
        assert torch.equal(C2, ref2)
        assert torch.equal(C3, ref3)
    assert sfc.device_status() == 0


def test_threads_on_separate_streams(sfc):
    shapes = [(1024, 768, 4096), (300, 2000, 1000), (2048, 2048, 512), (777, 555, 3333)]
    data = [inputs(M, N, K, 80 + i) for i, (M, N, K) in enumerate(shapes)]
    refs = [sfc.gemm(A, B, ca_c=c).clone() for (A, B), c in zip(data, (1, 2, 1, 3))]
    torch.cuda.synchronize()
    errors = []
    outs = [None] * len(shapes)

    def work(i):
        try:
            A, B = data[i]
            s = torch.cuda.Stream()
            with torch.cuda.stream(s):
                C = None
                for _ in range(20):
                    C = sfc.gemm(A, B, ca_c=(1, 2, 1, 3)[i], stream=s)
            s.synchronize()
            outs[i] = C
        except Exception as e:  # reported by the main thread
            errors.append(e)

    threads = [threading.Thread(target=work, args=(i,)) for i in range(len(shapes))]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors
    for out, ref in zip(outs, refs):
        assert torch.equal(out, ref)
    assert sfc.device_status() == 0


def test_graph_replays_beside_more_than_1024_eager_calls(sfc, oracle):
    """A captured graph keeps whatever the capture gave its launches.  Its
    replays on one stream run beside 1100 eager calls on another stream (more
    than any ring of per-launch counter slots would hold), all with dynamic
    dealing, so a counter two launches shared would drop or repeat tiles.  The
    graph adds A B into C at every replay (C += A B, integer data: exact), so
    a tile dropped or repeated by any replay shows in the final C; every eager
    call writes its own output."""
    # graph: 4096 x 2048 x 1024 on 2-SM pairs: 128 tiles for 76 pairs, so workers take tickets
    Ag, Bg = synth.gemm_inputs(4096, 2048, 1024, "int", seed=91)
    ref_g = torch.from_numpy(oracle.gemm_f64(Ag, Bg)).float()
    # eager: 2048 x 2048 x 128 on single SMs: 256 tiles for 152 workers
    Ae, Be = synth.gemm_inputs(2048, 2048, 128, "int", seed=92)
    ref_e = torch.from_numpy(oracle.round_bf16(oracle.gemm_f64(Ae, Be))).to(torch.bfloat16).cuda()
    Ag, Bg, Ae, Be = Ag.cuda(), Bg.cuda(), Ae.cuda(), Be.cuda()
    n_gemms, replays, eager = 8, 64, 1100
    Cg = [torch.zeros(4096, 2048, dtype=torch.float32, device="cuda") for _ in range(n_gemms)]
    outs = [torch.empty(2048, 2048, dtype=torch.bfloat16, device="cuda") for _ in range(eager)]
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    with torch.cuda.stream(s1):
        for C in Cg:  # set-up and warm-up before the capture, then back to zero
            sfc.gemm(Ag, Bg, C, ca_c=1, tile="pair256", assign="wave", beta=1.0, stream=s1)
            C.zero_()
    s1.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s1):
        for C in Cg:
            sfc.gemm(Ag, Bg, C, ca_c=1, tile="pair256", assign="wave", beta=1.0, stream=s1)
    for C in Cg:
        C.zero_()
    torch.cuda.synchronize()
    with torch.cuda.stream(s1):
        for _ in range(replays):
            g.replay()
    for C in outs:
        sfc.gemm(Ae, Be, C, ca_c=1, tile=128, assign="wave", stream=s2)
    torch.cuda.synchronize()
    assert sfc.device_status() == 0
    want = (ref_g * replays).cuda()
    for C in Cg:
        assert torch.equal(C, want)
    bad = [i for i, C in enumerate(outs) if not torch.equal(C, ref_e)]
    assert not bad, "eager calls with wrong results: %s" % bad[:10]
