"""The tensor cores' attainable rate (sfc_mma_peak): back-to-back pair MMAs
from resident operands report a per-SM rate within the hardware's range and a
device rate consistent with it at a plausible clock."""
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def test_mma_peak_is_plausible(sfc):
    per_clk, tflops = sfc.mma_peak(iters=2048)
    # a 2-SM pair's 256 x 256 x 16 MMA is 2 MFLOP; dense bf16 on this part is a few thousand FLOP/clk/SM
    assert 2000.0 < per_clk < 20000.0, per_clk
    sms = sfc.num_workers()
    clock_ghz = tflops * 1e12 / (per_clk * sms) / 1e9
    assert 0.5 < clock_ghz < 2.5, (tflops, per_clk, clock_ghz)
    assert sfc.device_status() == 0
