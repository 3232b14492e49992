"""The GPU decoder the GEMM kernel uses reproduces the oracle's curve bit-exactly."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sfc():
    from paper_2601_16294_gb300 import build_lib
    build_lib.build()
    import paper_2601_16294_gb300 as s
    return s


def test_device_order_all_small_grids(sfc, oracle):
    for Mt in range(1, 34):
        for Nt in range(1, 34):
            got = sfc.tile_order_device(Mt, Nt).cpu().numpy()
            assert np.array_equal(got, oracle.gilbert_order(Mt, Nt)), (Mt, Nt)


@pytest.mark.parametrize("Mt,Nt", [(4, 4), (16, 16), (128, 128), (128, 64), (64, 1002), (64, 501), (16, 1002),
                                   (2, 64), (24, 40), (8, 133), (48, 6), (12, 20), (4, 67), (1002, 64)])
def test_device_order_config_grids(sfc, oracle, Mt, Nt):
    got = sfc.tile_order_device(Mt, Nt).cpu().numpy()
    assert np.array_equal(got, oracle.gilbert_order(Mt, Nt))
