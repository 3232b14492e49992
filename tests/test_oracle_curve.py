"""Pins for the oracle's generalized Hilbert curve (Sec. II-B, II-D, II-E).

Nothing here re-types the oracle's construction: the checks are properties the
paper states (contiguity, patches, decompositions), brute force over every
small grid, and the textbook Hilbert d->(x,y) routine on power-of-two squares.
"""
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "paper_curve_pins.txt")


def coords(order, Nt):
    return order // Nt, order % Nt


def assert_curve_valid(order, Mt, Nt):
    # Q1: bijection onto the grid
    assert order.shape == (Mt * Nt,)
    assert np.array_equal(np.sort(order), np.arange(Mt * Nt))
    tm, tn = coords(order, Nt)
    # Q3: starts at tile (0, 0)
    assert tm[0] == 0 and tn[0] == 0
    # Q2: consecutive tiles share an edge (Sec. II-B: no big jumps)
    step = np.abs(np.diff(tm)) + np.abs(np.diff(tn))
    assert np.all(step == 1), "non-adjacent step on %dx%d at %s" % (Mt, Nt, np.nonzero(step != 1)[0][:5])


@pytest.mark.parametrize("Mt", range(1, 34))
def test_all_small_grids_bijective_and_adjacent(oracle, Mt):
    for Nt in range(1, 34):
        assert_curve_valid(oracle.gilbert_order(Mt, Nt), Mt, Nt)


@pytest.mark.parametrize("Mt,Nt", [(2, 64), (64, 2), (4, 1002), (64, 1002), (1002, 64), (128, 128),
                                   (24, 40), (8, 133), (48, 6), (4, 4), (128, 501), (1, 1002),
                                   (1002, 1), (63, 65), (65, 64)])
def test_config_grids(oracle, Mt, Nt):
    assert_curve_valid(oracle.gilbert_order(Mt, Nt), Mt, Nt)


def test_degenerate_grids_are_lines(oracle):
    assert oracle.gilbert_order(1, 1).tolist() == [0]
    for n in (2, 3, 7, 64):
        assert oracle.gilbert_order(1, n).tolist() == list(range(n))        # one row
        assert oracle.gilbert_order(n, 1).tolist() == list(range(n))        # one column


def textbook_hilbert_d2xy(n, d):
    """The classical Hilbert index -> (x, y) map on an n x n square, n = 2^k."""
    x = y = 0
    t = d
    s = 1
    while s < n:
        rx = 1 & (t // 2)
        ry = 1 & (t ^ rx)
        if ry == 0:
            if rx == 1:
                x, y = s - 1 - x, s - 1 - y
            x, y = y, x
        x += s * rx
        y += s * ry
        t //= 4
        s *= 2
    return x, y


@pytest.mark.parametrize("k", range(0, 8))
def test_power_of_two_squares_are_the_classical_hilbert_curve(oracle, k):
    # Q4: on 2^k squares the generalized curve reduces to the classical one
    # (x along tn, y along tm; the same fixed orientation for every k).
    n = 2 ** k
    order = oracle.gilbert_order(n, n)
    tm, tn = coords(order, n)
    ref = np.array([textbook_hilbert_d2xy(n, d) for d in range(n * n)])
    assert np.array_equal(tn, ref[:, 0]) and np.array_equal(tm, ref[:, 1])


@pytest.mark.parametrize("k", [2, 3, 4, 5, 6])
def test_dyadic_ranges_are_squares(oracle, k):
    # On 2^k squares every aligned index range [j 4^l, (j+1) 4^l) is a
    # 2^l x 2^l square: the recursive quadrant structure of Sec. II-B.
    n = 2 ** k
    order = oracle.gilbert_order(n, n)
    tm, tn = coords(order, n)
    for l in range(1, k + 1):
        size = 4 ** l
        side = 2 ** l
        for j in range(n * n // size):
            r = tm[j * size:(j + 1) * size]
            c = tn[j * size:(j + 1) * size]
            assert r.max() - r.min() + 1 == side and c.max() - c.min() + 1 == side
            assert r.min() % side == 0 and c.min() % side == 0


def _read_pins():
    pins = []
    with open(GOLDEN) as f:
        for line in f:
            line = line.split("#", 1)[0].strip()
            if line:
                pins.append(line.split())
    return pins


def _bbox(tm, tn):
    return int(tm.min()), int(tm.max()), int(tn.min()), int(tn.max())


def test_paper_patch_pins(oracle):
    # Sec. II-B, Fig. 2: on 16x16, indices 0-31 form an 8x4 patch at the top
    # left, indices 8-15 a 2x4 sub-patch inside it (w columns x h rows).
    pins = [p for p in _read_pins() if p[0] == "patch"]
    assert len(pins) == 2
    boxes = {}
    for _, Mt, Nt, lo, hi, w, h, where in pins:
        Mt, Nt, lo, hi, w, h = map(int, (Mt, Nt, lo, hi, w, h))
        order = oracle.gilbert_order(Mt, Nt)
        tm, tn = coords(order[lo:hi], Nt)
        r0, r1, c0, c1 = _bbox(tm, tn)
        assert (c1 - c0 + 1, r1 - r0 + 1) == (w, h)
        assert (r1 - r0 + 1) * (c1 - c0 + 1) == hi - lo        # a full rectangle
        boxes[(lo, hi)] = (r0, r1, c0, c1)
        if where == "topleft":
            assert (r0, c0) == (0, 0)
        else:
            plo, phi = map(int, where.split(":")[1:])
            pr0, pr1, pc0, pc1 = boxes[(plo, phi)]
            assert pr0 <= r0 and r1 <= pr1 and pc0 <= c0 and c1 <= pc1


def _segment_boxes(order, Nt, nseg):
    n = order.size
    assert n % nseg == 0
    size = n // nseg
    out = []
    for p in range(nseg):
        tm, tn = coords(order[p * size:(p + 1) * size], Nt)
        out.append(_bbox(tm, tn))
    return out, size


def test_paper_decomposition_pins(oracle):
    # Sec. II-D (Fig. 3) and Sec. II-E (Fig. 4): contiguous equal segments of
    # the curve form compact patches whose arrangement follows the grid shape.
    for pin in (p for p in _read_pins() if p[0] == "segments"):
        Mt, Nt, nseg = int(pin[1]), int(pin[2]), int(pin[3])
        order = oracle.gilbert_order(Mt, Nt)
        boxes, size = _segment_boxes(order, Nt, nseg)
        for r0, r1, c0, c1 in boxes:                   # every segment is a full rectangle
            assert (r1 - r0 + 1) * (c1 - c0 + 1) == size
        if pin[4] == "arrangement":
            rows, cols, side = int(pin[5]), int(pin[6]), int(pin[8])
            assert all(r1 - r0 + 1 == side and c1 - c0 + 1 == side for r0, r1, c0, c1 in boxes)
            assert len({b[0] for b in boxes}) == rows    # distinct row bands
            assert len({b[2] for b in boxes}) == cols    # distinct column bands
        else:
            area = int(pin[5])
            assert size == area
            assert all(max(r1 - r0 + 1, c1 - c0 + 1) == 2 * min(r1 - r0 + 1, c1 - c0 + 1)
                       for r0, r1, c0, c1 in boxes)      # 2:1 rectangles (2.5D layer)


def test_locality_beats_raster(oracle):
    # The property the method relies on (Sec. II-E): a contiguous segment of
    # the curve touches far fewer distinct A row-panels + B column-panels than
    # the same-sized segment of a row-major raster order.
    Mt, Nt, nseg = 64, 96, 48
    order = oracle.gilbert_order(Mt, Nt)
    raster = np.arange(Mt * Nt)
    size = Mt * Nt // nseg

    def panels(o):
        tot = 0
        for p in range(nseg):
            tm, tn = coords(o[p * size:(p + 1) * size], Nt)
            tot += np.unique(tm).size + np.unique(tn).size
        return tot

    assert panels(order) * 2 < panels(raster)
