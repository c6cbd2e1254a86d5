"""Oracle pins for the frontier and the spatial dependency mask (Sec. 3.1, 3.3)."""
import os

import numpy as np
import pytest

from oracle import frontier as fr

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def test_golden_spatial_offsets():
    """Sec. 3.3's example: on a width-48 grid, horizontal offsets +1..+3 and
    vertical offsets +48, +96, +144 in the flattened sequence."""
    for line in open(os.path.join(GOLDEN, "spatial_offsets.txt")):
        if line.startswith("#") or not line.strip():
            continue
        w, direction, step, off = line.split()
        w, step, off = int(w), int(step), int(off)
        y, x = 5, 7
        dy, dx = (step, 0) if direction == "vertical" else (0, step)
        a = fr.flat_position(y, x, prefix_len=100, row_stride=w)
        b = fr.flat_position(y + dy, x + dx, prefix_len=100, row_stride=w)
        assert b - a == off


@pytest.mark.parametrize("H,W,k_v", [(16, 16, 1), (24, 24, 1), (8, 5, 2), (3, 7, 3), (6, 9, 0)])
def test_frontier_sizes(H, W, k_v):
    P = 11
    for n_c in range(H * W + 1):
        coords = fr.frontier(H, W, P, P + n_c, k_v)
        y0, c = divmod(n_c, W)
        expect = 0
        if y0 < H:
            expect = (W - c) + W * min(k_v, H - 1 - y0)
        assert len(coords) == expect
        # the frontier is the next `expect` raster positions
        g = fr.grid_index(coords, W)
        assert list(g) == list(range(n_c, n_c + expect))


def test_frontier_workloads():
    # 16x16 after a 32-token prefix with 192 cached entries: 16 horizontal
    # drafts on row 10 plus 16 below them on row 11
    coords = fr.frontier(16, 16, 32, 192)
    assert len(coords) == 32
    assert coords[:16] == [(10, x) for x in range(16)]
    assert coords[16:] == [(11, x) for x in range(16)]
    assert fr.frontier(16, 16, 32, 112)[0] == (5, 0)
    # 24x24 sweep: 48 drafts until the last row, then 24, then none
    assert len(fr.frontier(24, 24, 120, 120)) == 48
    assert len(fr.frontier(24, 24, 120, 672)) == 24
    assert len(fr.frontier(24, 24, 120, 696)) == 0
    # mid-row: the remainder of the row plus the next row
    assert len(fr.frontier(32, 32, 64, 64 + 10)) == 64 - 10
    with pytest.raises(ValueError):
        fr.frontier(4, 4, 8, 7)


@pytest.mark.parametrize("extra", [0, 1])
def test_coordinate_mask_equals_flat_mask(extra):
    rng = np.random.default_rng(42)
    for _ in range(40):
        H, W = rng.integers(2, 7, size=2)
        P = int(rng.integers(0, 5))
        rs = int(W + extra)
        k_v = int(rng.integers(1, 3))
        n_c = int(rng.integers(0, H * W + 1))
        coords = fr.frontier(int(H), int(W), P, P + n_c, k_v)
        if extra:
            # with an end-of-line slot per row the committed cache covers whole
            # rows plus their EOL; place the cache just before the first draft
            if not coords:
                continue
            y, x = coords[0]
            cache_len = fr.flat_position(y, x, P, rs)
        else:
            cache_len = P + n_c
        m1 = fr.coord_mask(coords, cache_len, P, rs)
        m2 = fr.flat_mask(coords, cache_len, P, rs)
        assert np.array_equal(m1, m2)
        if coords:
            # every committed key is visible; draft-to-draft visibility is causal
            assert m1[:, :cache_len].all()
            n = len(coords)
            assert np.array_equal(m1[:, cache_len:], np.tril(np.ones((n, n), bool)))


def test_mask_eol_slots():
    # row_stride = W + 1: the end-of-line slot of row y' is seen by row y' + 1 only
    W, P = 4, 2
    coords = [(1, 0), (1, 3), (2, 1)]
    cache_len = fr.flat_position(1, 0, P, W + 1)
    m = fr.coord_mask(coords, cache_len, P, W + 1)
    eol_row0 = P + W  # slot of row 0's end-of-line token
    assert m[:, eol_row0].all()
    assert np.array_equal(m, fr.flat_mask(coords, cache_len, P, W + 1))
