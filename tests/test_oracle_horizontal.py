"""Oracle pins for the horizontal stage (Sec. 3.3: k_h horizontal heads draft
offsets +1 .. +k_h along the row; Sec. 4: one verification round with the
bonus token): the k_h frontier as a contiguous raster run, its reductions,
the bonus token against library routines, and the bonus commit."""
import numpy as np
import pytest
import scipy.special

from oracle import frontier as fr
from oracle import step as ostep


@pytest.mark.parametrize("H,W,k_h,k_v", [(6, 9, 5, 0), (6, 9, 5, 1), (4, 7, 1, 2), (5, 5, 9, 1)])
def test_k_h_frontier_is_a_contiguous_raster_run(H, W, k_h, k_v):
    P = 3
    for n_c in range(H * W + 1):
        coords = fr.frontier(H, W, P, P + n_c, k_v, k_h)
        g = fr.grid_index(coords, W)
        # raster positions n_c, n_c + 1, ... without gaps
        assert np.array_equal(g, np.arange(n_c, n_c + len(g)))
        if n_c == H * W:
            assert len(g) == 0
            continue
        y0, c = divmod(n_c, W)
        h = min(k_h, W - c)
        assert len(g) >= h and all(y == y0 for y, _ in coords[:h])
        if c + h < W:  # an unfinished row has no vertical part
            assert len(g) == h
        # k_h covering the rest of the row is the frontier without k_h
        if k_h >= W - c:
            assert coords == fr.frontier(H, W, P, P + n_c, k_v)


def _case(seed, B=3, W=8, H=6, P=4, D_max=16, V=40):
    rng = np.random.default_rng(seed)
    rows = B * D_max
    return (rng.standard_normal((rows, V)) * 2, rng.standard_normal((rows, V)) * 2,
            rng.random((rows, 2)), H, W, P, D_max)


@pytest.mark.parametrize("strategy", ["accept_reject", "greedy", "sample"])
def test_bonus_token_from_library_routines(strategy):
    lp, lq, u, H, W, P, D_max = _case(1)
    cache = np.array([P + 3, P + W * 2, P + W * 4 + 6])
    r = ostep.accept_step(H, W, P, 0, cache, D_max, lp, lq, u, strategy=strategy, k_h=5,
                          bonus=True)
    assert np.array_equal(r["n_drafts"], [5, 5, 2])
    for b in range(3):
        row = b * D_max + r["n_drafts"][b]
        assert r["bonus_row"][b] == row
        if strategy == "greedy":
            assert r["bonus_tok"][b] == np.argmax(lp[row])
        else:
            p = scipy.special.softmax(lp[row])
            c = np.cumsum(p)
            assert r["bonus_tok"][b] == np.searchsorted(c, u[row, 1] * c[-1], side="right")


def test_bonus_is_committed_when_every_draft_is_accepted():
    lp, lq, u, H, W, P, D_max = _case(2)
    cache = np.array([P + 3, P + W * 2, P + H * W - 2])  # the last one ends at the grid's end
    r = ostep.accept_step(H, W, P, 0, cache, D_max, lq, lq, u, k_h=5, bonus=True)  # p = q
    assert r["decisions"]["accepted"].all()
    n = r["n_drafts"]
    assert np.array_equal(n, [5, 5, 2])
    assert np.array_equal(r["next_cache_len"][:2], cache[:2] + n[:2] + 1)
    assert r["next_cache_len"][2] == cache[2] + 2  # no position after the grid's last
    # without the bonus: the plain prefix rule
    r0 = ostep.accept_step(H, W, P, 0, cache, D_max, lq, lq, u, k_h=5)
    assert np.array_equal(r0["next_cache_len"], cache + n)


def test_bonus_is_not_committed_after_a_rejection():
    lp, lq, u, H, W, P, D_max = _case(3)
    cache = np.array([P + 1, P + W, P + 2 * W + 1])
    r = ostep.accept_step(H, W, P, 0, cache, D_max, lp, lq, u, k_h=5, bonus=True)
    r0 = ostep.accept_step(H, W, P, 0, cache, D_max, lp, lq, u, k_h=5)
    for b in range(3):
        if r["accepted_prefix"][b] < r["n_drafts"][b]:
            assert r["next_cache_len"][b] == r0["next_cache_len"][b]
        else:
            assert r["next_cache_len"][b] == r0["next_cache_len"][b] + 1
