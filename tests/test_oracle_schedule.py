"""Oracle pins for the whole decoding schedule (Sec. 3.3, Sec. 4 "SSD
Configuration", App. "Configuration Selection" and "Multi-Row Anticipation
Ablations"):
  * the paper's step counts (51 sweep rows over three backbones) minus the
    vertical stage's forward passes leave one horizontal-stage count per
    backbone, inside the bounds the horizontal stage allows;
  * the oracle replay spends exactly those vertical forward passes for every
    (k_v, b, i) tried, and commits every grid token once, in raster order;
  * closed forms: identical target and draft distributions accept every draft
    (the horizontal stage then commits k_h drafts plus the bonus per step);
    drafts the target gives no mass to are always rejected (one token per
    horizontal step, S_h = W)."""
import math
import os

import numpy as np
import pytest

import synth
from oracle import schedule as sch

HERE = os.path.dirname(os.path.abspath(__file__))


def _rows():
    out = []
    for line in open(os.path.join(HERE, "golden", "schedule_steps.txt")):
        if line.strip() and not line.startswith("#"):
            bb, n, v, b, i, st = line.split()
            out.append((bb, int(n), int(v), int(b), int(i), int(st)))
    return out


def test_paper_step_counts_fit_the_schedule():
    per = {}
    for bb, n, v, b, i, steps in _rows():
        per.setdefault(bb, set()).add(steps - sch.vertical_steps(n, v, b, i))
    # one horizontal-stage count per backbone explains every sweep row
    assert per == {"janus": {11}, "lumina": {21}, "emu3": {37}}
    for bb, n in (("janus", 24), ("lumina", 48), ("emu3", 90)):
        (s_h,) = per[bb]
        assert math.ceil(n / 6) <= s_h <= n  # 1 to k_h + 1 = 6 tokens per step


def test_group_formula_cases():
    assert sch.group_steps(1, 2, 0) == 3          # r = 2: two rounds + commit
    assert sch.group_steps(2, 5, 4) == 11         # Lumina's b = 5, i = 4
    assert sch.vertical_steps(48, 2, 5, 4) == 259  # 23 groups of 11 + one row of 6
    assert sch.vertical_steps(24, 1, 2, 0) == 69
    assert sch.vertical_steps(1, 2, 5, 4) == 0


def _inputs(D_max, V, seed, mode="normal"):
    """step -> (tgt, drf, uniforms) from a pool of 3 logit sets."""
    pool = []
    for k in range(3):
        rng = np.random.default_rng(seed * 10 + k)
        if mode == "normal":
            tg, dr = synth._logits_normal(rng, D_max + 1, V)
        elif mode == "same":  # one distribution for every step and slot, target = draft
            row = synth._logits_normal(np.random.default_rng(seed), 1, V)[1]
            dr = np.repeat(row, D_max + 1, axis=0)
            tg = dr.copy()
        else:  # the draft's favourite token has no target mass
            dr = np.zeros((D_max + 1, V), np.float32)
            dr[:, 0] = 50.0
            tg = np.zeros((D_max + 1, V), np.float32)
            tg[:, 0] = -50.0
        pool.append((tg, dr))

    def f(t):
        tg, dr = pool[t % 3]
        return tg, dr, synth.philox_uniforms(seed, t, D_max + 1)
    return f


def _check_complete(H, W, grid, hist, prefix):
    assert (grid >= 0).all()
    caches = [h["cache_len"] for h in hist]
    assert caches == sorted(caches) and caches[0] == prefix


@pytest.mark.parametrize("k_v,b,i", [(1, 2, 0), (2, 2, 1), (3, 1, 2), (1, 0, 0), (2, 3, 0)])
def test_replay_spends_the_formula_steps(k_v, b, i):
    H, W, prefix, V = 7, 8, 4, 48
    D_max = k_v * W
    steps, grid, hist = sch.replay(H, W, prefix, 5, k_v, b, i, D_max, _inputs(D_max, V, 3))
    s_h = sum(h["kind"] == "horizontal" for h in hist)
    assert steps == len(hist) == s_h + sch.vertical_steps(H, k_v, b, i)
    if k_v == 1:
        assert sum(h["kind"] == "commit" for h in hist) == H - 1
    _check_complete(H, W, grid, hist, prefix)
    # every commit pass commits one row (a partial first one after the horizontal stage)
    commits = [h["committed"] for h in hist if h["kind"] == "commit"]
    assert sum(commits) + sum(len(h["tokens"]) for h in hist if h["kind"] == "horizontal") == H * W
    assert all(c <= W for c in commits)


def test_identical_distributions_accept_everything():
    H, W, prefix, V = 5, 8, 2, 40
    D_max = 2 * W
    f = _inputs(D_max, V, 5, mode="same")
    steps, grid, hist = sch.replay(H, W, prefix, 5, 2, 2, 1, D_max, f)
    hs = [h for h in hist if h["kind"] == "horizontal"]
    # 5 drafts + bonus, then the 2 drafts left (no bonus past the first row)
    assert [len(h["tokens"]) for h in hs] == [6, 2]
    for h in hist:
        if "accepted" in h:
            assert h["accepted"].all()
    # every vertical round keeps the draft tokens (the argmax of the draft logits)
    t_hat = int(np.argmax(f(0)[1][0]))
    for h in hist:
        if h["kind"] == "round":
            assert (h["tokens"] == t_hat).all()
    assert steps == len(hs) + sch.vertical_steps(H, 2, 2, 1)


def test_rejected_drafts_commit_one_token_per_horizontal_step():
    H, W, prefix, V = 4, 6, 0, 16
    D_max = W
    steps, grid, hist = sch.replay(H, W, prefix, 5, 1, 1, 0, D_max, _inputs(D_max, V, 7, "reject"))
    hs = [h for h in hist if h["kind"] == "horizontal"]
    assert len(hs) == W and all(len(h["tokens"]) == 1 for h in hs)
    assert all(not h["accepted"].any() for h in hist if "accepted" in h)
    # a rejected draft is replaced by a residual draw: never the draft's token 0
    assert (grid != 0).all()
    assert steps == W + sch.vertical_steps(H, 1, 1, 0)
