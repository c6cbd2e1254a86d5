"""Oracle pins for the accepted counts and the single-round replay: grid-order
and count invariants, and closed forms for the all-accept / all-reject cases."""
import numpy as np
import pytest

import synth
from oracle import counts as cnt
from oracle import step as st


def test_step_counts_cases():
    assert cnt.step_counts(np.array([1, 1, 0, 1], bool), 4, 100) == (3, 2, 103)
    assert cnt.step_counts(np.array([1, 1, 1, 1], bool), 4, 100) == (4, 4, 104)
    assert cnt.step_counts(np.array([0, 1, 1, 1], bool), 4, 100) == (3, 0, 101)
    assert cnt.step_counts(np.array([1, 1, 1, 1, 0, 0], bool), 4, 100) == (4, 4, 104)
    assert cnt.step_counts(np.zeros(8, bool), 0, 50) == (0, 0, 50)


def _stream(B, D_max, V, seed, kind="normal"):
    def inputs(t):
        rng = np.random.default_rng(seed * 7919 + t)
        if kind == "normal":
            lp = rng.standard_normal((B * D_max, V)).astype(np.float32) * 2
            lq = rng.standard_normal((B * D_max, V)).astype(np.float32) * 2
        elif kind == "same":
            lq = rng.standard_normal((B * D_max, V)).astype(np.float32) * 2
            lp = lq.copy()
        return lp, lq, synth.philox_uniforms(seed, t, B * D_max)
    return inputs


@pytest.mark.parametrize("H,W,k_v,B", [(8, 8, 1, 2), (6, 5, 2, 3)])
def test_replay_invariants(H, W, k_v, B):
    P = 7
    D_max = (k_v + 1) * W
    hist, grid_tok, final = st.replay(H, W, P, k_v, B, D_max, _stream(B, D_max, 64, 1))
    assert (final == P + H * W).all()
    assert (grid_tok >= 0).all() and (grid_tok < 64).all()
    total = np.zeros(B, np.int64)
    for h in hist:
        adv = h["next_cache_len"] - h["cache_len"]
        assert (adv >= 0).all()
        assert ((adv >= 1) | (h["n_drafts"] == 0)).all()
        assert ((0 <= h["accepted_count"]) & (h["accepted_count"] <= h["n_drafts"])).all()
        assert (h["accepted_prefix"] <= h["accepted_count"]).all()
        assert (adv <= h["n_drafts"]).all()
        total += adv
    assert (total == H * W).all()


def test_replay_all_accept_closed_form():
    """p == q: every draft is accepted, so each step commits its whole
    frontier (k_v + 1 rows from a row start) and the replay takes
    ceil(H / (k_v + 1)) steps."""
    for H, W, k_v in [(8, 8, 1), (7, 4, 1), (9, 3, 2)]:
        D_max = (k_v + 1) * W
        hist, grid_tok, final = st.replay(H, W, 3, k_v, 1, D_max, _stream(1, D_max, 32, 2, "same"))
        assert len(hist) == -(-H // (k_v + 1))
        assert all(h["accepted_prefix"][0] == h["n_drafts"][0] for h in hist)


def test_replay_all_reject_commits_one_token_per_step():
    """Draft and target disjoint in support (q puts its mass where p has
    none): alpha ~ 0, every draft is rejected, each step commits exactly the
    correction token, and the replay takes H * W steps."""
    H, W = 3, 4
    D_max = 2 * W
    V = 8

    def inputs(t):
        lp = np.full((D_max, V), -40.0, np.float32)
        lq = np.full((D_max, V), -40.0, np.float32)
        lp[:, :4] = 0.0
        lq[:, 4:] = 0.0
        return lp, lq, synth.philox_uniforms(0, t, D_max)

    hist, grid_tok, final = st.replay(H, W, 2, 1, 1, D_max, inputs)
    assert len(hist) == H * W
    assert (grid_tok < 4).all()
