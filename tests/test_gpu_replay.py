"""GPU parity of the single-round replay to grid completion: the CUDA path
drives its own cache lengths step after step (device state only), the
oracle runs its own replay on the same generated inputs; their whole
trajectories must agree."""
import numpy as np
import pytest
import torch

import synth
from oracle import step as ostep

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def stream(B, D_max, V, seed):
    def inputs(t):
        rng = np.random.default_rng(seed * 7919 + t)
        tgt, drf = synth._logits_zipf(rng, B * D_max, V)
        return tgt, drf, synth.philox_uniforms(seed, t, B * D_max)
    return inputs


def gpu_replay(H, W, P, B, V, Hq, d, inputs, max_steps=10000):
    from paper_2606_20543_gb300.step import VerifyStep
    D_max = 2 * W
    c = synth.make_case("replay", grid_h=H, grid_w=W, prefix_len=P, cache_len=[P] * B, Hq=Hq,
                        Hkv=Hq, d=d, V=V, seed=1, with_logits=False)
    s = VerifyStep(H, W, P, B, Hq, Hq, d, D_max, c.L_max, V)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v)
    hist = []
    for t in range(max_steps):
        lp, lq, u = inputs(t)
        s.upload(tgt_logits=lp, drf_logits=lq, uniforms=u)
        s.run()
        nd = s.n_drafts.cpu().numpy()
        if nd.sum() == 0:
            break
        hist.append(dict(cache_len=s.cache_len.cpu().numpy().copy(), n_drafts=nd.copy(),
                         accepted_count=s.accepted_count.cpu().numpy().copy(),
                         accepted_prefix=s.accepted_prefix.cpu().numpy().copy()))
        s.cache_len.copy_(s.next_cache_len)  # device state drives the next step
    assert s.status.item() == 0
    return hist, s.cache_len.cpu().numpy()


def test_reduced_replay_trajectory_matches_oracle(ssd):
    H = W = 16
    P, B, V = 32, 2, 4096
    inputs = stream(B, 2 * W, V, seed=21)
    g_hist, g_final = gpu_replay(H, W, P, B, V, 4, 64, inputs)
    o_hist, _, o_final = ostep.replay(H, W, P, 1, B, 2 * W, inputs)
    # the trajectory depends on the accept decisions only; compare it up to
    # (and including) the first step holding an accept near-tie, if any
    first_tie = next((t for t, h in enumerate(o_hist) if h["accept_ties"]), None)
    n_cmp = len(o_hist) if first_tie is None else first_tie + 1
    assert n_cmp >= 20
    for t in range(n_cmp):
        gh, oh = g_hist[t], o_hist[t]
        for key in ("cache_len", "n_drafts"):
            assert np.array_equal(gh[key], oh[key]), (t, key)
        if t != first_tie:
            for key in ("accepted_count", "accepted_prefix"):
                assert np.array_equal(gh[key], oh[key]), (t, key)
    if first_tie is None:
        assert len(g_hist) == len(o_hist)
        assert np.array_equal(g_final, o_final)
    assert (g_final == P + H * W).all()


def test_replay_resumes_from_a_dumped_state(ssd, tmp_path):
    """Checkpoint / resume: the replay's state (next step, seed, cache
    lengths, committed grid tokens) dumped halfway to a file and loaded into
    a fresh VerifyStep gives the same steps and the same grid as the
    uninterrupted replay; the grid equals the oracle replay's while no
    accept near-tie occurs."""
    from paper_2606_20543_gb300.step import ReplayState, VerifyStep
    H = W = 16
    P, B, V, seed = 32, 2, 4096, 23
    D_max = 2 * W
    inputs = stream(B, D_max, V, seed)
    c = synth.make_case("replay", grid_h=H, grid_w=W, prefix_len=P, cache_len=[P] * B, Hq=4,
                        Hkv=4, d=64, V=V, seed=1, with_logits=False)

    def fresh():
        s = VerifyStep(H, W, P, B, 4, 4, 64, D_max, c.L_max, V)
        s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v)
        s.track_grid()
        return s

    def advance(s, t0, t_stop=None):
        t = t0
        while t_stop is None or t < t_stop:
            lp, lq, u = inputs(t)
            s.upload(tgt_logits=lp, drf_logits=lq, uniforms=u)
            s.run()
            if s.n_drafts.sum().item() == 0:
                return t
            s.advance()
            t += 1
        return t

    full = fresh()
    T = advance(full, 0)
    grid_full = full.grid_tok.cpu().numpy()
    assert (full.cache_len.cpu().numpy() == P + H * W).all() and (grid_full >= 0).all()

    half = fresh()
    advance(half, 0, T // 2)
    path = tmp_path / "replay_state.npz"
    half.state(T // 2, seed).save(path)
    del half
    resumed = fresh()
    t0 = resumed.restore(ReplayState.load(path))
    assert t0 == T // 2
    assert advance(resumed, t0) == T
    assert np.array_equal(resumed.grid_tok.cpu().numpy(), grid_full)
    assert full.status.item() == 0 and resumed.status.item() == 0

    o_hist, o_grid, _ = ostep.replay(H, W, P, 1, B, D_max, inputs)
    if not any(h["accept_ties"] for h in o_hist):
        assert np.array_equal(grid_full, o_grid)
