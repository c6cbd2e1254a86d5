"""Parity at the full sizes of the five verification workloads, in the launch
configuration bench.py times: one ssd_verify_step over the whole batch.
Decisions, counts and frontiers of every row are compared with the oracle;
attention on every sequence (config 2, 3) or on sampled sequences and heads
(config 5, where the oracle computes rows one by one); the config-5 replay is
checked step by step against the oracle's own replay for its first steps and
by invariants to grid completion."""
import numpy as np
import pytest
import torch

import synth
from oracle import step as ostep
from tests.helpers import ATTN_TOL, attention_error, bf16_to_f64, committed_draws, compare_decisions

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def run_case(c):
    from paper_2606_20543_gb300.step import VerifyStep
    s = VerifyStep(c.grid_h, c.grid_w, c.prefix_len, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max, c.V,
                   k_v=c.k_v)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, tgt_logits=c.tgt_logits,
             drf_logits=c.drf_logits, uniforms=c.uniforms)
    s.run()
    torch.cuda.synchronize()
    return s, s.results()


def check_decisions(c, r):
    ref = ostep.accept_step(c.grid_h, c.grid_w, c.prefix_len, c.k_v, c.cache_len, c.D_max,
                            c.tgt_logits, c.drf_logits, c.uniforms)
    assert r["status"][0] == 0
    assert np.array_equal(r["n_drafts"], ref["n_drafts"])
    assert np.array_equal(r["draft_pos"], ref["draft_pos"])
    rows = ref["decisions"]["rows"]
    dec = committed_draws(ref["decisions"], r["accepted"][rows], c.D_max)
    ties = compare_decisions(dec, r["out_tok"][rows], r["accepted"][rows], r["ratio"][rows],
                             what=c.name)
    if ties == 0:
        assert np.array_equal(r["accepted_count"], ref["accepted_count"])
        assert np.array_equal(r["next_cache_len"], ref["next_cache_len"])
    return ties


def check_attention(c, r, seqs=None, heads=None):
    att = ostep.attention_step(c.grid_h, c.grid_w, c.prefix_len, c.row_stride, c.k_v,
                               c.cache_len, bf16_to_f64(c.q), bf16_to_f64(c.k), bf16_to_f64(c.v),
                               c.Hq, c.Hkv, None, seqs)
    for b, (o_ref, _) in att.items():
        n = o_ref.shape[0]
        for h in (range(c.Hq) if heads is None else heads):
            if n:
                assert attention_error(r["o"][b, :n, h], o_ref[:, h]) < ATTN_TOL, (b, h)


def test_config2_full_sweep(ssd):
    c = synth.config2()
    _, r = run_case(c)
    check_decisions(c, r)
    check_attention(c, r)


def test_config3_full_batch(ssd):
    c = synth.config3()
    _, r = run_case(c)
    check_decisions(c, r)
    check_attention(c, r)


def test_config1_both_cache_lengths(ssd):
    for cl in (192, 112):
        c = synth.config1(cache_len=cl)
        _, r = run_case(c)
        check_decisions(c, r)
        check_attention(c, r)


def _config5_runner(c, pool):
    from paper_2606_20543_gb300.step import VerifyStep
    s = VerifyStep(c.grid_h, c.grid_w, c.prefix_len, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max, c.V)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v)
    dev_pool = [(torch.from_numpy(t).cuda(), torch.from_numpy(d).cuda()) for t, d in pool]
    return s, dev_pool


def _step(s, dev_pool, seed, t):
    tg, dr = dev_pool[t % len(dev_pool)]
    s.args.tgt_logits, s.args.drf_logits = tg.data_ptr(), dr.data_ptr()
    s.set_rng(seed, t)
    s.run()


def test_config5_first_steps_match_oracle_replay(ssd):
    """Full size (8 x 64x64, V = 65536): the first replay steps, with device
    state driving the next cache length, against the oracle's own replay."""
    c = synth.config5(with_logits=False)
    pool = synth.replay_pool(c.B, c.D_max, c.V, seed=c.seed)
    s, dev_pool = _config5_runner(c, pool)
    n_steps = 3

    def inputs(t):
        tg, dr = pool[t % len(pool)]
        return tg, dr, synth.philox_uniforms(c.seed, t, c.B * c.D_max)

    o_hist, _, _ = ostep.replay(c.grid_h, c.grid_w, c.prefix_len, c.k_v, c.B, c.D_max, inputs,
                                max_steps=n_steps)
    for t in range(n_steps):
        _step(s, dev_pool, c.seed, t)
        torch.cuda.synchronize()
        oh = o_hist[t]
        assert np.array_equal(s.cache_len.cpu().numpy(), oh["cache_len"]), t
        assert np.array_equal(s.n_drafts.cpu().numpy(), oh["n_drafts"]), t
        if oh["accept_ties"] == 0:
            assert np.array_equal(s.accepted_count.cpu().numpy(), oh["accepted_count"]), t
            assert np.array_equal(s.accepted_prefix.cpu().numpy(), oh["accepted_prefix"]), t
        else:
            break
        if t == 0:
            # the first step row by row: accept flags, committed tokens and
            # ratios of every draft, and attention on every head of two sequences
            r = s.results()
            tg, dr, u = inputs(0)
            ref = ostep.accept_step(c.grid_h, c.grid_w, c.prefix_len, c.k_v, oh["cache_len"],
                                    c.D_max, tg, dr, u)
            rows = ref["decisions"]["rows"]
            dec = committed_draws(ref["decisions"], r["accepted"][rows], c.D_max)
            compare_decisions(dec, r["out_tok"][rows], r["accepted"][rows], r["ratio"][rows],
                              what="cfg5 step 0")
            check_attention(c, r, seqs=[0, 5])
        s.cache_len.copy_(s.next_cache_len)
    assert s.status.item() == 0


def test_config5_replay_to_completion_invariants(ssd):
    c = synth.config5(with_logits=False)
    pool = synth.replay_pool(c.B, c.D_max, c.V, seed=c.seed + 1)
    s, dev_pool = _config5_runner(c, pool)
    HW = c.grid_h * c.grid_w
    prev = s.cache_len.cpu().numpy().copy()
    total = np.zeros(c.B, np.int64)
    steps = 0
    for t in range(2 * HW):
        _step(s, dev_pool, c.seed + 1, t)
        nd = s.n_drafts.cpu().numpy()
        if nd.sum() == 0:
            break
        nxt = s.next_cache_len.cpu().numpy()
        cnt = s.accepted_count.cpu().numpy()
        pre = s.accepted_prefix.cpu().numpy()
        adv = nxt - prev
        assert ((adv >= 1) | (nd == 0)).all() and (adv <= nd).all()
        assert ((pre <= cnt) & (cnt <= nd)).all()
        total += adv
        prev = nxt.copy()
        s.cache_len.copy_(s.next_cache_len)
        steps += 1
    assert (prev == c.prefix_len + HW).all() and (total == HW).all()
    assert s.status.item() == 0
    assert steps >= HW // (2 * c.grid_w)  # at most two rows per step


@pytest.mark.parametrize("B", [8, 2])
def test_config5_late_step_every_row(ssd, B):
    """A teacher-forced late step of the 64x64 replay at full size (V = 65536,
    up to 128 drafts per sequence, caches of about 4100 to 4350 keys): every
    row's accept flag, committed token and ratio against the oracle, and the
    attention of every head of two sequences.  B = 8 is the bench's launch;
    with B = 2 the attention splits every KV cache over several CTAs and
    merges the partials (the split-KV path)."""
    rng = np.random.default_rng(50 + B)
    cl = 256 + 64 * rng.integers(59, 63, size=B) + rng.integers(0, 64, size=B)
    cl[0] = 256 + 64 * 62  # a frontier of two whole rows: 128 drafts
    c = synth.config5(B=B, cache_len=cl.astype(np.int32), seed=51 + B)
    _, r = run_case(c)
    check_decisions(c, r)
    check_attention(c, r, seqs=[0, B - 1])


@pytest.mark.parametrize("active", [1, 2])
def test_config5_tail_step_every_row(ssd, active):
    """The end of the 8-sequence replay: `active` sequences still have drafts
    (caches of about 4100 to 4350 keys), the other grids are complete (cache
    = prefix + 4096, empty frontier: no rows, no attention items, ranked last
    in the attention's dealing).  Every row's decisions and the attention of
    every head of the active sequences against the oracle."""
    B = 8
    rng = np.random.default_rng(70 + active)
    cl = np.full(B, 256 + 64 * 64)
    act = np.sort(rng.choice(B, size=active, replace=False))
    cl[act] = 256 + 64 * rng.integers(59, 63, size=active) + rng.integers(0, 64, size=active)
    c = synth.config5(B=B, cache_len=cl.astype(np.int32), seed=71 + active)
    _, r = run_case(c)
    assert (r["n_drafts"][np.setdiff1d(np.arange(B), act)] == 0).all()
    check_decisions(c, r)
    check_attention(c, r, seqs=[int(b) for b in act])
