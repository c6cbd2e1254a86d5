"""GPU parity of the whole verification step (steps a1-a5, a7) through
ssd_verify_step against the oracle: frontier and counts bit-exact,
attention within 2e-2, decisions bit-exact except counted near-ties."""
import numpy as np
import pytest
import torch

import synth
from oracle import step as ostep
from oracle import frontier as ofr
from tests.helpers import ATTN_TOL, attention_error, bf16_to_f64, committed_draws, compare_decisions

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def make_step(c, strategy="accept_reject"):
    from paper_2606_20543_gb300.step import VerifyStep
    s = VerifyStep(c.grid_h, c.grid_w, c.prefix_len, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max, c.V,
                   k_v=c.k_v, strategy=strategy)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, tgt_logits=c.tgt_logits,
             drf_logits=c.drf_logits, uniforms=c.uniforms)
    return s


def check_step(c, res, attention_seqs=None, strategy="accept_reject"):
    ref = ostep.accept_step(c.grid_h, c.grid_w, c.prefix_len, c.k_v, c.cache_len, c.D_max,
                            c.tgt_logits, c.drf_logits, c.uniforms, strategy=strategy)
    assert res["status"][0] == 0
    assert np.array_equal(res["n_drafts"], ref["n_drafts"])
    assert np.array_equal(res["draft_pos"], ref["draft_pos"])
    rows = ref["decisions"]["rows"]
    ties = 0
    if rows.size:
        dec = ref["decisions"]
        if strategy == "accept_reject":  # prefix rule: only the committed rejection is drawn
            dec = committed_draws(dec, res["accepted"][rows], c.D_max)
        ties = compare_decisions(dec, res["out_tok"][rows], res["accepted"][rows],
                                 res["ratio"][rows], what=c.name)
    # padding rows
    pad = np.setdiff1d(np.arange(c.B * c.D_max), rows)
    assert np.all(res["out_tok"][pad] == -1) and np.all(res["accepted"][pad] == 0)
    if ties == 0:
        assert np.array_equal(res["accepted_count"], ref["accepted_count"])
        assert np.array_equal(res["accepted_prefix"], ref["accepted_prefix"])
        assert np.array_equal(res["next_cache_len"], ref["next_cache_len"])
    att = ostep.attention_step(c.grid_h, c.grid_w, c.prefix_len, c.row_stride, c.k_v, c.cache_len,
                               bf16_to_f64(c.q), bf16_to_f64(c.k), bf16_to_f64(c.v), c.Hq, c.Hkv,
                               None, attention_seqs)
    for b, (o_ref, _) in att.items():
        n = o_ref.shape[0]
        for h in range(c.Hq):
            if n:
                assert attention_error(res["o"][b, :n, h], o_ref[:, h]) < ATTN_TOL
    return ties


def test_step_config1(ssd):
    for cl in (192, 112):
        c = synth.config1(cache_len=cl)
        s = make_step(c)
        s.run()
        torch.cuda.synchronize()
        check_step(c, s.results())


def test_step_config2_sweep_subset(ssd):
    c = synth.config2(points=[120, 312, 648, 672, 696])
    s = make_step(c)
    s.run()
    torch.cuda.synchronize()
    check_step(c, s.results())


def test_step_config3_shape(ssd):
    # config-3 shapes with fewer sequences (full size is in test_gpu_fullsize)
    c = synth.config3(B=4)
    s = make_step(c)
    s.run()
    torch.cuda.synchronize()
    check_step(c, s.results())


def test_frontier_all_cache_lengths(ssd):
    """Every cache length of a 24x24 grid, k_v = 0, 1 and 2, bit-exact."""
    dev = "cuda"
    for k_v in (0, 1, 2):
        H = W = 24
        P = 120
        cls = np.arange(P, P + H * W + 1, dtype=np.int32)
        D_max = (k_v + 1) * W
        g = ssd.grid(H, W, P, k_v=k_v)
        nd = torch.empty(len(cls), dtype=torch.int32, device=dev)
        pos = torch.empty((len(cls), D_max), dtype=torch.int32, device=dev)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        ssd.ssd_frontier(g, len(cls), torch.from_numpy(cls).to(dev), D_max, nd, pos, st)
        torch.cuda.synchronize()
        nd, pos = nd.cpu().numpy(), pos.cpu().numpy()
        assert st.item() == 0
        for i, cl in enumerate(cls):
            gidx = ofr.grid_index(ofr.frontier(H, W, P, int(cl), k_v), W)
            assert nd[i] == len(gidx)
            assert np.array_equal(pos[i, :nd[i]], gidx)
            assert np.all(pos[i, nd[i]:] == -1)


def test_counts_all_accept_and_all_reject(ssd):
    c = synth.config1(cache_len=192)
    # identical logits: every draft accepted, the whole frontier committed
    c.tgt_logits = c.drf_logits.copy()
    s = make_step(c)
    s.run()
    torch.cuda.synchronize()
    r = s.results()
    assert r["accepted_count"][0] == 32 and r["accepted_prefix"][0] == 32
    assert r["next_cache_len"][0] == 192 + 32
    # disjoint supports: every draft rejected, one correction token committed
    lp = np.full_like(c.drf_logits, -40.0)
    lq = np.full_like(c.drf_logits, -40.0)
    lp[:, :2048] = 0.0
    lq[:, 2048:] = 0.0
    s.upload(tgt_logits=lp, drf_logits=lq)
    s.run()
    torch.cuda.synchronize()
    r = s.results()
    assert r["accepted_count"][0] == 0 and r["accepted_prefix"][0] == 0
    assert r["next_cache_len"][0] == 193
    assert np.all(r["out_tok"][:32] < 2048)


def test_step_large_batch_of_small_grids(ssd):
    """1100 sequences of 4x4 grids with mixed cache lengths (some complete,
    n_drafts = 0): far more rows than CTAs, padding slots among them."""
    rng = np.random.default_rng(21)
    H = W = 4
    P = 8
    cls = rng.integers(P, P + H * W + 1, size=1100).astype(np.int32)
    c = synth.make_case("many", grid_h=H, grid_w=W, prefix_len=P, cache_len=cls, Hq=1, Hkv=1,
                        d=64, V=64, seed=21)
    s = make_step(c)
    s.run()
    torch.cuda.synchronize()
    check_step(c, s.results(), attention_seqs=[0, 1, 550, 1099])


@pytest.mark.parametrize("strategy", ["greedy", "sample"])
def test_step_strategies(ssd, strategy):
    """The whole step under strategies (A) and (B): the prefix rule of the
    counts reads the accepted flags (selected token == draft token)."""
    for c in (synth.config1(cache_len=192, seed=3), synth.config2(points=[120, 480, 672])):
        s = make_step(c, strategy)
        s.run()
        torch.cuda.synchronize()
        check_step(c, s.results(), strategy=strategy)


def test_frontier_with_k_h_all_cache_lengths(ssd):
    """The horizontal stage's frontier (k_h = 5) for every cache length of a
    24x24 grid, with and without rows below, bit-exact."""
    dev = "cuda"
    H = W = 24
    P = 120
    cls = np.arange(P, P + H * W + 1, dtype=np.int32)
    for k_v in (0, 1):
        D_max = (k_v + 1) * W
        g = ssd.grid(H, W, P, k_v=k_v, k_h=5)
        nd = torch.empty(len(cls), dtype=torch.int32, device=dev)
        pos = torch.empty((len(cls), D_max), dtype=torch.int32, device=dev)
        st = torch.zeros(1, dtype=torch.int32, device=dev)
        ssd.ssd_frontier(g, len(cls), torch.from_numpy(cls).to(dev), D_max, nd, pos, st)
        torch.cuda.synchronize()
        nd, pos = nd.cpu().numpy(), pos.cpu().numpy()
        assert st.item() == 0
        for i, cl in enumerate(cls):
            gidx = ofr.grid_index(ofr.frontier(H, W, P, int(cl), k_v, 5), W)
            assert nd[i] == len(gidx)
            assert np.array_equal(pos[i, :nd[i]], gidx)


@pytest.mark.parametrize("strategy", ["accept_reject", "greedy", "sample"])
def test_horizontal_stage_with_bonus(ssd, strategy):
    """k_h = 5 drafts, one round, prefix acceptance plus the bonus token."""
    from paper_2606_20543_gb300.step import VerifyStep
    H = W = 16
    P = 32
    cls = [P + 3, P + W * 2, P + W * 5 + 13, P + H * W - 2, P + W * 7 + 11]
    c = synth.make_case("horizontal", grid_h=H, grid_w=W, prefix_len=P, cache_len=cls, Hq=4,
                        Hkv=4, d=64, V=4096, seed=61, k_v=0)
    for same in (False, True):  # True: p = q, every draft accepted, the bonus committed
        tgt = c.drf_logits.copy() if same else c.tgt_logits
        s = VerifyStep(H, W, P, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max, c.V, k_v=0, k_h=5,
                       strategy=strategy, commit="prefix_bonus")
        s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, tgt_logits=tgt,
                 drf_logits=c.drf_logits, uniforms=c.uniforms)
        s.run()
        torch.cuda.synchronize()
        res = s.results()
        assert res["status"][0] == 0
        ref = ostep.accept_step(H, W, P, 0, c.cache_len, c.D_max, tgt, c.drf_logits, c.uniforms,
                                strategy=strategy, k_h=5, bonus=True)
        assert np.array_equal(res["n_drafts"], ref["n_drafts"])
        assert np.array_equal(res["n_drafts"], [5, 5, 3, 2, 5])
        rows = ref["decisions"]["rows"]
        lazy = strategy == "accept_reject"  # draws only what the counts commit
        dec = committed_draws(ref["decisions"], res["accepted"][rows], c.D_max) if lazy \
            else ref["decisions"]
        ties = compare_decisions(dec, res["out_tok"][rows], res["accepted"][rows],
                                 what=f"horizontal {strategy}")
        for b in range(c.B):
            br = ref["bonus_row"][b]
            if br < 0:
                continue
            all_acc = res["accepted_prefix"][b] == res["n_drafts"][b]
            if lazy and not all_acc:
                assert res["out_tok"][br] == -1  # not committed: not drawn
            elif not ref["bonus_tie"][b]:
                assert res["out_tok"][br] == ref["bonus_tok"][b]
                assert res["accepted"][br] == 1
        if ties == 0:
            assert np.array_equal(res["next_cache_len"], ref["next_cache_len"])
        if same and strategy != "sample":
            # every draft accepted: the bonus is committed except at the grid's end
            assert np.array_equal(res["next_cache_len"][[0, 1, 2, 4]],
                                  c.cache_len[[0, 1, 2, 4]] + res["n_drafts"][[0, 1, 2, 4]] + 1)
            assert res["next_cache_len"][3] == c.cache_len[3] + 2


def _full_draw(ssd, s, c, strategy="accept_reject"):
    """ssd_accept_strategy over every row of the padded batch with the step's
    logits and uniforms: the full (eager) draw of every row."""
    rows = c.B * c.D_max
    out_tok = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
    acc = torch.zeros(rows, dtype=torch.uint8, device="cuda")
    ratio = torch.zeros(rows, dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    ssd.ssd_accept_strategy(strategy, rows, c.V, s.tgt, s.drf, c.V, None, 1.0, s.rng, out_tok,
                            acc, ratio, None, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    return out_tok.cpu().numpy(), acc.cpu().numpy(), ratio.cpu().numpy()


def test_committed_draw_is_the_full_draw_bit_for_bit(ssd):
    """Under the prefix rule the step draws only each sequence's first
    rejected draft; that token, every accept flag and every ratio are the
    ones the full draw over every row gives, bit for bit (same block masses,
    scan, re-walk and Philox counters), on a ragged multi-tile batch."""
    c = synth.config2(points=[120, 192, 312, 480, 552, 648, 672, 696])
    s = make_step(c)
    s.run()
    torch.cuda.synchronize()
    r = s.results()
    tok_f, acc_f, ratio_f = _full_draw(ssd, s, c)
    firsts = 0
    for b in range(c.B):
        n = int(r["n_drafts"][b])
        rows = np.arange(b * c.D_max, b * c.D_max + n)
        assert np.array_equal(r["accepted"][rows], acc_f[rows])
        assert np.array_equal(r["ratio"][rows].view(np.uint32), ratio_f[rows].view(np.uint32))
        rej = rows[acc_f[rows] == 0]
        acc_rows = rows[acc_f[rows] == 1]
        assert np.array_equal(r["out_tok"][acc_rows], tok_f[acc_rows])
        if rej.size:
            firsts += 1
            assert r["out_tok"][rej[0]] == tok_f[rej[0]] >= 0
            assert np.all(r["out_tok"][rej[1:]] == -1)
            assert r["accepted_prefix"][b] == rej[0] - b * c.D_max
    assert firsts >= c.B // 2  # the synthetic drafts are rejected early in most sequences


def test_committed_bonus_is_the_full_draw_from_p(ssd):
    """Horizontal stage with p = q (every draft accepted): the bonus row's
    token is the draw from p that strategy (B) makes for that row."""
    from paper_2606_20543_gb300.step import VerifyStep
    H = W = 16
    P = 32
    cls = [P + 3, P + W * 2, P + W * 5 + 13, P + W * 7 + 11]
    c = synth.make_case("horizontal", grid_h=H, grid_w=W, prefix_len=P, cache_len=cls, Hq=4,
                        Hkv=4, d=64, V=4096, seed=62, k_v=0)
    s = VerifyStep(H, W, P, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max, c.V, k_v=0, k_h=5,
                   commit="prefix_bonus")
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, tgt_logits=c.drf_logits,
             drf_logits=c.drf_logits, uniforms=c.uniforms)
    s.run()
    torch.cuda.synchronize()
    r = s.results()
    assert r["status"][0] == 0
    tok_b, _, _ = _full_draw(ssd, s, c, "sample")
    for b in range(c.B):
        n = int(r["n_drafts"][b])
        assert r["accepted_prefix"][b] == n
        br = b * c.D_max + n
        assert r["out_tok"][br] == tok_b[br] >= 0


def test_verify_accept_matches_the_step(ssd):
    """ssd_verify_accept (the step without the attention, on one stream)
    gives the step's frontier, decisions, draws and counts bit for bit."""
    c = synth.config2(points=[120, 408, 696])
    s = make_step(c)
    s.run()
    torch.cuda.synchronize()
    r = s.results()
    for t in (s.out_tok, s.accepted, s.ratio, s.accepted_count, s.accepted_prefix,
              s.next_cache_len, s.n_drafts, s.draft_pos):
        t.fill_(-5 if t.dtype == torch.int32 else 0)
    ssd.ssd_verify_accept(s.args, s.out, s.workspace, s.ws_bytes)
    torch.cuda.synchronize()
    r2 = s.results()
    for k in ("n_drafts", "draft_pos", "out_tok", "accepted", "accepted_count", "accepted_prefix",
              "next_cache_len", "status"):
        assert np.array_equal(r[k], r2[k]), k
    assert np.array_equal(r["ratio"].view(np.uint32), r2["ratio"].view(np.uint32))


@pytest.mark.parametrize("strategy", ["accept_reject", "greedy", "sample"])
def test_horizontal_stage_large_batch(ssd, strategy):
    """The horizontal stage on a batch of 2 x (SM count) padded rows or more, so
    that (C) and (A) take the single-stream schedule (acceptance, attention,
    counts as a dependent beside it) and (B) the two-stream one, against the
    oracle: decisions, committed tokens, bonus tokens and next cache lengths."""
    from paper_2606_20543_gb300.step import VerifyStep
    H = W = 16
    P = 32
    rng = np.random.default_rng(5)
    cls = [int(P + x) for x in rng.choice(H * W - 1, size=20, replace=False)]
    c = synth.make_case("horizontal", grid_h=H, grid_w=W, prefix_len=P, cache_len=cls, Hq=4,
                        Hkv=4, d=64, V=4096, seed=71, k_v=0)
    assert c.B * c.D_max >= 2 * torch.cuda.get_device_properties(0).multi_processor_count
    s = VerifyStep(H, W, P, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max, c.V, k_v=0, k_h=5,
                   strategy=strategy, commit="prefix_bonus")
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, tgt_logits=c.tgt_logits,
             drf_logits=c.drf_logits, uniforms=c.uniforms)
    s.run()
    torch.cuda.synchronize()
    res = s.results()
    assert res["status"][0] == 0
    ref = ostep.accept_step(H, W, P, 0, c.cache_len, c.D_max, c.tgt_logits, c.drf_logits,
                            c.uniforms, strategy=strategy, k_h=5, bonus=True)
    assert np.array_equal(res["n_drafts"], ref["n_drafts"])
    rows = ref["decisions"]["rows"]
    lazy = strategy == "accept_reject"
    dec = committed_draws(ref["decisions"], res["accepted"][rows], c.D_max) if lazy \
        else ref["decisions"]
    ties = compare_decisions(dec, res["out_tok"][rows], res["accepted"][rows],
                             what=f"horizontal large {strategy}")
    for b in range(c.B):
        br = ref["bonus_row"][b]
        if br < 0:
            continue
        if lazy and res["accepted_prefix"][b] != res["n_drafts"][b]:
            assert res["out_tok"][br] == -1
        elif not ref["bonus_tie"][b]:
            assert res["out_tok"][br] == ref["bonus_tok"][b]
    if ties == 0:
        assert np.array_equal(res["accepted_count"], ref["accepted_count"])
        assert np.array_equal(res["next_cache_len"], ref["next_cache_len"])
    att = ostep.attention_step(H, W, P, c.row_stride, 0, c.cache_len, bf16_to_f64(c.q),
                               bf16_to_f64(c.k), bf16_to_f64(c.v), c.Hq, c.Hkv, k_h=5)
    for b, (o_ref, _) in att.items():
        n = o_ref.shape[0]
        for h in range(c.Hq):
            if n:
                assert attention_error(res["o"][b, :n, h], o_ref[:, h]) < ATTN_TOL


def test_step_with_masked_vocabulary(ssd):
    """The whole step (one-pass acceptance, committed draws, counts) on logits
    with masked (-inf) vocabulary entries: a quarter of the target's and
    another quarter of the draft's, and the draft tokens of every third row
    masked by the target (always rejected).  Against the oracle; no masked
    token is committed."""
    import copy
    c = copy.copy(synth.config2(points=[120, 312, 480, 672]))
    tg, dr = c.tgt_logits.copy(), c.drf_logits.copy()
    tg[:, :4096] = -np.inf
    dr[:, 8192:12288] = -np.inf
    dr[::3, 7] = 60.0
    c.tgt_logits, c.drf_logits = tg, dr
    s = make_step(c)
    s.run()
    torch.cuda.synchronize()
    res = s.results()
    check_step(c, res)
    assert not np.isin(res["out_tok"], np.arange(4096)).any()
