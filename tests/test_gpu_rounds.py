"""GPU parity of r verify-and-correct rounds and the staged schedule (Sec. 3.3;
App. multi-row drafting) against the oracle: tokens and accept flags round by
round (bit-exact except rows after a counted near-tie), the reference pointers
the library redirects, and the commits."""
import numpy as np
import pytest
import torch

import synth
from oracle import rounds as ord_
from oracle import step as ostep

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def _dev_f32(x):
    return torch.from_numpy(np.ascontiguousarray(x, dtype=np.float32)).cuda()


def _clean_rows(o, upto):
    """Rows with no near-tie in rounds 0..upto (their state is comparable)."""
    return ~o["tie"][:upto + 1].any(0)


@pytest.mark.parametrize("strategy", ["accept_reject", "sample"])
def test_rounds_match_oracle_with_reference_pointers(ssd, strategy):
    rng = np.random.default_rng(31)
    rows, V, r = 96, 16384, 3
    drf = synth._logits_normal(rng, rows, V)[1]
    tg = []
    for k in range(r):  # targets drift from round to round
        t = synth._logits_normal(rng, rows, V)[0]
        if k:
            t = 0.7 * tg[-1] + 0.3 * t
        tg.append(t.astype(np.float32))
    u = np.stack([synth.philox_uniforms(9, k, rows) for k in range(r)])
    o = ord_.verify_rounds(tg, drf, u, strategy=strategy)

    d_drf = _dev_f32(drf)
    d_tg = [_dev_f32(t) for t in tg]
    ref_rows = ssd.row_addresses(d_drf)
    tok = [torch.empty(rows, dtype=torch.int32, device="cuda") for _ in range(2)]
    acc = torch.empty(rows, dtype=torch.uint8, device="cuda")
    ratio = torch.empty(rows, dtype=torch.float32, device="cuda")
    st = torch.zeros(1, dtype=torch.int32, device="cuda")
    cur = 0
    for k in range(r):
        uk = torch.from_numpy(u[k].astype(np.float32)).cuda()
        ssd.ssd_accept_round(strategy, rows, V, d_tg[k], V, ref_rows,
                             None if k == 0 else tok[cur], 1.0, ssd.rng(0, 0, uk), tok[1 - cur],
                             acc, ratio, None, st)
        cur = 1 - cur
        torch.cuda.synchronize()
        assert st.item() == 0
        ok = _clean_rows(o, k)
        got_tok = tok[cur].cpu().numpy()
        assert np.array_equal(got_tok[ok], o["tokens"][k + 1][ok]), f"round {k + 1} tokens"
        assert np.array_equal(acc.cpu().numpy().astype(bool)[ok], o["accepted"][k][ok])
        # every clean row's reference points at the draft row or at the target
        # row of the round that last rejected it
        addr = ref_rows.cpu().numpy()
        want = np.where(o["ref"][k + 1] == 0, d_drf.data_ptr() + np.arange(rows) * V * 4, 0)
        for j in range(1, k + 2):
            sel = o["ref"][k + 1] == j
            want[sel] = d_tg[j - 1].data_ptr() + np.arange(rows)[sel] * V * 4
        assert np.array_equal(addr[ok], want[ok]), f"round {k + 1} references"
    assert _clean_rows(o, r - 1).sum() >= rows - rows // 10  # chained rounds: ties accumulate
    assert (~o["accepted"][0]).sum() > rows // 3  # the rounds really redirect references


def _round_case(seed, grid, W, P, cache_len, V, r, Hq=4, d=64):
    c = synth.make_case("rounds", grid_h=grid, grid_w=W, prefix_len=P, cache_len=cache_len,
                        Hq=Hq, Hkv=Hq, d=d, V=V, seed=seed)
    rng = np.random.default_rng(seed + 100)
    tg = [c.tgt_logits]
    for _ in range(r - 1):
        tg.append((0.6 * tg[-1] + 0.4 * synth._logits_normal(rng, c.B * c.D_max, V)[0])
                  .astype(np.float32))
    u = np.stack([synth.philox_uniforms(seed, k, c.B * c.D_max) for k in range(r)])
    return c, tg, u


def test_step_rounds_commit_the_block(ssd):
    from paper_2606_20543_gb300.step import VerifyRounds, VerifyStep
    r = 2
    c, tg, u = _round_case(41, 16, 16, 32, [32 + 16 * 5, 32 + 16 * 9 + 3], 4096, r)
    s = VerifyStep(c.grid_h, c.grid_w, c.prefix_len, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max,
                   c.V)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, tgt_logits=tg[0], drf_logits=c.drf_logits)
    rounds = VerifyRounds(s)
    d_tg = [_dev_f32(t) for t in tg]
    d_u = [torch.from_numpy(x.astype(np.float32)).cuda() for x in u]
    # round 1 (ref_init) must write every reference itself: start from a valid
    # address that is wrong for every row
    rounds.ref_rows.fill_(d_tg[1].data_ptr())
    rounds.run(d_tg, "block", uniforms_rounds=d_u)
    torch.cuda.synchronize()
    res = s.results()
    assert res["status"][0] == 0
    ref = ostep.accept_step(c.grid_h, c.grid_w, c.prefix_len, c.k_v, c.cache_len, c.D_max,
                            tg[0], c.drf_logits, u[0])
    rows = ref["decisions"]["rows"]
    o = ord_.verify_rounds([t[rows] for t in tg], c.drf_logits[rows], u[:, rows])
    ok = _clean_rows(o, r - 1)
    got = rounds.tokens.cpu().numpy()[rows]
    assert np.array_equal(got[ok], o["tokens"][-1][ok])
    assert np.array_equal(res["n_drafts"], ref["n_drafts"])
    # the last round commits the whole block
    assert np.array_equal(res["next_cache_len"], c.cache_len + res["n_drafts"])


def test_staged_schedule_matches_oracle(ssd):
    from paper_2606_20543_gb300.step import VerifyRounds, VerifyStep
    b, i, W, P = 2, 2, 16, 32
    c, tg, _ = _round_case(51, 16, W, P, [P + W * 4, P + W * 10], 4096, b + i)
    assert c.k_v == 1 and c.D_max == 2 * W
    rows_n = c.B * c.D_max
    rng = np.random.default_rng(52)
    u_oracle = rng.random((b + i, rows_n, 2)).astype(np.float32)  # oracle layout per sequence
    # GPU layout: the incremental rounds see the trailing row in slots 0..W-1
    u_gpu = u_oracle.copy()
    tg_gpu = [t.copy() for t in tg]
    for k in range(b, b + i):
        for bb in range(c.B):
            base = bb * c.D_max
            u_gpu[k][base:base + W] = u_oracle[k][base + W:base + 2 * W]
            tg_gpu[k][base:base + W] = tg[k][base + W:base + 2 * W]
    s = VerifyStep(c.grid_h, c.grid_w, c.prefix_len, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max,
                   c.V, k_v=1)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, tgt_logits=tg[0], drf_logits=c.drf_logits)
    rounds = VerifyRounds(s)
    d_tg = [_dev_f32(t) for t in tg_gpu]
    d_u = [torch.from_numpy(x).cuda() for x in u_gpu]
    # base stage only first, to read the first row after round b
    rounds.run(d_tg[:b], "first_row", uniforms_rounds=d_u[:b])
    torch.cuda.synchronize()
    after_base = rounds.tokens.cpu().numpy().copy()
    assert np.array_equal(s.next_cache_len.cpu().numpy(), c.cache_len + W)
    rounds.reset()
    s.upload(cache_len=c.cache_len)
    rounds.run_staged(b, i, d_tg, uniforms_rounds=d_u)
    torch.cuda.synchronize()
    assert s.status.item() == 0
    final = rounds.tokens.cpu().numpy()
    assert np.array_equal(s.next_cache_len.cpu().numpy(), c.cache_len + 2 * W)
    for bb in range(c.B):
        sl = slice(bb * c.D_max, (bb + 1) * c.D_max)
        first, trail, base, inc = ord_.verify_staged(
            b, i, W, [t[sl] for t in tg], c.drf_logits[sl], [x[sl] for x in u_oracle])
        ok_b = ~base["tie"].any(0)
        assert np.array_equal(after_base[sl][:W][ok_b[:W]], first[ok_b[:W]])
        ok_t = ok_b[W:] & ~inc["tie"].any(0)
        assert np.array_equal(final[sl][:W][ok_t], trail[ok_t])
