"""GPU parity of the fused lm_head + acceptance (step a6, tcgen05/TMEM)
against the oracle: logits H W in float64 from the same bf16 inputs, then
strategy (C).  Log-sum-exp and ratio within 1e-5 relative; decisions and
tokens bit-exact except counted near-ties."""
import numpy as np
import pytest
import torch

import synth
from oracle import lmhead as olm
from oracle import step as ostep
from tests.helpers import (FUSED_PROB_TOL, bf16_to_f64, committed_draws, compare_decisions,
                           max_excused_rows)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def _bf(x):
    return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()


def run_fused(ssd, ht, hd, wt, wd, u, draft_tok=None, T=1.0):
    rows, K = ht.shape
    V = wt.shape[1]
    dev = "cuda"
    out_tok = torch.full((rows,), -7, dtype=torch.int32, device=dev)
    acc = torch.full((rows,), 7, dtype=torch.uint8, device=dev)
    ratio = torch.zeros(rows, dtype=torch.float32, device=dev)
    lse = torch.zeros((rows, 2), dtype=torch.float32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    wsb = ssd.ssd_lmhead_accept_workspace(rows, V)
    ws = torch.empty(wsb, dtype=torch.uint8, device=dev)
    dt = None if draft_tok is None else torch.from_numpy(draft_tok.astype(np.int32)).to(dev)
    ssd.ssd_lmhead_accept(rows, V, K, _bf(ht), _bf(hd), _bf(wt), _bf(wd), dt, T,
                          ssd.rng(0, 0, torch.from_numpy(u).to(dev)), out_tok, acc, ratio, lse,
                          ws, wsb, status)
    torch.cuda.synchronize()
    return (out_tok.cpu().numpy(), acc.cpu().numpy(), ratio.cpu().numpy(), lse.cpu().numpy(),
            int(status.item()))


def make_inputs(rows, K, V, seed, w_std=0.02):
    rng = np.random.default_rng(seed)
    return (synth.bf16_normal(rng, (rows, K), 1.0), synth.bf16_normal(rng, (rows, K), 1.0),
            synth.bf16_normal(rng, (K, V), w_std), synth.bf16_normal(rng, (K, V), w_std),
            synth.philox_uniforms(seed, 0, rows))


@pytest.mark.parametrize("rows,K,V,w_std,seed", [
    (8, 128, 256, 0.1, 0),        # two vocabulary tiles, two K stages
    (48, 512, 2048, 0.05, 1),     # 16 tiles, ragged ring wrap-around (8 K blocks, 3 stages)
    (200, 256, 1024, 0.05, 2),    # two row tiles (rows 128..199 in the second)
    (48, 4096, 16384, 0.02, 3),   # the fused-head workload: 128 tiles, 64 K blocks
    (256, 4096, 16384, 0.02, 4),  # the most rows: two full row tiles, two rows per CTA's combine
])
def test_fused_lmhead_matches_oracle(ssd, rows, K, V, w_std, seed):
    ht, hd, wt, wd, u = make_inputs(rows, K, V, seed, w_std)
    tok, acc, ratio, lse, st = run_fused(ssd, ht, hd, wt, wd, u)
    assert st == 0
    ref = olm.lmhead_accept(bf16_to_f64(ht), bf16_to_f64(hd), bf16_to_f64(wt), bf16_to_f64(wd), u)
    ties = compare_decisions(ref, tok, acc, ratio, lse, what=f"rows={rows} V={V}",
                             tol=FUSED_PROB_TOL)
    assert ties <= max_excused_rows(rows)  # also enforced inside compare_decisions


def test_fused_given_token_and_temperature(ssd):
    rows, K, V = 32, 256, 1024
    ht, hd, wt, wd, u = make_inputs(rows, K, V, 7, 0.1)
    dt = np.random.default_rng(7).integers(0, V, rows)
    for T in (1.0, 0.6):
        tok, acc, ratio, lse, st = run_fused(ssd, ht, hd, wt, wd, u, draft_tok=dt, T=T)
        assert st == 0
        ref = olm.lmhead_accept(bf16_to_f64(ht), bf16_to_f64(hd), bf16_to_f64(wt),
                                bf16_to_f64(wd), u, draft_tok=dt, temperature=T)
        compare_decisions(ref, tok, acc, ratio, lse, what=f"T={T}", tol=FUSED_PROB_TOL)


def test_fused_identical_heads_accept_everything(ssd):
    rows, K, V = 16, 128, 512
    ht, _, wt, _, u = make_inputs(rows, K, V, 9, 0.1)
    u[:, 0] = 1 - 2**-24
    tok, acc, ratio, _, st = run_fused(ssd, ht, ht.copy(), wt, wt.copy(), u)
    assert st == 0 and acc.all() and np.all(ratio == 1.0)


@pytest.mark.parametrize("points", [[120, 672], [120, 130, 140, 150, 160]])
def test_verify_step_fused_path(ssd, points):
    """ssd_verify_step with hidden states + lm_head weights (config-4 shapes:
    a full 48-draft frontier and a 24-draft last row; five sequences, 240
    rows in two row tiles).  The prefix commit draws only each sequence's
    first rejected draft."""
    from paper_2606_20543_gb300.step import VerifyStep
    c = synth.config4(points=points)
    s = VerifyStep(c.grid_h, c.grid_w, c.prefix_len, c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max, c.V,
                   hidden=c.hidden)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v, h_tgt=c.h_tgt, h_drf=c.h_drf,
             w_tgt=c.w_tgt, w_drf=c.w_drf, uniforms=c.uniforms)
    s.run()
    torch.cuda.synchronize()
    r = s.results()
    assert r["status"][0] == 0
    lp = olm.logits(bf16_to_f64(c.h_tgt), bf16_to_f64(c.w_tgt))
    lq = olm.logits(bf16_to_f64(c.h_drf), bf16_to_f64(c.w_drf))
    ref = ostep.accept_step(c.grid_h, c.grid_w, c.prefix_len, c.k_v, c.cache_len, c.D_max, lp, lq,
                            c.uniforms)
    assert np.array_equal(r["n_drafts"], ref["n_drafts"])
    rows = ref["decisions"]["rows"]
    # a prefix-commit step draws only each sequence's first rejected draft
    dec = committed_draws(ref["decisions"], r["accepted"][rows], c.D_max)
    ties = compare_decisions(dec, r["out_tok"][rows], r["accepted"][rows],
                             r["ratio"][rows], what="fused step", tol=FUSED_PROB_TOL)
    pad = np.setdiff1d(np.arange(c.B * c.D_max), rows)
    assert np.all(r["out_tok"][pad] == -1) and np.all(r["accepted"][pad] == 0)
    if ties == 0:
        assert np.array_equal(r["next_cache_len"], ref["next_cache_len"])
