"""GPU parity of the acceptance kernel (steps a3-a5) against the oracle:
decisions and tokens bit-exact except counted near-ties, ratio and
log-sum-exp within 1e-5 relative."""
import numpy as np
import pytest
import torch

import synth
from oracle import accept as oacc
from tests.helpers import compare_decisions, max_excused_rows

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def run_accept(ssd, tgt, drf, uniforms=None, seed=0, offset=0, draft_tok=None, T=1.0, ld=None,
               strategy="accept_reject"):
    rows, V = tgt.shape
    ld = V if ld is None else ld
    dev = "cuda"
    tg = torch.zeros((rows, ld), dtype=torch.float32, device=dev)
    dg = torch.zeros((rows, ld), dtype=torch.float32, device=dev)
    tg[:, :V] = torch.from_numpy(np.ascontiguousarray(tgt))
    dg[:, :V] = torch.from_numpy(np.ascontiguousarray(drf))
    u = None if uniforms is None else torch.from_numpy(uniforms).to(dev)
    dt = None if draft_tok is None else torch.from_numpy(draft_tok.astype(np.int32)).to(dev)
    out_tok = torch.full((rows,), -7, dtype=torch.int32, device=dev)
    acc = torch.full((rows,), 7, dtype=torch.uint8, device=dev)
    ratio = torch.zeros((rows,), dtype=torch.float32, device=dev)
    lse = torch.zeros((rows, 2), dtype=torch.float32, device=dev)
    status = torch.zeros((1,), dtype=torch.int32, device=dev)
    ssd.ssd_accept_strategy(strategy, rows, V, tg, dg, ld, dt, T, ssd.rng(seed, offset, u),
                            out_tok, acc, ratio, lse, status)
    torch.cuda.synchronize()
    return (out_tok.cpu().numpy(), acc.cpu().numpy(), ratio.cpu().numpy(), lse.cpu().numpy(),
            int(status.item()))


@pytest.mark.parametrize("V,rows,logits,seed", [
    (4096, 64, "normal", 0),      # two 2048-entry chunks per row
    (16384, 48, "normal", 1),     # eight chunks, one row per CTA
    (16384, 40, "zipf", 2),       # skewed draft vs perturbed target
    (4100, 30, "normal", 3),      # ragged: a 4-entry last chunk
    (65536, 8, "zipf", 4),        # 32 chunks per row
    (12, 16, "normal", 5),        # tiny vocabulary
    (16384, 700, "normal", 6),    # more rows than CTAs: each CTA walks several
    (100000, 6, "normal", 7),     # large vocabulary, ragged last chunk
])
def test_accept_matches_oracle(ssd, V, rows, logits, seed):
    rng = np.random.default_rng(seed)
    if logits == "normal":
        tgt, drf = synth._logits_normal(rng, rows, V)
    else:
        tgt, drf = synth._logits_zipf(rng, rows, V)
    u = synth.philox_uniforms(seed, 11, rows)
    tok, acc, ratio, lse, st = run_accept(ssd, tgt, drf, u)
    assert st == 0
    dec = oacc.accept_rows(tgt, drf, u)
    ties = compare_decisions(dec, tok, acc, ratio, lse, what=f"V={V}")
    assert ties <= max_excused_rows(rows)  # also enforced inside compare_decisions


def test_device_philox_matches_generator(ssd):
    """uniforms=NULL draws Philox4x32-10 on the device; it must reproduce the
    generator's stream bit for bit, so both runs decide identically."""
    rng = np.random.default_rng(7)
    rows, V = 512, 4096
    tgt, drf = synth._logits_normal(rng, rows, V)
    a = run_accept(ssd, tgt, drf, synth.philox_uniforms(1234567890123, 99, rows))
    b = run_accept(ssd, tgt, drf, None, seed=1234567890123, offset=99)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    # and the decisions really depend on the uniforms
    c = run_accept(ssd, tgt, drf, None, seed=1234567890123, offset=100)
    assert not np.array_equal(a[0], c[0])


def test_given_draft_token_and_temperature(ssd):
    rng = np.random.default_rng(8)
    rows, V = 64, 8192
    tgt, drf = synth._logits_normal(rng, rows, V)
    dt = rng.integers(0, V, rows).astype(np.int64)
    u = synth.philox_uniforms(5, 0, rows)
    for T in (1.0, 0.7):
        tok, acc, ratio, lse, st = run_accept(ssd, tgt, drf, u, draft_tok=dt, T=T)
        assert st == 0
        dec = oacc.accept_rows(tgt, drf, u, draft_tok=dt, temperature=T)
        compare_decisions(dec, tok, acc, ratio, lse, what=f"T={T}")


def test_identical_distributions_all_accepted(ssd):
    rng = np.random.default_rng(9)
    rows, V = 64, 16384
    l = (rng.standard_normal((rows, V)) * 2).astype(np.float32)
    u = synth.philox_uniforms(3, 0, rows)
    u[:, 0] = 1 - 2**-24
    tok, acc, ratio, _, st = run_accept(ssd, l, l.copy(), u)
    assert st == 0 and acc.all()
    assert np.array_equal(tok, np.argmax(l, 1))
    assert np.all(ratio == 1.0)


def test_resampled_tokens_are_valid(ssd):
    rng = np.random.default_rng(10)
    rows, V = 256, 16384
    tgt, drf = synth._logits_normal(rng, rows, V)
    u = synth.philox_uniforms(4, 0, rows)
    tok, acc, _, _, st = run_accept(ssd, tgt, drf, u)
    p = np.exp(tgt - tgt.max(1, keepdims=True)); p /= p.sum(1, keepdims=True)
    q = np.exp(drf - drf.max(1, keepdims=True)); q /= q.sum(1, keepdims=True)
    rej = np.nonzero(acc == 0)[0]
    assert rej.size > 0
    t_hat = np.argmax(drf, 1)
    assert np.all(tok[rej] != t_hat[rej])
    assert np.all(p[rej, tok[rej]] > q[rej, tok[rej]])


def test_padded_leading_dimension(ssd):
    rng = np.random.default_rng(11)
    rows, V = 32, 4096
    tgt, drf = synth._logits_normal(rng, rows, V)
    u = synth.philox_uniforms(6, 0, rows)
    a = run_accept(ssd, tgt, drf, u, ld=V + 12)
    dec = oacc.accept_rows(tgt, drf, u)
    compare_decisions(dec, a[0], a[1], a[2], a[3], what="ld")


def test_out_of_range_draft_token_sets_status(ssd):
    rng = np.random.default_rng(12)
    tgt, drf = synth._logits_normal(rng, 4, 4096)
    dt = np.array([1, 4096, 3, -1])
    tok, acc, _, _, st = run_accept(ssd, tgt, drf, synth.philox_uniforms(0, 0, 4), draft_tok=dt)
    assert st == 6
    assert tok[1] == -1 and tok[3] == -1 and acc[1] == 0 and acc[3] == 0
    assert tok[0] >= 0 and tok[2] >= 0


# ---------------------------------------------------------------------------
# Strategies (A) greedy and (B) sampling of Sec. 3.3.

@pytest.mark.parametrize("strategy", ["greedy", "sample"])
@pytest.mark.parametrize("V,rows,logits,seed", [
    (16384, 48, "normal", 21),
    (16384, 40, "zipf", 22),
    (4100, 30, "normal", 23),     # ragged last chunk
    (12, 16, "normal", 24),       # tiny vocabulary
    (65536, 8, "zipf", 25),
])
def test_strategy_matches_oracle(ssd, strategy, V, rows, logits, seed):
    rng = np.random.default_rng(seed)
    if logits == "normal":
        tgt, drf = synth._logits_normal(rng, rows, V)
    else:
        tgt, drf = synth._logits_zipf(rng, rows, V)
    u = synth.philox_uniforms(seed, 3, rows)
    tok, acc, ratio, lse, st = run_accept(ssd, tgt, drf, u, strategy=strategy)
    assert st == 0
    dec = oacc.accept_rows(tgt, drf, u, strategy=strategy)
    ties = compare_decisions(dec, tok, acc, ratio, lse, what=f"{strategy} V={V}")
    if strategy == "greedy":
        assert ties == 0  # an argmax of raw fp32 logits has no rounding to excuse
    assert ties <= max_excused_rows(rows)  # also enforced inside compare_decisions


def test_greedy_ties_and_given_tokens(ssd):
    rng = np.random.default_rng(26)
    rows, V = 32, 8192
    tgt, drf = synth._logits_normal(rng, rows, V)
    for r in range(rows):  # the target maximum appears twice; the lower index wins
        i, j = sorted(rng.choice(V, 2, replace=False))
        tgt[r, [i, j]] = tgt[r].max() + 0.5
    dt = np.argmax(tgt, 1).astype(np.int64)
    dt[::2] = rng.integers(0, V, rows // 2)  # half the rows with another draft token
    u = synth.philox_uniforms(7, 0, rows)
    tok, acc, _, _, st = run_accept(ssd, tgt, drf, u, draft_tok=dt, strategy="greedy")
    assert st == 0
    assert np.array_equal(tok, np.argmax(tgt, 1))
    assert np.array_equal(acc.astype(bool), np.argmax(tgt, 1) == dt)


def test_sampling_with_given_tokens_and_temperature(ssd):
    rng = np.random.default_rng(27)
    rows, V = 64, 16384
    tgt, drf = synth._logits_normal(rng, rows, V)
    dt = rng.integers(0, V, rows).astype(np.int64)
    u = synth.philox_uniforms(8, 0, rows)
    tok, acc, ratio, _, st = run_accept(ssd, tgt, drf, u, draft_tok=dt, T=0.7, strategy="sample")
    assert st == 0
    dec = oacc.accept_rows(tgt, drf, u, draft_tok=dt, temperature=0.7, strategy="sample")
    compare_decisions(dec, tok, acc, ratio, what="sample T=0.7")


@pytest.mark.parametrize("strategy", ["accept_reject", "greedy"])
def test_masked_vocabulary_entries(ssd, strategy):
    """Degenerate distributions: a quarter of the vocabulary is masked (-inf)
    in the target and another quarter in the draft, and in every other row
    the draft's token is one the target masks (p(t) = 0: ratio 0, always
    rejected, the residual token drawn from the target's unmasked entries).
    Decisions, tokens and ratios against the oracle; no masked token is ever
    drawn."""
    rng = np.random.default_rng(9)
    rows, V = 32, 4096
    tgt, drf = synth._logits_normal(rng, rows, V)
    tgt, drf = tgt.astype(np.float32), drf.astype(np.float32)
    tgt[:, :1024] = -np.inf
    drf[:, 2048:3072] = -np.inf
    drf[::2, 5] = 50.0
    u = synth.philox_uniforms(9, 3, rows)
    tok, acc, ratio, lse, st = run_accept(ssd, tgt, drf, u, strategy=strategy)
    assert st == 0
    dec = oacc.accept_rows(tgt, drf, u, strategy=strategy)
    compare_decisions(dec, tok, acc, ratio, lse, what=f"masked {strategy}")
    assert not np.isin(tok, np.arange(1024)).any()
    if strategy == "accept_reject":
        assert not acc[::2].any() and np.all(ratio[::2] == 0.0)
