"""Oracle pins for strategy (C) of Sec. 3.3: the accept/resample rule checked
against its closed-form output law by exhaustive enumeration of the
uniforms, the speculative-sampling marginal (output ~ p when t_hat ~ q), the
paper-implied special cases, and library softmax."""
import os

import numpy as np
import pytest
import scipy.special

from oracle import accept as acc

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
NQ = 2 ** 12  # uniforms enumerated on the midpoints of a 2^-12 grid


def closed_form_law(p, q, t_hat):
    """P(out = v | t_hat): alpha at t_hat plus (1 - alpha) times the residual law."""
    alpha = min(p[t_hat] / q[t_hat], 1.0)
    res = np.clip(p - q, 0, None)
    law = (1 - alpha) * res / res.sum() if res.sum() > 0 else np.zeros_like(p)
    law[t_hat] += alpha
    return law


def enumerate_law(lp, lq, t_hat):
    """Empirical output law of the oracle over the full 2^12 x 2^12 grid of
    (u_acc, u_res).  Acceptance only reads u_acc and resampling only u_res,
    so the grid factorises: P(v) = P_acc * [v == t] + (1 - P_acc) * P_res(v)."""
    grid = (np.arange(NQ) + 0.5) / NQ
    V = len(lp)
    rows = np.repeat(np.asarray(lp)[None], NQ, 0), np.repeat(np.asarray(lq)[None], NQ, 0)
    dt = np.full(NQ, t_hat)
    a = acc.accept_rows(rows[0], rows[1], np.stack([grid, np.zeros(NQ)], 1), dt)
    p_acc = a["accepted"].mean()
    r = acc.accept_rows(rows[0], rows[1], np.stack([np.full(NQ, 0.999999999), grid], 1), dt)
    assert not r["accepted"].any() or p_acc == 1.0
    p_res = np.bincount(r["out_tok"], minlength=V) / NQ
    law = (1 - p_acc) * p_res
    law[t_hat] += p_acc
    return law


def _random_logits(rng, V, scale=2.0):
    return rng.standard_normal(V) * scale, rng.standard_normal(V) * scale


def test_golden_worked_example():
    vals = {}
    for line in open(os.path.join(GOLDEN, "accept_worked_example.txt")):
        if line.startswith("#") or not line.strip():
            continue
        key, *nums = line.split()
        vals[key] = np.array([float(x) for x in nums])
    p, q = vals["p"], vals["q"]
    lp, lq = np.log(p), np.log(q)
    t = int(vals["t_hat"][0])
    assert int(acc.draft_token(lq[None])[0]) == t
    out = acc.accept_rows(lp[None], lq[None], np.array([[0.25, 0.5]]))
    assert np.isclose(out["alpha"][0], vals["alpha"][0], rtol=1e-12)
    assert np.allclose(enumerate_law(lp, lq, t), vals["out_law_t_hat"], atol=2.0 / NQ)
    marg = sum(q[s] * enumerate_law(lp, lq, s) for s in range(3))
    assert np.allclose(marg, vals["marginal_t_hat_from_q"], atol=2.0 / NQ)


@pytest.mark.parametrize("V,seed", [(2, 0), (3, 1), (5, 2), (8, 3), (8, 4)])
def test_enumeration_matches_closed_form(V, seed):
    rng = np.random.default_rng(seed)
    lp, lq = _random_logits(rng, V)
    p, q = scipy.special.softmax(lp), scipy.special.softmax(lq)
    for t in range(V):
        assert np.allclose(enumerate_law(lp, lq, t), closed_form_law(p, q, t), atol=2.0 / NQ)


@pytest.mark.parametrize("V,seed", [(4, 5), (8, 6)])
def test_marginal_is_target_when_draft_from_q(V, seed):
    """Speculative sampling (Leviathan et al., cited in Sec. 1-2): with
    t_hat ~ q the accept/resample output is distributed exactly as p."""
    rng = np.random.default_rng(seed)
    lp, lq = _random_logits(rng, V)
    p, q = scipy.special.softmax(lp), scipy.special.softmax(lq)
    marg = sum(q[t] * enumerate_law(lp, lq, t) for t in range(V))
    assert np.allclose(marg, p, atol=2.0 / NQ)


def test_identical_distributions_accept_everything():
    rng = np.random.default_rng(7)
    l = rng.standard_normal((300, 1000)) * 2
    u = rng.random((300, 2))
    u[:, 0] = np.maximum(u[:, 0], 1 - 2**-24)  # even the largest uniform
    out = acc.accept_rows(l, l.copy(), u)
    assert out["accepted"].all()
    assert np.array_equal(out["out_tok"], np.argmax(l, 1))
    assert np.allclose(out["ratio"], 1.0, rtol=0, atol=0)


def test_target_at_least_draft_is_always_accepted():
    rng = np.random.default_rng(8)
    V = 64
    for _ in range(50):
        lp, lq = _random_logits(rng, V)
        t = int(np.argmax(lq))
        lp[t] = lq[t] + 3.0  # p(t) >= q(t) after normalisation is not implied; check alpha
        p, q = scipy.special.softmax(lp), scipy.special.softmax(lq)
        out = acc.accept_rows(np.repeat(lp[None], 20, 0), np.repeat(lq[None], 20, 0),
                              np.stack([np.linspace(0, 1 - 2**-24, 20), np.zeros(20)], 1))
        if p[t] >= q[t]:
            assert out["accepted"].all()
        else:
            assert out["accepted"].mean() < 1


def test_resampled_token_properties():
    rng = np.random.default_rng(9)
    lp = rng.standard_normal((400, 257)) * 2
    lq = rng.standard_normal((400, 257)) * 2
    u = rng.random((400, 2))
    out = acc.accept_rows(lp, lq, u)
    p, q = scipy.special.softmax(lp, 1), scipy.special.softmax(lq, 1)
    rej = ~out["accepted"]
    assert rej.sum() > 100
    for r in np.nonzero(rej)[0]:
        v = out["out_tok"][r]
        assert v != out["t_hat"][r]
        assert p[r, v] > q[r, v]


def test_softmax_matches_library_and_sums_to_one():
    rng = np.random.default_rng(10)
    l = rng.standard_normal((20, 4096)) * 2
    for T in (1.0, 0.7, 2.5):
        p, lse = acc.softmax(l, T)
        assert np.allclose(p, scipy.special.softmax(l / T, axis=1), rtol=1e-12, atol=0)
        assert np.allclose(lse, scipy.special.logsumexp(l / T, axis=1), rtol=1e-14)
        assert np.allclose(p.sum(1), 1.0, atol=1e-12)


def test_argmax_ties_lowest_index():
    l = np.zeros((1, 10))
    l[0, [3, 7]] = 5.0
    assert acc.draft_token(l)[0] == 3


def test_temperature_equals_prescaled_logits():
    rng = np.random.default_rng(11)
    lp = rng.standard_normal((50, 300)) * 2
    lq = rng.standard_normal((50, 300)) * 2
    u = rng.random((50, 2))
    a = acc.accept_rows(lp, lq, u, temperature=0.5)
    b = acc.accept_rows(lp / 0.5, lq / 0.5, u, temperature=1.0)
    assert np.array_equal(a["out_tok"], b["out_tok"])
    assert np.array_equal(a["accepted"], b["accepted"])


def test_given_draft_token_is_used():
    rng = np.random.default_rng(12)
    lp = rng.standard_normal((30, 50))
    lq = rng.standard_normal((30, 50))
    t = rng.integers(0, 50, 30)
    out = acc.accept_rows(lp, lq, rng.random((30, 2)), draft_tok=t)
    assert np.array_equal(out["t_hat"], t)
    assert np.array_equal(out["out_tok"][out["accepted"]], t[out["accepted"]])


def test_monte_carlo_marginal_chi2():
    """Monte-Carlo check of the marginal with random uniforms: t_hat ~ q."""
    rng = np.random.default_rng(13)
    V, N = 6, 60000
    lp, lq = _random_logits(rng, V, 1.0)
    p, q = scipy.special.softmax(lp), scipy.special.softmax(lq)
    t = rng.choice(V, size=N, p=q)
    out = acc.accept_rows(np.repeat(lp[None], N, 0), np.repeat(lq[None], N, 0),
                          rng.random((N, 2)), draft_tok=t)
    counts = np.bincount(out["out_tok"], minlength=V)
    chi2 = ((counts - N * p) ** 2 / (N * p)).sum()
    assert chi2 < 25.0  # 5 degrees of freedom; p-value ~1e-4


# ---------------------------------------------------------------------------
# Strategies (A) greedy and (B) sampling of Sec. 3.3.

@pytest.mark.parametrize("seed", [0, 1, 2])
def test_greedy_is_the_library_argmax_of_the_target(seed):
    rng = np.random.default_rng(seed)
    rows, V = 64, 300
    lp = rng.standard_normal((rows, V))
    lq = rng.standard_normal((rows, V))
    # planted ties of the target maximum: the lower index must win
    lp[0, [7, 200]] = lp[0].max() + 1.0
    lp[1, [0, 299]] = lp[1].max() + 1.0
    u = rng.random((rows, 2))
    d = acc.accept_rows(lp, lq, u, strategy="greedy")
    assert np.array_equal(d["out_tok"], np.argmax(lp, axis=1))
    assert d["out_tok"][0] == 7 and d["out_tok"][1] == 0
    assert np.array_equal(d["accepted"], np.argmax(lp, 1) == np.argmax(lq, 1))
    # the uniforms and the draft distribution do not move the greedy token
    d2 = acc.accept_rows(lp, lq[::-1], 1.0 - u, strategy="greedy")
    assert np.array_equal(d2["out_tok"], d["out_tok"])


@pytest.mark.parametrize("seed", [0, 1])
def test_sampling_is_the_library_inverse_cdf_of_p_with_u_res(seed):
    rng = np.random.default_rng(seed)
    rows, V = 200, 97
    lp = rng.standard_normal((rows, V)) * 2
    lq = rng.standard_normal((rows, V)) * 2
    u = np.stack([rng.random(rows), rng.random(rows)], 1)  # u_acc differs from u_res
    d = acc.accept_rows(lp, lq, u, strategy="sample")
    p = scipy.special.softmax(lp, axis=1)
    c = np.cumsum(p, axis=1)
    ref = np.array([np.searchsorted(c[r], u[r, 1] * c[r, -1], side="right") for r in range(rows)])
    ok = ~d["tie_resample"]
    assert ok.sum() > rows * 0.95
    assert np.array_equal(d["out_tok"][ok], ref[ok])
    assert np.array_equal(d["accepted"], d["out_tok"] == np.argmax(lq, 1))


def test_sampling_law_on_a_stratified_grid_of_uniforms():
    """N midpoint uniforms through an inverse CDF give each token a count
    within one of N * p (the grid points falling in an interval of length p)."""
    rng = np.random.default_rng(5)
    V, N = 11, 4096
    lp = rng.standard_normal(V) * 1.5
    lq = rng.standard_normal(V)
    grid = (np.arange(N) + 0.5) / N
    u = np.stack([np.zeros(N), grid], 1)
    d = acc.accept_rows(np.repeat(lp[None], N, 0), np.repeat(lq[None], N, 0), u,
                        strategy="sample")
    counts = np.bincount(d["out_tok"], minlength=V)
    p = scipy.special.softmax(lp)
    assert np.all(np.abs(counts - N * p) <= 1.0 + 1e-9)


def test_strategies_share_ratio_and_lse():
    rng = np.random.default_rng(8)
    lp, lq = rng.standard_normal((16, 50)), rng.standard_normal((16, 50))
    u = rng.random((16, 2))
    base = acc.accept_rows(lp, lq, u)
    for s in ("greedy", "sample"):
        d = acc.accept_rows(lp, lq, u, strategy=s)
        assert np.allclose(d["ratio"], base["ratio"]) and np.allclose(d["lse_p"], base["lse_p"])
    with pytest.raises(ValueError):
        acc.accept_rows(lp, lq, u, strategy="top_k")
