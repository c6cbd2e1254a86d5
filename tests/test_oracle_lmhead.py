"""Oracle pins for the fused lm_head + acceptance (Sec. 3.3, GenHead after
Eq. 2: logits = hidden @ W with W stored [hidden, V], then strategy (C)).

Each pin is fixed by the mathematics, not by re-running the oracle's own
matrix product:
  * one-hot weight columns: column v of W selects hidden entry k(v), so the
    logits are those hidden entries (a transposed or mis-strided W, or the
    hidden states read as [hidden, rows], fails on the non-square shapes);
  * a rank-one weight W = a b^T gives logits (h . a) b^T;
  * a brute-force triple loop in plain Python on a tiny case;
  * identical target and draft (hidden states and weights) accept every row;
  * the decisions equal strategy (C) on the logits of the one-hot closed form,
    which a swap of the target and draft sides would break.
"""
import numpy as np

from oracle import accept as acc
from oracle import lmhead as olm

import synth


def _uniforms(rows, seed=0):
    return synth.philox_uniforms(seed, 0, rows)


def test_one_hot_columns_select_hidden_entries():
    rng = np.random.default_rng(0)
    rows, K, V = 5, 12, 20                      # non-square everywhere
    h = rng.standard_normal((rows, K))
    sel = rng.integers(0, K, size=V)            # column v picks hidden entry sel[v]
    W = np.zeros((K, V))
    W[sel, np.arange(V)] = 1.0
    assert np.array_equal(olm.logits(h, W), h[:, sel])
    # scaled one-hot: W[k, v] = c_v picks c_v * h[:, k]
    c = rng.standard_normal(V)
    W2 = np.zeros((K, V))
    W2[sel, np.arange(V)] = c
    assert np.allclose(olm.logits(h, W2), h[:, sel] * c[None], rtol=0, atol=1e-15)


def test_rank_one_weight_closed_form():
    rng = np.random.default_rng(1)
    rows, K, V = 3, 7, 11
    h = rng.standard_normal((rows, K))
    a, b = rng.standard_normal(K), rng.standard_normal(V)
    want = np.array([[sum(h[r, k] * a[k] for k in range(K)) * b[v] for v in range(V)]
                     for r in range(rows)])
    assert np.allclose(olm.logits(h, np.outer(a, b)), want, rtol=1e-12, atol=1e-12)


def test_brute_force_triple_loop():
    rng = np.random.default_rng(2)
    rows, K, V = 4, 6, 9
    h = rng.standard_normal((rows, K))
    W = rng.standard_normal((K, V))
    want = np.zeros((rows, V))
    for r in range(rows):
        for v in range(V):
            s = 0.0
            for k in range(K):
                s += h[r, k] * W[k, v]
            want[r, v] = s
    assert np.allclose(olm.logits(h, W), want, rtol=1e-13, atol=1e-13)


def test_identical_target_and_draft_accept_every_row():
    rng = np.random.default_rng(3)
    rows, K, V = 16, 24, 40
    h = rng.standard_normal((rows, K))
    W = rng.standard_normal((K, V)) * 0.3
    out = olm.lmhead_accept(h, h, W, W, _uniforms(rows))
    assert out["accepted"].all()
    assert np.allclose(out["ratio"], 1.0, rtol=0, atol=1e-12)
    assert np.array_equal(out["out_tok"], np.argmax(h @ W, axis=1))


def test_decisions_follow_the_one_hot_logits_and_are_side_sensitive():
    rng = np.random.default_rng(4)
    rows, K, V = 64, 10, 30
    ht = 2.0 * rng.standard_normal((rows, K))
    hd = 2.0 * rng.standard_normal((rows, K))
    st, sd = rng.integers(0, K, size=V), rng.integers(0, K, size=V)
    Wt = np.zeros((K, V))
    Wt[st, np.arange(V)] = 1.0
    Wd = np.zeros((K, V))
    Wd[sd, np.arange(V)] = 1.0
    u = _uniforms(rows, seed=9)
    out = olm.lmhead_accept(ht, hd, Wt, Wd, u)
    ref = acc.accept_rows(ht[:, st], hd[:, sd], u)
    assert np.array_equal(out["accepted"], ref["accepted"])
    assert np.array_equal(out["out_tok"], ref["out_tok"])
    assert np.allclose(out["ratio"], ref["ratio"], rtol=1e-12)
    # the target and draft sides are not interchangeable: swapping them changes
    # the draft token (argmax of the draft logits) and the ratio
    swapped = olm.lmhead_accept(hd, ht, Wd, Wt, u)
    assert not np.array_equal(swapped["t_hat"], out["t_hat"])
    assert not np.allclose(swapped["ratio"], out["ratio"])
