"""Oracle pins for the r verify-and-correct rounds, the staged schedule and
the commit (Sec. 3.3; App. multi-row drafting): reductions to the single-round
rule, the reference-update invariant checked through closed forms, ratios
recomputed from library softmax, and the commit arithmetic."""
import numpy as np
import pytest
import scipy.special

from oracle import accept as acc
from oracle import rounds as rd


def _case(seed, r, rows=24, V=60, scale=2.0):
    rng = np.random.default_rng(seed)
    tg = [rng.standard_normal((rows, V)) * scale for _ in range(r)]
    dq = rng.standard_normal((rows, V)) * scale
    u = rng.random((r, rows, 2))
    return tg, dq, u


@pytest.mark.parametrize("seed", [0, 1])
def test_one_round_is_the_single_round_rule(seed):
    tg, dq, u = _case(seed, 1)
    o = rd.verify_rounds(tg, dq, u)
    d = acc.accept_rows(tg[0], dq, u[0])
    assert np.array_equal(o["tokens"][1], d["out_tok"])
    assert np.array_equal(o["accepted"][0], d["accepted"])
    assert np.array_equal(o["tokens"][0], np.argmax(dq, 1))
    assert np.array_equal(o["ref"][1], np.where(d["accepted"], 0, 1))


def test_targets_equal_to_the_draft_accept_everything():
    _, dq, u = _case(2, 4)
    o = rd.verify_rounds([dq.copy() for _ in range(4)], dq, u)
    assert o["accepted"].all()
    assert (o["tokens"] == np.argmax(dq, 1)[None]).all()
    assert (o["ref"] == 0).all()


@pytest.mark.parametrize("seed", [3, 4, 5])
def test_a_repeated_target_accepts_every_position_it_rejected(seed):
    """If round rho's backbone distribution equals round rho-1's, a position
    rejected in round rho-1 now has that very distribution as its reference:
    its ratio is exactly 1 and it is accepted with its resampled token."""
    tg, dq, u = _case(seed, 3)
    tg[1] = tg[0].copy()
    o = rd.verify_rounds(tg, dq, u)
    rej = ~o["accepted"][0]
    assert rej.sum() > 5
    assert np.allclose(o["ratio"][1][rej], 1.0, rtol=1e-12)
    assert o["accepted"][1][rej].all()
    assert np.array_equal(o["tokens"][2][rej], o["tokens"][1][rej])


@pytest.mark.parametrize("seed", [6, 7])
def test_ratios_recomputed_from_library_softmax(seed):
    tg, dq, u = _case(seed, 4)
    o = rd.verify_rounds(tg, dq, u)
    rows = dq.shape[0]
    for rho in range(4):
        p = scipy.special.softmax(tg[rho], axis=1)
        for k in range(rows):
            ref = o["ref"][rho][k]
            q = scipy.special.softmax(dq[k] if ref == 0 else tg[ref - 1][k])
            t = o["tokens"][rho][k]
            assert np.isclose(o["ratio"][rho][k], p[k, t] / q[t], rtol=1e-9)
        # the state after the round: rejected rows point at this round
        rej = ~o["accepted"][rho]
        assert np.all(o["ref"][rho + 1][rej] == rho + 1)
        assert np.all(o["ref"][rho + 1][~rej] == o["ref"][rho][~rej])
        assert np.all(o["tokens"][rho + 1][~rej] == o["tokens"][rho][~rej])


def test_staged_schedule_reductions():
    W, b, i = 6, 3, 2
    tg, dq, u = _case(8, b + i, rows=2 * W)
    first, trail, base, inc = rd.verify_staged(b, i, W, tg, dq, u)
    # the base stage is r = b rounds on the whole block
    o = rd.verify_rounds(tg[:b], dq, u[:b])
    assert np.array_equal(base["tokens"], o["tokens"])
    assert np.array_equal(first, o["tokens"][-1][:W])
    # i = 0: the trailing row keeps the tokens of round b
    f0, t0, _, _ = rd.verify_staged(b, 0, W, tg[:b], dq, u[:b])
    assert np.array_equal(t0, o["tokens"][-1][W:])
    assert inc["tokens"].shape == (i + 1, W)


def test_staged_references_cross_the_stage_boundary():
    """Round b + 1 repeats round b's target on the trailing row: every
    trailing position rejected in round b is accepted (ratio 1)."""
    W, b, i = 8, 2, 2
    tg, dq, u = _case(9, b + i, rows=2 * W)
    tg[b] = tg[b - 1].copy()
    first, trail, base, inc = rd.verify_staged(b, i, W, tg, dq, u)
    rej = ~base["accepted"][-1][W:]
    assert rej.sum() > 2
    assert np.allclose(inc["ratio"][0][rej], 1.0, rtol=1e-12)
    assert inc["accepted"][0][rej].all()


def test_commit_modes():
    acc_row = np.array([True, True, False, True, False])
    assert rd.commit_next("prefix", acc_row, 5, 3, 100) == 103
    assert rd.commit_next("none", acc_row, 5, 3, 100) == 100
    assert rd.commit_next("block", acc_row, 5, 3, 100) == 105
    assert rd.commit_next("first_row", acc_row, 5, 3, 100) == 103
    assert rd.commit_next("first_row", acc_row, 2, 3, 100) == 102
    assert rd.commit_next("block", acc_row, 0, 3, 100) == 100
    with pytest.raises(ValueError):
        rd.commit_next("rollback", acc_row, 5, 3, 100)
