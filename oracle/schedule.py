"""Oracle: the whole SSD decoding schedule of one image, replayed to grid
completion.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.3 (the SSD factorisation): the k_h horizontal heads draft along the
raster order until the current row is complete; then the vertical heads
draft up to k_v rows below it in parallel, and the drafted rows are verified
and corrected ("Verification as Auto Correction": r rounds, then one more
forward pass that commits the corrected block and updates the KV cache).
Sec. 4 "SSD Configuration": the horizontal stage drafts 5 tokens per step
with 1 verification round; Janus-Pro and Emu3 draft k_v = 1 row with r = 2
and r = 5 rounds, Lumina-mGPT k_v = 2 rows with staged verification, b = 5
base rounds on both rows, then i = 4 incremental rounds on the trailing row.
App. "Multi-Row Anticipation Ablations": staged verification runs b base
rounds on all drafted rows, commits the first row, then refines the trailing
row against the corrected context.

The paper's "Steps" count backbone forward passes.  Its configuration
sweeps (App. "Configuration Selection", Tables app_sel_janus / lumina /
emu3, and the schedule ablation) fit one rule for the vertical stage: a
group of k drafted rows costs b rounds plus a commit pass for its first row,
then i rounds plus a commit pass for each of its k - 1 trailing rows:
    steps(group) = (b + 1) + (k - 1) (i + 1),
over the n - 1 rows below the first in groups of k_v (the last group takes
the rows left), plus the horizontal stage's steps S_h on the first row.

Readings (the paper states the schedule in words and counts):
  * the horizontal stage covers the first grid row only; each step is one
    verification round with the prefix rule and the bonus token of
    ``oracle.counts.step_counts_bonus``, the bonus only while the position
    after the drafts is still in the first row (a later position belongs to
    the vertical stage);
  * r rounds for k_v = 1 are the staged schedule with b = r, i = 0;
  * a commit pass reads no logits and changes no token: it keeps the tokens
    the last round left (the first row of the block, or the whole block when
    it is the group's last row);
  * after a commit, the trailing rows keep their tokens and their reference
    distributions and form the next frontier;
  * every step t (round or commit pass) has its own inputs: the target logits
    and uniforms of step t; a block's draft logits are those of its group's
    first base round; references are kept as (step, slot) of the logits they
    point at.
"""
from __future__ import annotations

import numpy as np

from . import accept as acc
from . import counts as cnt
from . import frontier as fr


def group_steps(k, b, i):
    """Forward passes of one vertical group of k drafted rows."""
    return (b + 1) + (k - 1) * (i + 1)


def vertical_steps(n, k_v, b, i):
    """Forward passes of the vertical stage over the n - 1 rows below the
    first row, in groups of k_v rows (the last group takes what is left)."""
    rows, total = n - 1, 0
    while rows > 0:
        k = min(k_v, rows)
        total += group_steps(k, b, i)
        rows -= k
    return total


def _frontier(H, W, prefix, cache_len, k_v, k_h):
    coords = fr.frontier(H, W, prefix, int(cache_len), k_v, k_h)
    return len(coords)


def replay(H, W, prefix, k_h, k_v, b, i, D_max, step_inputs, temperature=1.0,
           max_steps=100000):
    """One image (batch 1) from an empty grid to completion.

    step_inputs(t) -> (tgt_logits [D_max + 1, V], drf_logits [D_max + 1, V],
    uniforms [D_max + 1, 2]) for step t; slot j of a step's arrays belongs to
    draft j of that step's frontier (slot n_d: the horizontal stage's bonus
    row).  Returns (steps, grid_tok, hist): hist has one entry per step with
    its kind ('horizontal', 'round', 'commit'), the cache length before it,
    its draft count, and for rounds and horizontal steps the accept flags,
    the tokens after it, the near-tie rows (tie_rows: accept or draw within
    the bands of ``oracle.accept``; bonus_tie for the bonus draw) and their
    count."""
    HW = H * W
    cache = prefix
    grid = np.full(HW, -1, np.int64)
    hist = []
    t = 0

    def record(kind, n_d, **kw):
        hist.append(dict(kind=kind, step=t, cache_len=cache, n_drafts=n_d, **kw))

    # ---- horizontal stage: the first row
    while cache - prefix < W and t < max_steps:
        n_d = _frontier(H, W, prefix, cache, 0, k_h)
        lp, lq, u = step_inputs(t)
        dec = acc.accept_rows(np.asarray(lp)[:n_d], np.asarray(lq)[:n_d], np.asarray(u)[:n_d],
                              None, temperature)
        n_c = cache - prefix
        exists = n_c + n_d < W  # the bonus stays in the first row
        p, _ = acc.softmax(np.asarray(lp, dtype=np.float64)[n_d][None], temperature)
        bonus, margin = acc.inverse_cdf(p[0], float(np.asarray(u)[n_d, 1]))
        _, prefix_len, nxt = cnt.step_counts_bonus(dec["accepted"], n_d, cache, exists)
        toks = np.array(dec["out_tok"], copy=True)
        adv = nxt - cache
        committed = list(toks[:min(adv, n_d)])
        if adv > n_d:
            committed.append(bonus)
        grid[n_c:n_c + adv] = committed
        tie = dec["tie_accept"] | dec["tie_resample"]
        record("horizontal", n_d, accepted=dec["accepted"].copy(), tokens=np.array(committed),
               tie_rows=tie.copy(), bonus_tie=bool(margin < acc.NEAR_TIE_CDF),
               ties=int(tie.sum() + (margin < acc.NEAR_TIE_CDF)))
        cache = nxt
        t += 1

    # ---- vertical stage: groups of k_v rows
    while cache - prefix < HW and t < max_steps:
        n_c = cache - prefix
        y0 = n_c // W
        k = min(k_v, H - y0)
        n_d = _frontier(H, W, prefix, cache, k - 1, 0)
        # the block: tokens, reference (step, slot) per draft slot
        _, lq0, _ = step_inputs(t)
        lq0 = np.asarray(lq0, dtype=np.float64)[:n_d]
        tok = acc.draft_token(lq0)
        ref = [("drf", t, j) for j in range(n_d)]
        offset = 0  # slot of the block's first remaining draft
        for stage in range(k):
            rounds = b if stage == 0 else i
            m = n_d - offset  # drafts still in the frontier
            for _ in range(rounds):
                lp, _, u = step_inputs(t)
                lp = np.asarray(lp, dtype=np.float64)[:m]
                refl = np.stack([np.asarray(step_inputs(s)[1 if kind == "drf" else 0],
                                            dtype=np.float64)[slot] for kind, s, slot in
                                 ref[offset:]])
                d = acc.accept_rows(lp, refl, np.asarray(u)[:m], tok[offset:], temperature)
                rej = ~d["accepted"]
                for j in np.nonzero(rej)[0]:
                    ref[offset + j] = ("tgt", t, j)
                tok[offset:] = d["out_tok"]
                tie = d["tie_accept"] | d["tie_resample"]
                record("round", m, accepted=d["accepted"].copy(), tokens=tok[offset:].copy(),
                       tie_rows=tie.copy(), ties=int(tie.sum()))
                t += 1
            # the commit pass: the frontier's first row, or what is left
            first = W - (cache - prefix) % W
            adv = first if stage < k - 1 else m
            grid[cache - prefix:cache - prefix + adv] = tok[offset:offset + adv]
            record("commit", m, committed=adv)
            cache += adv
            t += 1
            # the trailing rows become the next frontier (their slots move to
            # the front; tokens and references stay as the last round left them)
            offset += adv
    return t, grid, hist
