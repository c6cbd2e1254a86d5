"""Oracle: one whole verification step and the single-round replay.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Chains the pieces in the order of Sec. 3.3: the frontier of each sequence,
the drafted block's attention over cache + block, strategy (C) on each
drafted position, then the accepted counts and the next cache length.
"""
from __future__ import annotations

import numpy as np

from . import accept as acc
from . import attention as att
from . import counts as cnt
from . import frontier as fr


def sequence_frontier(grid_h, grid_w, prefix_len, cache_len, k_v=1, k_h=0):
    coords = fr.frontier(grid_h, grid_w, prefix_len, int(cache_len), k_v, k_h)
    return coords, fr.grid_index(coords, grid_w)


def accept_step(grid_h, grid_w, prefix_len, k_v, cache_len, D_max, tgt_logits, drf_logits,
                uniforms, draft_tok=None, temperature=1.0, strategy="accept_reject", k_h=0,
                bonus=False):
    """Frontier + acceptance + counts for a batch (no attention).

    Row b*D_max + j of the logit / uniform arrays belongs to draft j of
    sequence b.  Returns per-sequence lists and the per-row decision dict
    restricted to valid rows (key "rows" lists their global row indices).
    With bonus (the horizontal stage), row b*D_max + n_d holds the backbone's
    logits at the position after the last draft: its token is the argmax
    under strategy (A) and otherwise the inverse-CDF draw from p with u_res
    (keys bonus_tok, bonus_tie, bonus_row); when every draft is accepted and
    that position exists it is committed too."""
    B = len(cache_len)
    n_d = np.zeros(B, np.int64)
    pos = np.full((B, D_max), -1, np.int64)
    rows = []
    for b in range(B):
        coords, g = sequence_frontier(grid_h, grid_w, prefix_len, cache_len[b], k_v, k_h)
        n_d[b] = len(coords)
        pos[b, :len(g)] = g
        rows += [b * D_max + j for j in range(len(g))]
    rows = np.array(rows, dtype=np.int64)
    if rows.size:
        dt = None if draft_tok is None else np.asarray(draft_tok)[rows]
        dec = acc.accept_rows(np.asarray(tgt_logits)[rows], np.asarray(drf_logits)[rows],
                              np.asarray(uniforms)[rows], dt, temperature, strategy)
    else:
        dec = {k: np.zeros(0) for k in ("out_tok", "accepted", "tie_accept", "tie_resample")}
    dec["rows"] = rows
    accepted_full = np.zeros(B * D_max, bool)
    accepted_full[rows] = dec["accepted"]
    counts = np.zeros(B, np.int64)
    prefix = np.zeros(B, np.int64)
    nxt = np.zeros(B, np.int64)
    bonus_tok = np.full(B, -1, np.int64)
    bonus_tie = np.zeros(B, bool)
    bonus_row = np.full(B, -1, np.int64)
    for b in range(B):
        exists = False
        if bonus and 0 < n_d[b] < D_max:
            row = b * D_max + int(n_d[b])
            bonus_row[b] = row
            lp = np.asarray(tgt_logits, dtype=np.float64)[row]
            if strategy == "greedy":
                bonus_tok[b] = int(np.argmax(lp))
            else:
                p, _ = acc.softmax(lp[None], temperature)
                bonus_tok[b], margin = acc.inverse_cdf(p[0], float(np.asarray(uniforms)[row, 1]))
                bonus_tie[b] = margin < acc.NEAR_TIE_CDF
            exists = int(cache_len[b]) - prefix_len + int(n_d[b]) < grid_h * grid_w
        counts[b], prefix[b], nxt[b] = cnt.step_counts_bonus(
            accepted_full[b * D_max:(b + 1) * D_max], int(n_d[b]), int(cache_len[b]), exists)
    return dict(n_drafts=n_d, draft_pos=pos, accepted_count=counts, accepted_prefix=prefix,
                next_cache_len=nxt, decisions=dec, bonus_tok=bonus_tok, bonus_tie=bonus_tie,
                bonus_row=bonus_row)


def attention_step(grid_h, grid_w, prefix_len, row_stride, k_v, cache_len, q, k, v, Hq, Hkv,
                   scale=None, seqs=None, k_h=0):
    """Frontier attention for the sequences in ``seqs`` (default: all).

    q [B, D_max, Hq, d], k/v [B, Hkv, L_max, d] (float).  Returns
    {b: (o [n_d, Hq, d], lse [Hq, n_d])}."""
    B = len(cache_len)
    res = {}
    for b in (range(B) if seqs is None else seqs):
        coords, _ = sequence_frontier(grid_h, grid_w, prefix_len, cache_len[b], k_v, k_h)
        n = len(coords)
        res[b] = att.verify_attention(q[b, :n], k[b], v[b], int(cache_len[b]), coords,
                                      prefix_len, row_stride, Hq, Hkv, scale)
    return res


def replay(grid_h, grid_w, prefix_len, k_v, B, D_max, step_inputs, max_steps=100000,
           temperature=1.0):
    """Single-round replay to grid completion.

    step_inputs(t) -> (tgt_logits, drf_logits, uniforms) for step t.
    Returns the per-step history: cache_len before the step, n_drafts,
    accepted_count, accepted_prefix, and the committed tokens per sequence.
    Stops when every sequence has an empty frontier."""
    cache_len = np.full(B, prefix_len, np.int64)
    grid_tok = np.full((B, grid_h * grid_w), -1, np.int64)
    hist = []
    for t in range(max_steps):
        lp, lq, u = step_inputs(t)
        r = accept_step(grid_h, grid_w, prefix_len, k_v, cache_len, D_max, lp, lq, u,
                        None, temperature)
        if int(r["n_drafts"].sum()) == 0:
            break
        dec = r["decisions"]
        tok_full = np.full(B * D_max, -1, np.int64)
        tok_full[dec["rows"]] = dec["out_tok"]
        for b in range(B):
            n_c = int(cache_len[b]) - prefix_len
            adv = int(r["next_cache_len"][b] - cache_len[b])
            grid_tok[b, n_c:n_c + adv] = tok_full[b * D_max:b * D_max + adv]
        hist.append(dict(cache_len=cache_len.copy(), n_drafts=r["n_drafts"].copy(),
                         accepted_count=r["accepted_count"].copy(),
                         accepted_prefix=r["accepted_prefix"].copy(),
                         next_cache_len=r["next_cache_len"].copy(),
                         accept_ties=int(np.sum(dec["tie_accept"])),
                         resample_ties=int(np.sum(dec["tie_resample"]))))
        cache_len = r["next_cache_len"].copy()
    return hist, grid_tok, cache_len
