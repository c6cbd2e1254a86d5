"""Oracle: r verify-and-correct rounds, the staged schedule and the commit.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.3 "Verification as Auto Correction" (the vertical stage):
  * every drafted position is verified in every round, independently and in
    parallel, by strategy (C) (or (A)/(B));
  * after a round, a rejected position is replaced by a sample of its residual
    distribution and the backbone distribution of that round becomes its
    reference distribution for the next round; an accepted position keeps
    its token and its reference;
  * the procedure is repeated for a fixed number of rounds r; after the last
    round one more forward pass commits the corrected block.
Sec. 4 / App. (multi-row drafting, Lumina-mGPT with k_v = 2, "b = 5, i = 4"):
  staged verification runs b base rounds on both drafted rows, commits the
  first row, then runs i incremental rounds on the trailing row with the
  corrected first row as context, then commits it.

Readings (the paper gives the procedure in words only):
  * round 1 verifies the draft tokens t_hat (argmax q unless given) against
    the draft distribution q; round rho >= 2 verifies the tokens round
    rho - 1 left, against each position's current reference;
  * each round draws its own uniforms (the GPU path uses Philox offset =
    round index); here they are given per round;
  * the per-round target logits are inputs (the backbone that produces them
    is out of scope); the reference of a position is the draft logits until
    its first rejection, then the target logits of the round that last
    rejected it;
  * the commit after the last round keeps every drafted position of the
    block (no prefix rollback): next cache length = cache + n_d; a round
    that is not the last commits nothing; the staged schedule's first commit
    keeps the frontier's first row: next = cache + (W - x0) where x0 is the
    column the frontier starts at;
  * in the staged schedule the trailing row enters round b + 1 with the
    tokens and references round b left it.
"""
from __future__ import annotations

import numpy as np

from . import accept as acc

COMMIT_MODES = ("prefix", "none", "block", "first_row")


def _reference_rows(drf_logits, tgt_rounds, ref):
    """Logit row of each position's reference: 0 -> draft, k -> target of round k."""
    out = np.array(drf_logits, dtype=np.float64, copy=True)
    for k in range(1, len(tgt_rounds) + 1):
        sel = ref == k
        if sel.any():
            out[sel] = np.asarray(tgt_rounds[k - 1], dtype=np.float64)[sel]
    return out


def verify_rounds(tgt_rounds, drf_logits, uniforms_rounds, draft_tok=None, temperature=1.0,
                  strategy="accept_reject", tokens=None, ref=None):
    """r rounds on every row.

    tgt_rounds: r arrays [rows, V] (the backbone's logits of each round);
    drf_logits: [rows, V]; uniforms_rounds: [r, rows, 2] (u_acc, u_res).
    tokens / ref: the state to start from (default: the draft tokens and the
    draft distribution); ref[k] = 0 for the draft logits, rho for round rho.
    Returns a dict: tokens [r + 1, rows] (tokens[0] the input), ref [r + 1,
    rows] (the reference each round used is ref[rho]), accepted [r, rows],
    ratio [r, rows], tie [r, rows] (near-tie of the accept or of the draw).
    """
    r = len(tgt_rounds)
    lq = np.asarray(drf_logits, dtype=np.float64)
    rows = lq.shape[0]
    tok = (acc.draft_token(lq) if draft_tok is None else np.asarray(draft_tok, np.int64)) \
        if tokens is None else np.asarray(tokens, np.int64)
    ref = np.zeros(rows, np.int64) if ref is None else np.asarray(ref, np.int64).copy()
    out = dict(tokens=[tok.copy()], ref=[ref.copy()], accepted=[], ratio=[], tie=[])
    for rho in range(r):
        ref_logits = _reference_rows(lq, tgt_rounds, ref)
        d = acc.accept_rows(tgt_rounds[rho], ref_logits, uniforms_rounds[rho], draft_tok=tok,
                            temperature=temperature, strategy=strategy)
        rejected = ~d["accepted"]
        ref = np.where(rejected, rho + 1, ref)
        tok = d["out_tok"].astype(np.int64)
        out["tokens"].append(tok.copy())
        out["ref"].append(ref.copy())
        out["accepted"].append(d["accepted"].copy())
        out["ratio"].append(d["ratio"].copy())
        out["tie"].append(d["tie_accept"] | d["tie_resample"])
    for k in ("tokens", "ref", "accepted", "ratio", "tie"):
        out[k] = np.array(out[k])
    return out


def verify_staged(b, i, W, tgt_rounds, drf_logits, uniforms_rounds, draft_tok=None,
                  temperature=1.0, strategy="accept_reject"):
    """The staged schedule on one 2-row block of W columns per sequence.

    Rows 0..W-1 of the arrays are the block's first row, W..2W-1 its trailing
    row.  Rounds 1..b verify all 2W positions; rounds b+1..b+i verify the
    trailing row only (tgt_rounds[b:] and uniforms_rounds[b:] are read at
    rows W..2W-1).  Returns (first-row tokens after round b, trailing-row
    tokens after round b + i, the per-round dicts of both stages)."""
    lq = np.asarray(drf_logits, dtype=np.float64)
    assert lq.shape[0] == 2 * W and len(tgt_rounds) == b + i
    base = verify_rounds(tgt_rounds[:b], lq, uniforms_rounds[:b], draft_tok, temperature,
                         strategy)
    first = base["tokens"][-1][:W]
    tail = slice(W, 2 * W)
    # the trailing row keeps its tokens and its references (which keep
    # pointing at the rounds that set them) into the incremental rounds
    tgt_tail = [np.asarray(t, dtype=np.float64)[tail] for t in tgt_rounds]
    inc = _incremental(tgt_tail, lq[tail], uniforms_rounds, b, i, W, base["tokens"][-1][tail],
                       base["ref"][-1][tail], temperature, strategy)
    return first, inc["tokens"][-1], base, inc


def _incremental(tgt_tail, lq_tail, uniforms_rounds, b, i, W, tok, ref, temperature, strategy):
    """Rounds b+1..b+i on the trailing row: round numbers continue from b so
    that a reference set in round rho < b keeps pointing at that round."""
    out = dict(tokens=[np.asarray(tok, np.int64).copy()], ref=[ref.copy()], accepted=[], ratio=[],
               tie=[])
    ref = ref.copy()
    tok = np.asarray(tok, np.int64).copy()
    for rho in range(b, b + i):
        ref_logits = _reference_rows(lq_tail, tgt_tail, ref)
        d = acc.accept_rows(tgt_tail[rho], ref_logits, np.asarray(uniforms_rounds[rho])[W:2 * W],
                            draft_tok=tok, temperature=temperature, strategy=strategy)
        rejected = ~d["accepted"]
        ref = np.where(rejected, rho + 1, ref)
        tok = d["out_tok"].astype(np.int64)
        out["tokens"].append(tok.copy())
        out["ref"].append(ref.copy())
        out["accepted"].append(d["accepted"].copy())
        out["ratio"].append(d["ratio"].copy())
        out["tie"].append(d["tie_accept"] | d["tie_resample"])
    for k in ("tokens", "ref", "accepted", "ratio", "tie"):
        out[k] = np.array(out[k])
    return out


def commit_next(mode, accepted_row, n_d, first_row_len, cache_len):
    """Next cache length after a round under one of COMMIT_MODES (see readings)."""
    if mode == "prefix":
        from .counts import step_counts
        return step_counts(accepted_row, n_d, cache_len)[2]
    if mode == "none":
        return cache_len
    if mode == "block":
        return cache_len + n_d
    if mode == "first_row":
        return cache_len + min(first_row_len, n_d)
    raise ValueError(mode)
