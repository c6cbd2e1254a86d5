"""Oracle: target/draft softmax, acceptance and residual resampling (float64).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.3 "Verification as Auto Correction" names three ways to select the
final token of every drafted position, applied independently per position:
  (A) greedy selection: argmax_v p_k(v);
  (B) sampling: a draw from p_k;
  (C) acceptance-rejection sampling (the default), below.
Strategy (C):
  * q_k is the draft distribution, p_k the backbone's distribution;
  * the draft token is t_hat = argmax_v q_k(v);
  * t_hat is accepted with probability alpha = min(p_k(t_hat) / q_k(t_hat), 1);
  * on rejection the token is drawn from the residual distribution
    [p_k - q_k]_+ / sum_v' [p_k - q_k]_+.
Sec. 4 / App. "Configuration": temperature 1.0.

Readings (the paper states the distributions, not the mechanism):
  * p = softmax(l_p / T), q = softmax(l_q / T);
  * argmax ties go to the lowest vocabulary index; the argmax is taken on the
    raw logits (T > 0 keeps the order);
  * the ratio is evaluated in log space; if q(t_hat) is 0 the draft is
    accepted;
  * accept iff u_acc < alpha with u_acc uniform on [0, 1) (probability alpha);
  * the residual draw is the inverse CDF in ascending vocabulary order with
    one uniform u_res: the smallest v with sum_{v' <= v} w_v' > u_res * Z,
    w = [p - q]_+, Z = sum w; if rounding runs past the end the last v with
    w_v > 0 is taken; if Z == 0 the draw is made from p instead;
  * (A) takes the argmax of the raw target logits, lowest index on ties;
  * (B) draws from p by the same inverse CDF with u_res;
  * under (A) and (B) a position counts as accepted when the selected token
    equals the draft token t_hat (so the commit rule of one round is the
    same prefix rule for all three strategies).
"""
from __future__ import annotations

import numpy as np

STRATEGIES = ("accept_reject", "greedy", "sample")  # (C), (A), (B) of Sec. 3.3
NEAR_TIE = 1e-4      # |alpha - u_acc| below this: the accept decision is a near-tie
NEAR_TIE_CDF = 1e-6  # u_res * Z within this fraction of Z of a CDF boundary: resample near-tie


def softmax(logits: np.ndarray, temperature: float = 1.0):
    """Row softmax in float64.  Returns (probabilities, log-sum-exp of l/T)."""
    x = np.asarray(logits, dtype=np.float64) / float(temperature)
    m = x.max(axis=-1, keepdims=True)
    e = np.exp(x - m)
    s = e.sum(axis=-1, keepdims=True)
    return e / s, (m + np.log(s))[..., 0]


def draft_token(drf_logits: np.ndarray) -> np.ndarray:
    """argmax_v q(v) per row, lowest index on ties (np.argmax returns the first)."""
    return np.argmax(np.asarray(drf_logits), axis=-1).astype(np.int64)


def inverse_cdf(w: np.ndarray, u: float):
    """Smallest index v with cumsum(w)[v] > u * sum(w); see module readings.

    Returns (v, margin) where margin = distance of u*Z to the nearest CDF
    boundary of the chosen bin, relative to Z (for the near-tie report)."""
    c = np.cumsum(w)
    Z = c[-1]
    target = u * Z
    idx = np.nonzero(c > target)[0]
    if idx.size:
        v = int(idx[0])
    else:
        v = int(np.nonzero(w > 0)[0][-1])
    lo = c[v - 1] if v > 0 else 0.0
    margin = min(abs(target - lo), abs(c[v] - target)) / Z
    return v, margin


def accept_rows(tgt_logits, drf_logits, uniforms, draft_tok=None, temperature=1.0,
                strategy="accept_reject"):
    """One of the strategies of Sec. 3.3 on every row (default (C)).

    tgt_logits, drf_logits: [rows, V]; uniforms: [rows, 2] = (u_acc, u_res);
    draft_tok: [rows] or None (then t_hat = argmax q).
    Returns a dict of per-row arrays: out_tok, accepted, t_hat, ratio, alpha,
    lse_p, lse_q, resampled_from_p (Z == 0 fallback), accept_margin = |alpha -
    u_acc|, tie_accept (accept_margin < NEAR_TIE), cdf_margin (distance of
    u_res * Z to the nearest boundary of the chosen bin, over Z), tie_resample
    (cdf_margin < NEAR_TIE_CDF).  Under "greedy" out_tok is the argmax of the
    target logits; under "sample" it is the inverse-CDF draw from p with
    u_res; under both, accepted = (out_tok == t_hat) and tie_accept is False.
    """
    if strategy not in STRATEGIES:
        raise ValueError(f"unknown strategy {strategy!r}")
    lp = np.asarray(tgt_logits, dtype=np.float64)
    lq = np.asarray(drf_logits, dtype=np.float64)
    u = np.asarray(uniforms, dtype=np.float64)
    rows = lp.shape[0]
    p, lse_p = softmax(lp, temperature)
    q, lse_q = softmax(lq, temperature)
    t = draft_token(lq) if draft_tok is None else np.asarray(draft_tok, dtype=np.int64)
    out = dict(out_tok=np.zeros(rows, np.int64), accepted=np.zeros(rows, bool),
               t_hat=t.copy(), ratio=np.zeros(rows), alpha=np.zeros(rows),
               lse_p=lse_p, lse_q=lse_q, resampled_from_p=np.zeros(rows, bool),
               tie_accept=np.zeros(rows, bool), tie_resample=np.zeros(rows, bool),
               accept_margin=np.zeros(rows), cdf_margin=np.full(rows, np.inf))
    for r in range(rows):
        tr = int(t[r])
        log_ratio = (lp[r, tr] / temperature - lse_p[r]) - (lq[r, tr] / temperature - lse_q[r])
        ratio = np.exp(log_ratio)
        alpha = min(ratio, 1.0)
        out["ratio"][r] = ratio
        out["alpha"][r] = alpha
        if strategy == "greedy":
            v = int(np.argmax(lp[r]))
            out["out_tok"][r] = v
            out["accepted"][r] = v == tr
            continue
        if strategy == "sample":
            v, margin = inverse_cdf(p[r], u[r, 1])
            out["out_tok"][r] = v
            out["accepted"][r] = v == tr
            out["cdf_margin"][r] = margin
            out["tie_resample"][r] = margin < NEAR_TIE_CDF
            continue
        out["accept_margin"][r] = abs(alpha - u[r, 0])
        out["tie_accept"][r] = abs(alpha - u[r, 0]) < NEAR_TIE
        if u[r, 0] < alpha:
            out["accepted"][r] = True
            out["out_tok"][r] = tr
            continue
        w = np.maximum(p[r] - q[r], 0.0)
        if w.sum() > 0.0:
            v, margin = inverse_cdf(w, u[r, 1])
        else:
            v, margin = inverse_cdf(p[r], u[r, 1])
            out["resampled_from_p"][r] = True
        out["out_tok"][r] = v
        out["cdf_margin"][r] = margin
        out["tie_resample"][r] = margin < NEAR_TIE_CDF
    return out

