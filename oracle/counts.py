"""Oracle: accepted counts and the next cache length (integer only).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.3: after verification, accepted drafts are kept and rejected ones are
replaced by residual samples; the committed block extends the KV cache.
Sec. 4 "SSD Configuration": the horizontal stage uses one verification round
per step, i.e. the usual speculative prefix rule.

reading (single-round replay): a step commits its drafts in raster order up
to and including the first rejected one, which carries its resampled token
(the correction); if every draft is accepted the whole frontier is
committed.  next_cache_len = cache_len + min(accepted_prefix + 1, n_d), and
a sequence with no drafts (grid complete) stays where it is.
"""
from __future__ import annotations

import numpy as np


def step_counts(accepted_row: np.ndarray, n_d: int, cache_len: int):
    """accepted_row: bool [>= n_d] in frontier (raster) order.

    Returns (accepted_count, accepted_prefix, next_cache_len)."""
    a = np.asarray(accepted_row[:n_d], dtype=bool)
    count = int(a.sum())
    prefix = 0
    while prefix < n_d and a[prefix]:
        prefix += 1
    advance = min(prefix + 1, n_d) if n_d > 0 else 0
    return count, prefix, cache_len + advance


def step_counts_bonus(accepted_row: np.ndarray, n_d: int, cache_len: int, bonus_exists: bool):
    """The horizontal stage (Sec. 4 "SSD Configuration": k_h drafts, one
    verification round): the prefix rule, and when every draft is accepted
    the token at the next position, drawn from the backbone's distribution
    there, is committed as well (reading: only if that position exists)."""
    count, prefix, nxt = step_counts(accepted_row, n_d, cache_len)
    if n_d > 0 and prefix == n_d and bonus_exists:
        nxt = cache_len + n_d + 1
    return count, prefix, nxt
