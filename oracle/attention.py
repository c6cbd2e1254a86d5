"""Oracle: frontier attention in float64.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.3 "Verification as Auto Correction": the whole drafted block goes
through the frozen backbone in parallel.  Inside each attention layer every
draft query attends to the committed KV cache plus the drafted block's own
keys, under the spatial dependency mask of ``oracle.frontier`` (App.
"Deviation from AR": the context may still hold drafted tokens).

reading: scaled dot-product attention with scale 1/sqrt(d) unless given;
grouped-query attention maps query head h to KV head h // (Hq / Hkv)
(contiguous groups).  The paper names neither.
"""
from __future__ import annotations

import numpy as np

from . import frontier as fr


def attend_one(q: np.ndarray, k: np.ndarray, v: np.ndarray, visible: np.ndarray, scale: float):
    """softmax(scale * q k^T + mask) v for one query vector.

    q [d], k/v [L, d], visible bool [L].  Returns (o [d], lse) with
    lse = log sum_j exp(scale * q.k_j) over visible keys.
    """
    s = scale * (k[visible] @ q)
    m = s.max()
    w = np.exp(s - m)
    l = w.sum()
    o = (w @ v[visible]) / l
    return o, m + np.log(l)


def verify_attention(q, k, v, cache_len, draft_coords, prefix_len, row_stride, Hq, Hkv,
                     scale=None):
    """Attention of one sequence's drafts.

    q: float [n_d, Hq, d] (the drafts' queries, in frontier order)
    k, v: float [Hkv, >= cache_len + n_d, d]; slots [0, cache_len) are the
          committed cache, slots cache_len + j hold draft j's key/value.
    Returns (o float64 [n_d, Hq, d], lse float64 [Hq, n_d]).
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    n_d = len(draft_coords)
    d = q.shape[-1]
    if scale is None or scale == 0.0:
        scale = 1.0 / np.sqrt(d)
    L = cache_len + n_d
    mask = fr.coord_mask(draft_coords, cache_len, prefix_len, row_stride)
    group = Hq // Hkv
    o = np.zeros((n_d, Hq, d))
    lse = np.zeros((Hq, n_d))
    for h in range(Hq):
        g = h // group
        for j in range(n_d):
            o[j, h], lse[h, j] = attend_one(q[j, h], k[g, :L], v[g, :L], mask[j], scale)
    return o, lse
