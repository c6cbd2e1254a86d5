"""Oracle: the fused lm_head followed by acceptance (float64).

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.3, after Eq. 2: tokens are decoded through the base model's GenHead,
a linear map from the (normalised) hidden state to vocabulary logits.  The
verification pass evaluates it for the target (backbone) and the draft
hidden states; strategy (C) then runs on the two logit rows.

reading: the hidden states arrive already normalised (the final RMSNorm is
part of the layers before this step); logits = H @ W with W stored
[hidden, V]; target and draft may use distinct weights.
"""
from __future__ import annotations

import numpy as np

from . import accept as acc


def logits(h: np.ndarray, w: np.ndarray) -> np.ndarray:
    """[rows, hidden] @ [hidden, V] in float64."""
    return np.asarray(h, dtype=np.float64) @ np.asarray(w, dtype=np.float64)


def lmhead_accept(h_tgt, h_drf, w_tgt, w_drf, uniforms, draft_tok=None, temperature=1.0):
    lp = logits(h_tgt, w_tgt)
    lq = logits(h_drf, w_drf)
    out = acc.accept_rows(lp, lq, uniforms, draft_tok, temperature)
    out["tgt_logits"] = lp
    out["drf_logits"] = lq
    return out
