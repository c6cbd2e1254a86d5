"""CPU oracle for the SSD verification pass — TEST INFRASTRUCTURE ONLY.

Plain, slow, float64 NumPy restatements of what one verification step of
Spatially Speculative Decoding (SSD) computes.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s CPU-baseline / reference arm
may import or run anything in this package.  The product (the CUDA library
and its Python binding) never does, and shares no code with it: no kernels,
no helpers, no tables or constants.  Inputs come from the seeded generators
in ``synth`` (random draws only) or from a test.

Modules and the passage each follows:
  frontier   Sec. 3.1 (Eq. 1, raster order), Sec. 3.3 (horizontal offsets,
             vertical offsets, column-wise independence, the SSD
             factorisation): which grid positions one step drafts, and the
             spatial dependency mask among them.
  attention  Sec. 3.3 "Verification as Auto Correction" and App. "Deviation
             from AR": the drafted block passes through the frozen backbone
             in parallel, each draft attending to its raster prefix (which may
             hold drafted tokens).
  accept     Sec. 3.3 "Verification as Auto Correction", strategy (C):
             softmax, acceptance with probability min(p/q, 1), residual
             resampling from [p - q]_+ / sum [p - q]_+.
  counts     Sec. 3.3 (verify rounds, commit) and Sec. 4 "SSD Configuration"
             (horizontal prefix acceptance): accepted counts and the next
             cache length of a single-round replay.
  lmhead     Sec. 3.3, Eq. 2's GenHead: logits = hidden @ W, then accept.
  predictor  Sec. 3.3 "Draft Prediction in Latent Space", Eq. 2: the spatial
             draft predictor f_phi and the draft token argmax GenHead(RMSNorm).
  rounds     Sec. 3.3 (r verify-and-correct rounds: rejected positions take
             the residual sample and this round's p as their reference; the
             commit after the last round) and App. multi-row drafting (the
             staged b / i schedule).
  step       the above chained in the order of Sec. 3.3, and the
             single-round replay to grid completion.

Readings where the paper is silent are marked "reading:" in each function
and collected in the design notes of the repository.
"""
from . import frontier, attention, accept, counts, lmhead, step  # noqa: F401
