"""Oracle: the spatial draft predictor f_phi of Eq. 2 and the draft tokens.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__``).

Sec. 3.3 "Draft Prediction in Latent Space", Eq. 2:
    h_hat = f(z),  z = [h ; e]  (hidden state and token embedding, 2d)
    f(z)  = W0 z + SwiGLU(RMSNorm(W0 z)),
    SwiGLU(x) = W2 (silu(W1 x) * W3 x),
    W0: d x 2d, W1, W3: m x d, W2: d x m, bias-free;
and the draft token t_hat = argmax_v GenHead(RMSNorm(h_hat))_v.
App. "Configuration": 134.2 M parameters per head, i.e. 2 d^2 + 3 d m with
d = 4096 and m = 2 d.

Readings (the paper gives the formula, not the numerics):
  * RMSNorm(x) = x / sqrt(mean(x^2) + eps) * gamma with a gain vector gamma
    per norm (gamma1 inside f, gamma2 before GenHead); eps is an input;
  * GenHead is a [d, V] matrix (the base model's output layer);
  * RMSNorm(x) g = s(x) * (x * g) with the row scale s(x) = 1 / sqrt(mean(x^2)
    + eps); s(x) is a scalar per row, so s(x) W (x * g) = W RMSNorm(x) g
    exactly, and GenHead's argmax does not depend on a positive row scale;
  * precision follows the GPU path's data flow, so that both sides take the
    argmax on the same numbers: the inputs of every matrix product are bf16
    (z, the weights, A * g1, the SwiGLU gate, h_hat * g2), the row scale is
    applied to the product's output; W0 z, h_hat and the logits are kept at
    full precision (fp32 on the GPU, float64 here); the argmax takes the
    lowest index on ties.  Without the rounding (round_like_gpu=False) the
    function is Eq. 2 as written.
"""
from __future__ import annotations

import numpy as np

from synth import bf16_bits_to_f32, f32_to_bf16_bits  # bf16 storage rounding only


def param_count(d: int, m: int) -> int:
    """Weights of one predictor: W0 (d x 2d) + W1, W3 (m x d) + W2 (d x m)."""
    return d * 2 * d + 3 * m * d


def _bf(x):
    """Round to bf16 as the GPU stores a GEMM input (fp32 value, nearest-even)."""
    return bf16_bits_to_f32(f32_to_bf16_bits(np.asarray(x, dtype=np.float32))).astype(np.float64)


def rmsnorm(x, gamma, eps):
    x = np.asarray(x, dtype=np.float64)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * np.asarray(gamma, np.float64)


def row_scale(x, eps):
    """s(x) = 1 / sqrt(mean(x^2) + eps) per row, as a column [rows, 1]."""
    x = np.asarray(x, dtype=np.float64)
    return 1.0 / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps)


def silu(x):
    return x / (1.0 + np.exp(-x))


def predict(z, W0, W1, W2, W3, gamma1, gamma2, W_head, eps=1e-6, round_like_gpu=True):
    """Eq. 2 for rows of z [rows, 2d].  Weights as [out, in] matrices (bf16
    values given as float arrays), W_head [d, V].  Returns (h_hat [rows, d],
    logits [rows, V], tokens [rows])."""
    r = _bf if round_like_gpu else (lambda x: np.asarray(x, dtype=np.float64))
    g1 = np.asarray(gamma1, dtype=np.float64)
    g2 = np.asarray(gamma2, dtype=np.float64)
    z = r(z)
    A = z @ r(W0).T                                  # W0 z
    Ag = r(A * g1)                                   # A * g1, a GEMM input
    s1 = row_scale(A, eps)                           # RMSNorm(A) g1 = s1 * Ag
    U = s1 * (Ag @ r(W1).T)
    Vg = s1 * (Ag @ r(W3).T)
    G = r(silu(U) * Vg)                              # the SwiGLU gate, a GEMM input
    h_hat = A + G @ r(W2).T                          # residual
    Hg = r(h_hat * g2)                               # h_hat * g2, GenHead's input
    logits = row_scale(h_hat, eps) * (Hg @ r(W_head))  # GenHead(RMSNorm(h_hat) g2)
    return h_hat, logits, np.argmax(logits, axis=1).astype(np.int64)


def top2_gap(logits):
    """Per row: (largest - second largest logit); a small gap is an argmax near-tie."""
    s = np.sort(np.asarray(logits, dtype=np.float64), axis=1)
    return s[:, -1] - s[:, -2]
