"""Oracle pins for the spatial draft predictor (Eq. 2) and its draft tokens:
the paper's parameter count, RMSNorm and SiLU against library routines, the
closed forms W2 = 0 and W0 = [I 0], and the whole predictor against an
independent torch float64 restatement (without the bf16 rounding the GPU
path implies, which it may differ from by bf16-level error only)."""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from oracle import predictor as pr


def test_parameter_count_matches_the_paper():
    # App. "Configuration": 134.2 M parameters per head at d = 4096, m = 2d
    assert round(pr.param_count(4096, 8192) / 1e6, 1) == 134.2


def _weights(seed, d=32, m=64, V=50):
    rng = np.random.default_rng(seed)
    W0 = rng.standard_normal((d, 2 * d)) / np.sqrt(2 * d)
    W1 = rng.standard_normal((m, d)) / np.sqrt(d)
    W3 = rng.standard_normal((m, d)) / np.sqrt(d)
    W2 = rng.standard_normal((d, m)) / np.sqrt(m)
    g1 = 1 + 0.1 * rng.standard_normal(d)
    g2 = 1 + 0.1 * rng.standard_normal(d)
    Wh = rng.standard_normal((d, V)) / np.sqrt(d)
    z = rng.standard_normal((12, 2 * d))
    return z, W0, W1, W2, W3, g1, g2, Wh


def test_rmsnorm_and_silu_match_torch():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((7, 40))
    g = rng.standard_normal(40)
    ref = F.rms_norm(torch.from_numpy(x), (40,), torch.from_numpy(g), eps=1e-6).numpy()
    assert np.allclose(pr.rmsnorm(x, g, 1e-6), ref, rtol=1e-12, atol=1e-12)
    assert np.allclose(pr.silu(x), F.silu(torch.from_numpy(x)).numpy(), rtol=1e-12, atol=1e-14)


def test_closed_forms():
    z, W0, W1, W2, W3, g1, g2, Wh = _weights(2)
    d = W0.shape[0]
    # W2 = 0: f(z) = W0 z
    h, _, _ = pr.predict(z, W0, W1, np.zeros_like(W2), W3, g1, g2, Wh, round_like_gpu=False)
    assert np.allclose(h, z @ W0.T, rtol=1e-12)
    # W0 = [I 0]: f(z) = h + SwiGLU(RMSNorm(h)) with h the first half of z
    I0 = np.concatenate([np.eye(d), np.zeros((d, d))], axis=1)
    h2, _, _ = pr.predict(z, I0, W1, W2, W3, g1, g2, Wh, round_like_gpu=False)
    hz = z[:, :d]
    n = hz / np.sqrt(np.mean(hz ** 2, 1, keepdims=True) + 1e-6) * g1
    sw = (F.silu(torch.from_numpy(n @ W1.T)).numpy() * (n @ W3.T)) @ W2.T
    assert np.allclose(h2, hz + sw, rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("seed", [3, 4])
def test_against_a_torch_restatement(seed):
    z, W0, W1, W2, W3, g1, g2, Wh = _weights(seed)
    t = {k: torch.from_numpy(v) for k, v in dict(z=z, W0=W0, W1=W1, W2=W2, W3=W3, g1=g1,
                                                  g2=g2, Wh=Wh).items()}
    lin = F.linear
    a = lin(t["z"], t["W0"])
    n = F.rms_norm(a, (a.shape[-1],), t["g1"], eps=1e-6)
    h = a + lin(F.silu(lin(n, t["W1"])) * lin(n, t["W3"]), t["W2"])
    logits = F.rms_norm(h, (h.shape[-1],), t["g2"], eps=1e-6) @ t["Wh"]
    h_o, l_o, tok = pr.predict(z, W0, W1, W2, W3, g1, g2, Wh, round_like_gpu=False)
    assert np.allclose(h_o, h.numpy(), rtol=1e-10, atol=1e-12)
    assert np.allclose(l_o, logits.numpy(), rtol=1e-10, atol=1e-12)  # the row scales included
    assert np.array_equal(tok, torch.argmax(logits, 1).numpy())
    # with the GPU's bf16 rounding points the result moves by bf16-level error only
    h_b, l_b, _ = pr.predict(z, W0, W1, W2, W3, g1, g2, Wh)
    assert np.abs(h_b - h_o).max() / np.abs(h_o).max() < 3e-2
    assert np.array_equal(np.argmax(l_o, 1), tok)


def test_argmax_ties_and_gap():
    l = np.array([[1.0, 3.0, 3.0, 0.0], [2.0, 1.0, 0.5, 1.9]])
    assert np.array_equal(np.argmax(l, 1), [1, 0])
    assert np.allclose(pr.top2_gap(l), [0.0, 0.1])
