"""Oracle pins for frontier attention (Sec. 3.3 "Verification as Auto
Correction"): against the library's scaled_dot_product_attention on the
concatenated sequence with a causal mask, and against closed forms."""
import numpy as np
import pytest
import torch

from oracle import attention as att
from oracle import frontier as fr


def _sdpa_full_causal(q_all, k_all, v_all, scale):
    """Textbook causal attention of a whole sequence (torch, float64, CPU)."""
    L = q_all.shape[0]
    mask = torch.ones(L, L, dtype=torch.bool).tril()
    q = torch.from_numpy(q_all).permute(1, 0, 2)[None]
    k = torch.from_numpy(k_all).permute(1, 0, 2)[None]
    v = torch.from_numpy(v_all).permute(1, 0, 2)[None]
    o = torch.nn.functional.scaled_dot_product_attention(q, k, v, attn_mask=mask, scale=scale)
    return o[0].permute(1, 0, 2).numpy()


@pytest.mark.parametrize("H,W,P,n_c,Hq,Hkv,d", [
    (6, 6, 4, 0, 2, 2, 16), (6, 6, 4, 9, 4, 2, 16), (5, 7, 3, 20, 4, 1, 32), (4, 4, 0, 12, 2, 2, 8)])
def test_matches_full_causal_sdpa(H, W, P, n_c, Hq, Hkv, d):
    """Drafts sit at the end of the raster sequence, so their rows of full causal
    attention over [cache ; drafts] are exactly frontier attention."""
    rng = np.random.default_rng(0)
    coords = fr.frontier(H, W, P, P + n_c)
    n = len(coords)
    cache_len = P + n_c
    L = cache_len + n
    # a whole sequence of queries/keys/values; the drafts' queries are the last n
    q_all = rng.standard_normal((L, Hq, d))
    k_all = rng.standard_normal((L, Hkv, d))
    v_all = rng.standard_normal((L, Hkv, d))
    g = Hq // Hkv
    k_rep = np.repeat(k_all, g, axis=1)
    v_rep = np.repeat(v_all, g, axis=1)
    scale = 1 / np.sqrt(d)
    ref = _sdpa_full_causal(q_all, k_rep, v_rep, scale)[cache_len:]
    o, lse = att.verify_attention(q_all[cache_len:], k_all.transpose(1, 0, 2),
                                  v_all.transpose(1, 0, 2), cache_len, coords, P, W, Hq, Hkv)
    assert np.allclose(o, ref, rtol=1e-10, atol=1e-12)
    # lse: log of the softmax denominator, checked against a direct sum
    for h in range(Hq):
        for j in range(n):
            s = scale * (k_all[:cache_len + j + 1, h // g] @ q_all[cache_len + j, h])
            assert np.isclose(lse[h, j], np.log(np.exp(s).sum()), rtol=1e-12)


def test_single_visible_key():
    """Empty prefix and cache: the first draft sees only its own key, so its
    output is its own value row for any query."""
    rng = np.random.default_rng(1)
    coords = fr.frontier(3, 3, 0, 0)
    n = len(coords)
    q = rng.standard_normal((n, 2, 8)) * 10
    k = rng.standard_normal((2, n, 8))
    v = rng.standard_normal((2, n, 8))
    o, lse = att.verify_attention(q, k, v, 0, coords, 0, 3, 2, 2)
    assert np.allclose(o[0], v[:, 0], rtol=0, atol=1e-14)
    assert np.allclose(lse[:, 0], (q[0] * k[:, 0]).sum(-1) / np.sqrt(8), rtol=1e-13)


def test_zero_query_gives_mean_of_visible_values():
    rng = np.random.default_rng(2)
    P, W = 5, 4
    coords = fr.frontier(4, W, P, P + 6)
    n = len(coords)
    cache_len = P + 6
    q = np.zeros((n, 1, 8))
    k = rng.standard_normal((1, cache_len + n, 8))
    v = rng.standard_normal((1, cache_len + n, 8))
    o, _ = att.verify_attention(q, k, v, cache_len, coords, P, W, 1, 1)
    for j in range(n):
        assert np.allclose(o[j, 0], v[0, :cache_len + j + 1].mean(0), atol=1e-14)


def test_gqa_group_mapping():
    """Query head h reads KV head h // (Hq / Hkv): perturbing KV head 1 changes
    exactly the query heads of group 1."""
    rng = np.random.default_rng(3)
    coords = fr.frontier(4, 4, 2, 6)
    n = len(coords)
    q = rng.standard_normal((n, 8, 16))
    k = rng.standard_normal((4, 6 + n, 16))
    v = rng.standard_normal((4, 6 + n, 16))
    o1, _ = att.verify_attention(q, k, v, 6, coords, 2, 4, 8, 4)
    v2 = v.copy()
    v2[1] += 1.0
    o2, _ = att.verify_attention(q, k, v2, 6, coords, 2, 4, 8, 4)
    changed = np.abs(o1 - o2).max(axis=(0, 2)) > 1e-9
    assert list(np.nonzero(changed)[0]) == [2, 3]


def test_keys_past_the_block_are_ignored():
    """Slots beyond cache_len + n_d hold garbage and must not matter."""
    rng = np.random.default_rng(4)
    coords = fr.frontier(4, 4, 2, 6)
    n = len(coords)
    q = rng.standard_normal((n, 2, 16))
    k = rng.standard_normal((2, 64, 16))
    v = rng.standard_normal((2, 64, 16))
    o1, _ = att.verify_attention(q, k, v, 6, coords, 2, 4, 2, 2)
    k[:, 6 + n:] = 1e3
    v[:, 6 + n:] = -1e3
    o2, _ = att.verify_attention(q, k, v, 6, coords, 2, 4, 2, 2)
    assert np.array_equal(o1, o2)
