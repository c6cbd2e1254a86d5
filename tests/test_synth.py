"""The seeded input generators: Philox against its published vectors, exact
uniforms, bf16 rounding against torch's conversion (a library routine)."""
import os

import numpy as np
import torch

import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _kat():
    rows = []
    for line in open(os.path.join(GOLDEN, "philox4x32_10_kat.txt")):
        if line.startswith("#") or not line.strip():
            continue
        w = [int(x, 16) for x in line.split()]
        rows.append((w[0:4], w[4:6], w[6:10]))
    return rows


def test_philox_known_answers():
    for ctr, key, out in _kat():
        got = synth.philox4x32_10(np.array(ctr, np.uint32), np.array(key, np.uint32))
        assert [int(x) for x in got] == out


def test_philox_batched_matches_scalar():
    rng = np.random.default_rng(1)
    ctr = rng.integers(0, 2**32, size=(64, 4), dtype=np.uint64).astype(np.uint32)
    key = np.array([0x12345678, 0x9ABCDEF0], np.uint32)
    batched = synth.philox4x32_10(ctr, key)
    for i in range(64):
        assert (synth.philox4x32_10(ctr[i], key) == batched[i]).all()


def test_uniforms_exact_and_in_range():
    u = synth.philox_uniforms(seed=7, offset=3, rows=5000)
    assert u.dtype == np.float32 and u.shape == (5000, 2)
    assert (u >= 0).all() and (u < 1).all()
    scaled = u.astype(np.float64) * 2**24
    assert (scaled == np.round(scaled)).all()
    # different offsets / seeds give different streams; same arguments repeat
    assert not np.array_equal(u, synth.philox_uniforms(7, 4, 5000))
    assert not np.array_equal(u, synth.philox_uniforms(8, 3, 5000))
    assert np.array_equal(u, synth.philox_uniforms(7, 3, 5000))
    # the uniforms are the top 24 bits of words 0 and 1 of block (row, offset, 0, 0)
    blk = synth.philox4x32_10(np.array([11, 3, 0, 0], np.uint32), np.array([7, 0], np.uint32))
    assert u[11, 0] == (int(blk[0]) >> 8) * 2.0**-24
    assert u[11, 1] == (int(blk[1]) >> 8) * 2.0**-24
    # mean / variance of a uniform on [0, 1)
    assert abs(u.mean() - 0.5) < 0.01 and abs(u.var() - 1 / 12) < 0.005


def test_bf16_rounding_matches_torch():
    x = np.random.default_rng(0).standard_normal(200000).astype(np.float32) * 5
    x[:4] = [0.0, -0.0, 1e-40, 3.4e38]
    mine = synth.f32_to_bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(mine, ref)
    back = synth.bf16_bits_to_f32(mine)
    assert np.array_equal(back, torch.from_numpy(x).to(torch.bfloat16).float().numpy())


def test_workload_shapes():
    c = synth.config1()
    assert (c.B, c.Hq, c.Hkv, c.d, c.V, c.D_max, c.L_max) == (1, 8, 8, 64, 4096, 32, 288)
    assert c.q.shape == (1, 32, 8, 64) and c.k.shape == (1, 8, 288, 64)
    assert c.tgt_logits.shape == (32, 4096) and c.uniforms.shape == (32, 2)
    assert list(synth.config2_points()) == list(range(120, 697, 24)) and len(synth.config2_points()) == 25
    c3 = synth.config3(with_attention=False, with_logits=False)
    assert c3.B == 16 and c3.cache_len.min() >= 64 and c3.cache_len.max() <= 1088
    # Zipf draft logits: a permutation of -1.1 ln(rank)
    c3s = synth.make_case("z", grid_h=4, grid_w=4, prefix_len=2, cache_len=[2], Hq=2, Hkv=1,
                          d=64, V=64, seed=1, logits="zipf")
    row = np.sort(c3s.drf_logits[0])[::-1]
    assert np.allclose(row, -1.1 * np.log(np.arange(1, 65)), atol=1e-5)
