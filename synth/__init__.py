"""Seeded synthetic inputs for the SSD verification pass.

This module is shared by the CUDA path's tests, by ``bench.py`` and by the CPU
oracle's tests.  It holds none of the method's arithmetic: only random draws,
bf16 rounding of those draws, and the Philox4x32-10 counter-based generator
(Salmon, Moraes, Dror, Shaw, "Parallel random numbers: as easy as 1, 2, 3",
SC'11) from which the per-draft uniforms are taken.  The frontier (which
positions are drafted), the mask, softmax, acceptance and resampling live in
``oracle/`` (CPU) and in the CUDA library, never here.

Workload shapes follow the paper's backbones (Sec. 4 "Models": 24x24, 48x48,
90x90 grids; App. "Generalization", codebooks 8192-32768) and the five
verification workloads this library is measured on; see ``WORKLOADS``.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional

import numpy as np

# ----------------------------------------------------------------------------
# Philox4x32-10 (Salmon et al., SC'11, Sec. 4.3): a 4x32-bit counter and a
# 2x32-bit key, ten rounds.  Each round multiplies words 0 and 2 by the two
# round multipliers, and mixes the high halves with the other words and the
# key; the key is bumped by the two Weyl constants between rounds.
# ----------------------------------------------------------------------------
PHILOX_M0 = np.uint64(0xD2511F53)
PHILOX_M1 = np.uint64(0xCD9E8D57)
PHILOX_W0 = np.uint64(0x9E3779B9)
PHILOX_W1 = np.uint64(0xBB67AE85)
_MASK32 = np.uint64(0xFFFFFFFF)
_SHIFT32 = np.uint64(32)


def philox4x32_10(ctr: np.ndarray, key: np.ndarray) -> np.ndarray:
    """Philox4x32-10 block function.

    ctr: uint32 array of shape (..., 4); key: uint32 array broadcastable to
    (..., 2).  Returns the uint32 output block of shape (..., 4).
    """
    ctr = np.asarray(ctr, dtype=np.uint32)
    key = np.asarray(key, dtype=np.uint32)
    c0 = ctr[..., 0].astype(np.uint64)
    c1 = ctr[..., 1].astype(np.uint64)
    c2 = ctr[..., 2].astype(np.uint64)
    c3 = ctr[..., 3].astype(np.uint64)
    k0 = np.broadcast_to(key[..., 0], c0.shape).astype(np.uint64)
    k1 = np.broadcast_to(key[..., 1], c0.shape).astype(np.uint64)
    for _ in range(10):
        prod0 = PHILOX_M0 * c0
        prod1 = PHILOX_M1 * c2
        hi0, lo0 = prod0 >> _SHIFT32, prod0 & _MASK32
        hi1, lo1 = prod1 >> _SHIFT32, prod1 & _MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
        k0 = (k0 + PHILOX_W0) & _MASK32
        k1 = (k1 + PHILOX_W1) & _MASK32
    return np.stack([c0, c1, c2, c3], axis=-1).astype(np.uint32)


def philox_uniforms(seed: int, offset: int, rows: int, row0: int = 0) -> np.ndarray:
    """Per-draft uniforms, float32 [rows, 2] = (u_acc, u_res).

    Counter = (row, offset_lo, offset_hi, 0), key = (seed_lo, seed_hi); the
    uniforms are the top 24 bits of output words 0 and 1 times 2^-24, so they
    lie in [0, 1 - 2^-24] and are exact in float32 and float64.
    """
    r = np.arange(row0, row0 + rows, dtype=np.uint64)
    ctr = np.zeros((rows, 4), dtype=np.uint32)
    ctr[:, 0] = (r & _MASK32).astype(np.uint32)
    ctr[:, 1] = np.uint32(offset & 0xFFFFFFFF)
    ctr[:, 2] = np.uint32((offset >> 32) & 0xFFFFFFFF)
    key = np.array([seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF], dtype=np.uint32)
    out = philox4x32_10(ctr, key)
    u = (out[:, :2] >> np.uint32(8)).astype(np.float64) * (2.0 ** -24)
    return u.astype(np.float32)


# ----------------------------------------------------------------------------
# bf16 storage: uint16 bit patterns, rounded to nearest-even from float32.
# ----------------------------------------------------------------------------
def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 to bf16 (nearest-even) and return the uint16 bit patterns."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = np.uint32(0x7FFF) + ((b >> np.uint32(16)) & np.uint32(1))
    out = ((b + rounding) >> np.uint32(16)).astype(np.uint16)
    nan = np.isnan(np.asarray(x, dtype=np.float32))
    if nan.any():
        out[nan] = np.uint16(0x7FC0)
    return out


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns (uint16) to float32 exactly."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def bf16_normal(rng: np.random.Generator, shape, std: float) -> np.ndarray:
    """bf16 bits of N(0, std^2) draws (float32 draw, then nearest-even)."""
    x = rng.standard_normal(size=shape, dtype=np.float32) * np.float32(std)
    return f32_to_bf16_bits(x)


# ----------------------------------------------------------------------------
# Workloads
# ----------------------------------------------------------------------------
@dataclass
class Case:
    """One verification problem (a batch of B sequences), host arrays only.

    Layouts (row-major, innermost last):
      q        bf16 bits [B, D_max, Hq, d]    draft queries, slot j of seq b
      k, v     bf16 bits [B, Hkv, L_max, d]   cache slots [0, cache_len) then
                                              the drafts' own K/V at
                                              [cache_len, cache_len + n_d)
      tgt_logits, drf_logits float32 [B*D_max, V]   row b*D_max + j
      h_tgt, h_drf bf16 bits [B*D_max, hidden] (fused-head workloads)
      w_tgt, w_drf bf16 bits [hidden, V]
      uniforms float32 [B*D_max, 2]           (u_acc, u_res) per row
    """
    name: str
    grid_h: int
    grid_w: int
    prefix_len: int
    row_stride: int
    k_v: int
    B: int
    Hq: int
    Hkv: int
    d: int
    D_max: int
    L_max: int
    V: int
    cache_len: np.ndarray
    seed: int
    offset: int
    q: Optional[np.ndarray] = None
    k: Optional[np.ndarray] = None
    v: Optional[np.ndarray] = None
    tgt_logits: Optional[np.ndarray] = None
    drf_logits: Optional[np.ndarray] = None
    uniforms: Optional[np.ndarray] = None
    hidden: int = 0
    h_tgt: Optional[np.ndarray] = None
    h_drf: Optional[np.ndarray] = None
    w_tgt: Optional[np.ndarray] = None
    w_drf: Optional[np.ndarray] = None
    meta: dict = field(default_factory=dict)

    @property
    def rows(self) -> int:
        return self.B * self.D_max


def _logits_normal(rng, rows, V, std=2.0):
    tgt = rng.standard_normal(size=(rows, V), dtype=np.float32) * np.float32(std)
    drf = rng.standard_normal(size=(rows, V), dtype=np.float32) * np.float32(std)
    return tgt, drf


def _logits_zipf(rng, rows, V, s=1.1, std=2.0):
    """Draft logits -s*ln(rank) over a seeded per-row permutation of the
    vocabulary (a Zipf(s) draft distribution); target = draft + N(0, std^2)."""
    base = (-s * np.log(np.arange(1, V + 1, dtype=np.float64))).astype(np.float32)
    drf = np.empty((rows, V), dtype=np.float32)
    for r in range(rows):
        drf[r] = base[rng.permutation(V)]
    tgt = drf + rng.standard_normal(size=(rows, V), dtype=np.float32) * np.float32(std)
    return tgt, drf


def make_case(name, *, grid_h, grid_w, prefix_len, cache_len, Hq, Hkv, d, V,
              seed, offset=0, k_v=1, row_stride=None, qkv_std=1.0 / 8.0,
              logits="normal", logits_std=2.0, hidden=0, per_seq_seed=False,
              with_attention=True, with_logits=True, L_max=None) -> Case:
    """Generate one seeded Case.

    ``cache_len`` lists each sequence's committed KV length.  D_max is the
    frontier's upper bound (k_v + 1) * W (the remainder of the current row
    plus k_v full rows), L_max the full sequence prefix + H * row_stride.
    With ``per_seq_seed`` sequence b draws from its own generator seeded
    ``seed + b`` (one seed per sweep point); otherwise one generator serves
    the whole batch.
    """
    row_stride = grid_w if row_stride is None else row_stride
    cache_len = np.asarray(cache_len, dtype=np.int32)
    B = int(cache_len.shape[0])
    D_max = (k_v + 1) * grid_w
    L_max = prefix_len + grid_h * row_stride if L_max is None else L_max
    c = Case(name=name, grid_h=grid_h, grid_w=grid_w, prefix_len=prefix_len,
             row_stride=row_stride, k_v=k_v, B=B, Hq=Hq, Hkv=Hkv, d=d,
             D_max=D_max, L_max=L_max, V=V, cache_len=cache_len, seed=seed,
             offset=offset, hidden=hidden)
    gens = ([np.random.default_rng(np.random.PCG64(seed + b)) for b in range(B)]
            if per_seq_seed else [np.random.default_rng(np.random.PCG64(seed))] * B)
    if with_attention:
        c.q = np.empty((B, D_max, Hq, d), dtype=np.uint16)
        c.k = np.empty((B, Hkv, L_max, d), dtype=np.uint16)
        c.v = np.empty((B, Hkv, L_max, d), dtype=np.uint16)
        for b in range(B):
            g = gens[b]
            c.q[b] = bf16_normal(g, (D_max, Hq, d), qkv_std)
            c.k[b] = bf16_normal(g, (Hkv, L_max, d), qkv_std)
            c.v[b] = bf16_normal(g, (Hkv, L_max, d), qkv_std)
    if with_logits and hidden == 0:
        c.tgt_logits = np.empty((B * D_max, V), dtype=np.float32)
        c.drf_logits = np.empty((B * D_max, V), dtype=np.float32)
        for b in range(B):
            g = gens[b]
            sl = slice(b * D_max, (b + 1) * D_max)
            if logits == "normal":
                c.tgt_logits[sl], c.drf_logits[sl] = _logits_normal(g, D_max, V, logits_std)
            elif logits == "zipf":
                c.tgt_logits[sl], c.drf_logits[sl] = _logits_zipf(g, D_max, V, 1.1, logits_std)
            else:
                raise ValueError(logits)
    if hidden:
        g = gens[0]
        c.h_tgt = bf16_normal(g, (B * D_max, hidden), 1.0)
        c.h_drf = bf16_normal(g, (B * D_max, hidden), 1.0)
        c.w_tgt = bf16_normal(g, (hidden, V), 0.02)
        c.w_drf = bf16_normal(g, (hidden, V), 0.02)
    c.uniforms = philox_uniforms(seed, offset, B * D_max)
    return c


def config1(cache_len=192, seed=0, **kw) -> Case:
    """16x16 grid after a 32-token prefix, one sequence, 8 heads x 64,
    vocabulary 4096, N(0, 2^2) logits.  cache_len 192 puts the frontier on
    grid rows 10-11; 112 puts it on rows 5-6."""
    return make_case("cfg1_16x16_b1", grid_h=16, grid_w=16, prefix_len=32,
                     cache_len=[cache_len], Hq=8, Hkv=8, d=64, V=4096, seed=seed, **kw)


def config2_points():
    """The cache lengths of the 24x24 sweep: 120 -> 696 in steps of one row."""
    return list(range(120, 696 + 1, 24))


def config2(points=None, seed0=0, **kw) -> Case:
    """24x24 grid after a 120-token prefix, 16 heads x 128 (MHA), vocabulary
    16384, N(0, 2^2) logits.  Each sweep point is an independent batch-1
    problem with its own seed (seed0 + index); they are stacked as B rows."""
    pts = config2_points() if points is None else list(points)
    return make_case("cfg2_24x24_sweep", grid_h=24, grid_w=24, prefix_len=120,
                     cache_len=pts, Hq=16, Hkv=16, d=128, V=16384, seed=seed0,
                     per_seq_seed=True, **kw)


def config3(seed=3, B=16, **kw) -> Case:
    """16 sequences of 32x32 after 64-token prefixes, GQA 32/8 x 128, cache
    lengths uniform in [64, 1088], vocabulary 16384, Zipf(1.1) draft vs
    N(0, 2^2)-perturbed target logits."""
    rng = np.random.default_rng(np.random.PCG64(seed + 1_000_003))
    cl = rng.integers(64, 1088 + 1, size=B).astype(np.int32)
    return make_case("cfg3_32x32_b16_gqa", grid_h=32, grid_w=32, prefix_len=64,
                     cache_len=cl, Hq=32, Hkv=8, d=128, V=16384, seed=seed,
                     logits="zipf", **kw)


def config4(points=None, seed0=4, hidden=4096, **kw) -> Case:
    """Config-2 shapes with the lm_head fused: hidden states bf16 N(0,1)
    [rows x 4096] for target and draft, lm_head weights bf16 N(0, 0.02^2)
    [4096 x 16384] for target and draft."""
    pts = [120] if points is None else list(points)
    return make_case("cfg4_24x24_fused_head", grid_h=24, grid_w=24, prefix_len=120,
                     cache_len=pts, Hq=16, Hkv=16, d=128, V=16384, seed=seed0,
                     per_seq_seed=True, hidden=hidden, **kw)


def config5(seed=5, B=8, cache_len=None, **kw) -> Case:
    """8 sequences of 64x64 after 256-token prefixes, 32 heads x 128 MHA,
    vocabulary 65536, Zipf(1.1) draft vs N(0, 2^2)-perturbed target logits.
    The replay starts every sequence at cache_len = prefix (empty grid)."""
    cl = [256] * B if cache_len is None else cache_len
    return make_case("cfg5_64x64_b8_replay", grid_h=64, grid_w=64, prefix_len=256,
                     cache_len=cl, Hq=32, Hkv=32, d=128, V=65536, seed=seed,
                     logits="zipf", **kw)


WORKLOADS = {
    1: config1,
    2: config2,
    3: config3,
    4: config4,
    5: config5,
}


def replay_pool(B, D_max, V, seed, sets=2, logits="zipf"):
    """Logit sets for a replay: step t uses set t % sets (rows b * D_max + j)
    and Philox uniforms with offset t.  Returns a list of (tgt, drf) pairs."""
    out = []
    for k in range(sets):
        rng = np.random.default_rng(np.random.PCG64(seed * 1000 + k))
        if logits == "zipf":
            out.append(_logits_zipf(rng, B * D_max, V))
        else:
            out.append(_logits_normal(rng, B * D_max, V))
    return out
