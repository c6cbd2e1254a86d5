"""ssd_verify_attention_noalloc: frontier attention for callers that cannot
allocate device memory (for example a plugin whose host process has reserved
all device memory for its own pool, or a decode loop that may not call
cudaMalloc because it can synchronise the device).  It uses the library's
static device scratch instead of a caller workspace and runs the same kernels
with the same plan as ssd_verify_attention, so its outputs must equal that
entry point's bit for bit, call after call, whatever an earlier call left in
the shared scratch; one case is also compared with the oracle.  Collected
last on purpose: if it fails, a run stopping at the first failure has
already run every other test."""
import numpy as np
import pytest
import torch

import synth
from oracle import step as ostep
from tests.helpers import ATTN_TOL, attention_error, bf16_to_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def _bf(x):
    return torch.from_numpy(np.ascontiguousarray(x).view(np.int16)).view(torch.bfloat16).cuda()


def _cases():
    return [
        # tcgen05 kernel, cache split over several CTAs (d = 64, 32 query rows per head)
        synth.config1(cache_len=192, seed=0),
        # tcgen05 kernel, GQA 8/4, long caches split over CTAs
        synth.make_case("long_gqa", grid_h=64, grid_w=64, prefix_len=256,
                        cache_len=[256 + 64 * 30 + 5, 256 + 64 * 7], Hq=8, Hkv=4, d=128,
                        V=64, seed=3, with_logits=False),
        # mma.sync kernel (a query group of 3 does not divide 128) with split-KV
        # partials and the combine kernel, both in the scratch
        synth.make_case("mma_sync_split", grid_h=32, grid_w=32, prefix_len=64,
                        cache_len=[64 + 32 * 29 + 3, 64 + 32 * 20 + 31], Hq=6, Hkv=2, d=128,
                        V=64, seed=4, with_logits=False),
    ]


def _both(ssd, c):
    """Run the case through the workspace entry point and the no-allocation one."""
    dev = "cuda"
    g = ssd.grid(c.grid_h, c.grid_w, c.prefix_len, c.row_stride, c.k_v)
    cl = torch.from_numpy(c.cache_len.astype(np.int32)).to(dev)
    nd = torch.empty(c.B, dtype=torch.int32, device=dev)
    pos = torch.empty((c.B, c.D_max), dtype=torch.int32, device=dev)
    st = torch.zeros(1, dtype=torch.int32, device=dev)
    ssd.ssd_frontier(g, c.B, cl, c.D_max, nd, pos, st)
    q, k, v = _bf(c.q), _bf(c.k), _bf(c.v)
    shape = (c.B, c.D_max, c.Hq, c.d)
    o_ws = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
    o_na = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
    lse_ws = torch.zeros((c.B, c.Hq, c.D_max), dtype=torch.float32, device=dev)
    lse_na = torch.zeros((c.B, c.Hq, c.D_max), dtype=torch.float32, device=dev)
    wsb = ssd.ssd_verify_attention_workspace(c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max)
    ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device=dev)
    ssd.ssd_verify_attention(g, c.B, c.Hq, c.Hkv, c.d, cl, nd, pos, c.D_max, c.L_max, q, k, v,
                             0.0, o_ws, lse_ws, ws, wsb, st)
    ssd.ssd_verify_attention_noalloc(g, c.B, c.Hq, c.Hkv, c.d, cl, nd, pos, c.D_max, c.L_max,
                                     q, k, v, 0.0, o_na, lse_na, st)
    torch.cuda.synchronize()
    assert st.item() == 0
    return dict(nd=nd.cpu().numpy(), o_ws=o_ws.float().cpu().numpy(),
                o_na=o_na.float().cpu().numpy(), lse_ws=lse_ws.cpu().numpy(),
                lse_na=lse_na.cpu().numpy(), wsb=wsb)


def _assert_same(c, r):
    for b in range(c.B):
        n = int(r["nd"][b])
        assert n > 0
        assert np.array_equal(r["o_na"][b, :n], r["o_ws"][b, :n]), (c.name, b)
        assert np.array_equal(r["lse_na"][b, :, :n], r["lse_ws"][b, :, :n]), (c.name, b)


def test_noalloc_matches_workspace_entry_point_two_calls_in_a_row(ssd):
    # different problems back to back, then the first one again: no call may
    # depend on what an earlier call left in the shared scratch
    cases = _cases()
    first = None
    for c in cases + [cases[0]]:
        r = _both(ssd, c)
        assert r["wsb"] > 256  # the problem really uses split-KV scratch
        _assert_same(c, r)
        if first is None:
            first = r
    assert np.array_equal(r["o_na"], first["o_na"]) and np.array_equal(r["lse_na"], first["lse_na"])


def test_noalloc_matches_oracle(ssd):
    c = _cases()[2]  # the mma.sync kernel with split-KV partials and the combine
    r = _both(ssd, c)
    att = ostep.attention_step(c.grid_h, c.grid_w, c.prefix_len, c.row_stride, c.k_v,
                               c.cache_len, bf16_to_f64(c.q), bf16_to_f64(c.k), bf16_to_f64(c.v),
                               c.Hq, c.Hkv)
    for b, (o_ref, lse_ref) in att.items():
        n = o_ref.shape[0]
        assert n == int(r["nd"][b]) and n > 0
        for h in range(c.Hq):
            assert attention_error(r["o_na"][b, :n, h], o_ref[:, h]) < ATTN_TOL, (b, h)
        assert np.abs(r["lse_na"][b, :, :n] - lse_ref).max() < 2e-2
