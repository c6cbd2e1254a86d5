"""ssd_verify_attention_noalloc: frontier attention for callers that cannot
allocate device memory (for example a plugin whose host process has reserved
all device memory, or a decode loop that may not call cudaMalloc because it
can synchronise the device).  It uses the library's static device scratch
instead of a caller workspace; its results must match ssd_verify_attention
with a workspace, call after call.  Collected last on purpose: if it fails,
a run stopping at the first failure has already run every other test."""
import numpy as np
import pytest
import torch

import synth
from tests.helpers import ATTN_TOL, attention_error

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
    return (nd.cpu().numpy(), o_ws.float().cpu().numpy(), o_na.float().cpu().numpy(),
            lse_ws.cpu().numpy(), lse_na.cpu().numpy(), wsb)


def test_noalloc_matches_workspace_entry_point_two_calls_in_a_row(ssd):
    # two different problems back to back: the second call must not depend on
    # what the first one left in the shared scratch
    cases = [synth.config1(cache_len=192, seed=0),          # cache split over 3 CTAs
             synth.make_case("long", grid_h=64, grid_w=64, prefix_len=256,
                             cache_len=[256 + 64 * 30 + 5, 256 + 64 * 7], Hq=8, Hkv=4, d=128,
                             V=64, seed=3, with_logits=False)]
    for c in cases:
        nd, o_ws, o_na, lse_ws, lse_na, wsb = _both(ssd, c)
        assert wsb > 256  # the problem really uses split-KV scratch
        for b in range(c.B):
            n = int(nd[b])
            assert n > 0
            for h in range(c.Hq):
                assert attention_error(o_na[b, :n, h], o_ws[b, :n, h]) < ATTN_TOL
            assert np.abs(lse_na[b, :, :n] - lse_ws[b, :, :n]).max() < 2e-2
