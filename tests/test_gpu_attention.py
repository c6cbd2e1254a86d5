"""GPU parity of frontier attention (step a2) against the oracle: normwise
max relative error 2e-2 per (sequence, head) for bf16 inputs, log-sum-exp
within 2e-2 absolute."""
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


def run_attention(ssd, c, scale=0.0, edit_pos=None, ws=None):
    dev = "cuda"
    g = ssd.grid(c.grid_h, c.grid_w, c.prefix_len, c.row_stride, c.k_v)
    cl = torch.from_numpy(c.cache_len.astype(np.int32)).to(dev)
    nd = torch.empty(c.B, dtype=torch.int32, device=dev)
    pos = torch.empty((c.B, c.D_max), dtype=torch.int32, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    ssd.ssd_frontier(g, c.B, cl, c.D_max, nd, pos, status)
    if edit_pos is not None:
        edit_pos(pos)
    q, k, v = _bf(c.q), _bf(c.k), _bf(c.v)
    o = torch.zeros((c.B, c.D_max, c.Hq, c.d), dtype=torch.bfloat16, device=dev)
    lse = torch.zeros((c.B, c.Hq, c.D_max), dtype=torch.float32, device=dev)
    wsb = ssd.ssd_verify_attention_workspace(c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max)
    if ws is None:
        ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device=dev)
    ssd.ssd_verify_attention(g, c.B, c.Hq, c.Hkv, c.d, cl, nd, pos, c.D_max, c.L_max, q, k, v,
                             scale, o, lse, ws, wsb, status)
    torch.cuda.synchronize()
    return (o.float().cpu().numpy(), lse.cpu().numpy(), nd.cpu().numpy(), int(status.item()))


def check_case(ssd, c, seqs=None, scale=0.0, edit_pos=None, want_status=0):
    o, lse, nd, st = run_attention(ssd, c, scale, edit_pos)
    assert st == want_status
    q, k, v = bf16_to_f64(c.q), bf16_to_f64(c.k), bf16_to_f64(c.v)
    ref = ostep.attention_step(c.grid_h, c.grid_w, c.prefix_len, c.row_stride, c.k_v, c.cache_len,
                               q, k, v, c.Hq, c.Hkv, scale if scale else None, seqs)
    worst = 0.0
    for b, (o_ref, lse_ref) in ref.items():
        n = o_ref.shape[0]
        assert nd[b] == n
        for h in range(c.Hq):
            if n == 0:
                continue
            e = attention_error(o[b, :n, h], o_ref[:, h])
            worst = max(worst, e)
            assert e < ATTN_TOL, f"b={b} h={h} err={e}"
            assert np.abs(lse[b, h, :n] - lse_ref[h]).max() < 2e-2
    return worst


def test_config1_shape(ssd):
    check_case(ssd, synth.config1(cache_len=192))
    check_case(ssd, synth.config1(cache_len=112))


def test_config2_sweep_points(ssd):
    # first, middle, last-with-drafts and empty-frontier points of the sweep
    c = synth.config2(points=[120, 144, 408, 672, 696], with_logits=False)
    check_case(ssd, c)


def test_gqa_ragged_batch(ssd):
    # config-3 shapes (GQA 32/8 x 128) on a smaller ragged batch
    rng = np.random.default_rng(5)
    cl = rng.integers(64, 1088 + 1, size=5).astype(np.int32)
    cl[0] = 64          # empty cache beyond the prefix, drafts start at row 0
    cl[1] = 64 + 1024   # complete grid: no drafts
    cl[2] = 64 + 31     # one draft left on the row plus the next row
    c = synth.make_case("gqa", grid_h=32, grid_w=32, prefix_len=64, cache_len=cl, Hq=32, Hkv=8,
                        d=128, V=64, seed=5, with_logits=False)
    check_case(ssd, c)


def test_head_dim_64_and_custom_scale(ssd):
    c = synth.make_case("d64", grid_h=12, grid_w=12, prefix_len=7, cache_len=[7, 50, 100, 151],
                        Hq=6, Hkv=2, d=64, V=64, seed=6, with_logits=False)
    check_case(ssd, c)
    check_case(ssd, c, scale=0.05)


def test_long_cache_many_splits(ssd):
    # a long cache on one sequence: the key range is split over CTAs and merged
    c = synth.make_case("long", grid_h=64, grid_w=64, prefix_len=256, cache_len=[256 + 64 * 40 + 9],
                        Hq=4, Hkv=4, d=128, V=64, seed=7, with_logits=False)
    check_case(ssd, c)


def test_split_merge_ignores_workspace_contents(ssd):
    """A KV cache split over CTAs: partials in the workspace, merged by the
    combine kernel.  Whatever the workspace held before (all ones, zeros, the
    partials of earlier launches of this and of another case), the result is
    the same, bit for bit."""
    c = synth.make_case("long", grid_h=64, grid_w=64, prefix_len=256, cache_len=[256 + 64 * 40 + 9],
                        Hq=4, Hkv=4, d=128, V=64, seed=7, with_logits=False)
    other = synth.make_case("long2", grid_h=64, grid_w=64, prefix_len=256,
                            cache_len=[256 + 64 * 21 + 3], Hq=4, Hkv=4, d=128, V=64, seed=8,
                            with_logits=False)
    wsb = ssd.ssd_verify_attention_workspace(c.B, c.Hq, c.Hkv, c.d, c.D_max, c.L_max)
    ws = torch.empty(max(wsb, 256), dtype=torch.uint8, device="cuda")
    outs = []
    for fill in (0xFF, 0x00, None, "other", None):
        if fill == "other":
            run_attention(ssd, other, ws=ws)
        elif fill is not None:
            ws.fill_(fill)
        outs.append(run_attention(ssd, c, ws=ws))
    for o, lse, nd, st in outs:
        assert st == 0
        assert np.array_equal(o, outs[0][0]) and np.array_equal(lse, outs[0][1])
    check_case(ssd, c)


def test_k_v_two_rows(ssd):
    c = synth.make_case("kv2", grid_h=10, grid_w=10, prefix_len=5, cache_len=[5, 38, 85],
                        Hq=8, Hkv=8, d=128, V=64, seed=8, k_v=2, with_logits=False)
    check_case(ssd, c)


def test_bad_cache_length_sets_status(ssd):
    c = synth.config1(cache_len=192)
    c.cache_len = np.array([10], np.int32)  # below the prefix
    o, lse, nd, st = run_attention(ssd, c)
    assert st == 6 and nd[0] == 0


def test_head_dim_64_gqa_tensor_core_path(ssd):
    # 32 drafts x 4 query heads per KV head = 128 rows per KV group, d = 64
    c = synth.make_case("d64gqa", grid_h=16, grid_w=16, prefix_len=32, cache_len=[32, 96, 200],
                        Hq=8, Hkv=2, d=64, V=64, seed=9, with_logits=False)
    check_case(ssd, c)


def test_mma_sync_and_tensor_core_paths_agree(ssd):
    """Related problems on both kernels: 3 query heads per KV head (128 is not
    a multiple of 3: mma.sync), and MHA and 2 heads per KV head on the same
    caches (tcgen05); all must match the oracle."""
    c = synth.make_case("gqa3", grid_h=24, grid_w=24, prefix_len=120, cache_len=[120, 408],
                        Hq=12, Hkv=4, d=128, V=64, seed=10, with_logits=False)
    check_case(ssd, c)
    c1 = synth.make_case("mha48", grid_h=24, grid_w=24, prefix_len=120, cache_len=[120, 408],
                         Hq=16, Hkv=16, d=128, V=64, seed=10, with_logits=False)
    check_case(ssd, c1)
    c2 = synth.make_case("gqa96", grid_h=24, grid_w=24, prefix_len=120, cache_len=[120, 408],
                         Hq=16, Hkv=8, d=128, V=64, seed=10, with_logits=False)
    check_case(ssd, c2)


def _gqa_batch(B, seed):
    rng = np.random.default_rng(seed)
    cl = rng.integers(64, 1088 + 1, size=B).astype(np.int32)
    return synth.make_case("gqa_many", grid_h=32, grid_w=32, prefix_len=64, cache_len=cl, Hq=32,
                           Hkv=8, d=128, V=64, seed=seed, with_logits=False)


def test_tensor_core_items_outnumber_sms(ssd):
    """24 sequences x 8 KV heads x 2 query tiles = 384 work items: every CTA
    of the persistent tcgen05 kernel takes two or three items in turn (item
    slots, Q buffers and O buffers reused)."""
    check_case(ssd, _gqa_batch(24, 11))


def test_tensor_core_bad_draft_position_skips_only_its_sequence(ssd):
    c = _gqa_batch(20, 12)
    hw = c.grid_h * c.grid_w

    def corrupt(pos):
        pos[3, 0] = hw + 5  # sequence 3 reads past the grid

    o, lse, nd, st = run_attention(ssd, c, edit_pos=corrupt)
    assert st == 6
    q, k, v = bf16_to_f64(c.q), bf16_to_f64(c.k), bf16_to_f64(c.v)
    seqs = [b for b in range(c.B) if b != 3]
    ref = ostep.attention_step(c.grid_h, c.grid_w, c.prefix_len, c.row_stride, c.k_v, c.cache_len,
                               q, k, v, c.Hq, c.Hkv, None, seqs)
    for b, (o_ref, _) in ref.items():
        n = o_ref.shape[0]
        for h in range(c.Hq):
            if n:
                assert attention_error(o[b, :n, h], o_ref[:, h]) < ATTN_TOL, f"b={b} h={h}"
    assert not o[3].any()  # the bad sequence is not written


def _check_permuted_frontier(ssd, c):
    """The drafts of every sequence in a shuffled order (valid, not increasing
    positions): the kernels take the general visibility path.  The oracle gets
    the same draft order."""
    from oracle import attention as oatt
    rng = np.random.default_rng(13)
    perms = {}

    def permute(pos):
        host = pos.cpu().numpy()
        nd_all = [len(ostep.sequence_frontier(c.grid_h, c.grid_w, c.prefix_len, c.cache_len[b],
                                             c.k_v)[0]) for b in range(c.B)]
        for b in range(c.B):
            n = nd_all[b]
            perms[b] = rng.permutation(n)
            host[b, :n] = host[b, :n][perms[b]]
        pos.copy_(torch.from_numpy(host))

    o, lse, nd, st = run_attention(ssd, c, edit_pos=permute)
    assert st == 0
    q, k, v = bf16_to_f64(c.q), bf16_to_f64(c.k), bf16_to_f64(c.v)
    for b in range(c.B):
        coords, _ = ostep.sequence_frontier(c.grid_h, c.grid_w, c.prefix_len, c.cache_len[b], c.k_v)
        n = len(coords)
        if n == 0:
            continue
        pc = [coords[i] for i in perms[b]]
        o_ref, lse_ref = oatt.verify_attention(q[b, :n], k[b], v[b], int(c.cache_len[b]), pc,
                                               c.prefix_len, c.row_stride, c.Hq, c.Hkv)
        for h in range(c.Hq):
            assert attention_error(o[b, :n, h], o_ref[:, h]) < ATTN_TOL, f"b={b} h={h}"
            assert np.abs(lse[b, h, :n] - lse_ref[h]).max() < 2e-2


def test_tensor_core_shuffled_draft_order(ssd):
    _check_permuted_frontier(ssd, _gqa_batch(6, 14))


def test_mma_sync_shuffled_draft_order(ssd):
    # 3 query heads per KV head: the mma.sync kernel
    c = synth.make_case("gqa3_shuffled", grid_h=24, grid_w=24, prefix_len=120,
                        cache_len=[120, 144, 408, 672], Hq=12, Hkv=4, d=128, V=64, seed=15,
                        with_logits=False)
    _check_permuted_frontier(ssd, c)


def test_sweep_shape_shuffled_draft_order(ssd):
    c = synth.config2(points=[120, 144, 408, 672], with_logits=False)
    _check_permuted_frontier(ssd, c)


@pytest.mark.parametrize("B", [1, 20])
def test_empty_cache_and_no_prefix(ssd, B):
    """The first verification pass of an image with no text prefix: cache
    length 0, so every draft attends to itself and the drafts before it only
    (the whole key range is the drafted block).  B = 1 splits nothing; B = 20
    adds sequences at their last row and finished ones (no drafts)."""
    cl = [0] + [24 * 23 + (k % 24) for k in range(1, B)]
    if B > 1:
        cl[1] = 24 * 24  # finished grid: empty frontier
    c = synth.make_case("no_prefix", grid_h=24, grid_w=24, prefix_len=0, cache_len=cl, Hq=8,
                        Hkv=8, d=128, V=64, seed=17, with_logits=False)
    check_case(ssd, c)
