"""The C-ABI library builds, loads and exports every entry point that
include/ssd.h declares; host-side argument checks return their codes without
touching a GPU."""
import ctypes
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "ssd.h")


@pytest.fixture(scope="module")
def lib():
    if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
        pytest.skip("nvcc not available")
    from paper_2606_20543_gb300 import build
    build.build()
    import paper_2606_20543_gb300 as ssd
    return ssd


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(ssd_[a-z_]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("ssd_verify_attention", "ssd_accept", "ssd_verify_step", "ssd_frontier",
                     "ssd_lmhead_accept"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    so = ctypes.CDLL(lib.LIB_PATH)
    for name in declared_functions():
        assert hasattr(so, name), name
    assert set(declared_functions()) == set(lib.EXPORTED)


def test_abi_version_and_status_strings(lib):
    assert lib.ssd_abi_version() == 9
    for code, name in lib.STATUS_NAMES.items():
        assert lib.ssd_status_string(code) == name


def test_host_side_validation(lib):
    so = lib.load()
    g = lib.grid(16, 16, 32)
    r = lib.rng(0, 0)
    P = ctypes.c_void_p
    fake = P(0x1000)  # never dereferenced: every call below fails its checks first
    # bad head_dim / group / D_max
    assert so.ssd_verify_attention(ctypes.byref(g), 1, 8, 8, 96, fake, fake, fake, 32, 288, fake,
                                   fake, fake, 0.0, fake, None, fake, 1 << 20, fake, None) == 3
    assert so.ssd_verify_attention(ctypes.byref(g), 1, 8, 3, 64, fake, fake, fake, 32, 288, fake,
                                   fake, fake, 0.0, fake, None, fake, 1 << 20, fake, None) == 2
    assert so.ssd_verify_attention(ctypes.byref(g), 1, 8, 8, 64, fake, fake, fake, 200, 288, fake,
                                   fake, fake, 0.0, fake, None, fake, 1 << 20, fake, None) == 3
    # null pointers
    assert so.ssd_verify_attention(ctypes.byref(g), 1, 8, 8, 64, None, fake, fake, 32, 288, fake,
                                   fake, fake, 0.0, fake, None, fake, 1 << 20, fake, None) == 1
    # accept: vocabulary not a multiple of 4, bad temperature, null rng
    assert so.ssd_accept(4, 4098, fake, fake, 4100, None, 1.0, ctypes.byref(r), fake, fake, None,
                         None, fake, None) == 2
    assert so.ssd_accept(4, 4096, fake, fake, 4096, None, 0.0, ctypes.byref(r), fake, fake, None,
                         None, fake, None) == 1
    assert so.ssd_accept(4, 4096, fake, fake, 4096, None, 1.0, None, fake, fake, None, None, fake,
                         None) == 1
    # misaligned logits
    assert so.ssd_accept(4, 4096, P(0x1004), fake, 4096, None, 1.0, ctypes.byref(r), fake, fake,
                         None, None, fake, None) == 1
    # zero rows is a no-op
    assert so.ssd_accept(0, 4096, None, None, 4096, None, 1.0, ctypes.byref(r), fake, fake, None,
                         None, fake, None) == 0
    # strategies: unknown codes are rejected before anything else; known ones
    # reach the same argument checks as ssd_accept
    for bad in (-1, 3, 99):
        assert so.ssd_accept_strategy(bad, 0, 4096, None, None, 4096, None, 1.0, ctypes.byref(r),
                                      fake, fake, None, None, fake, None) == 1
    # rounds: the reference pointers are required; shift: 2W must fit D_max
    assert so.ssd_accept_round(0, 4, 4096, fake, 4096, None, None, 1.0, ctypes.byref(r), fake,
                               fake, None, None, fake, None) == 1
    assert so.ssd_accept_round(5, 4, 4096, fake, 4096, fake, None, 1.0, ctypes.byref(r), fake,
                               fake, None, None, fake, None) == 1
    assert so.ssd_stage_shift(2, 48, 25, fake, None, None) == 2
    # commit pass: only the rules that need no decisions
    assert so.ssd_commit_pass(ctypes.byref(g), 1, fake, 32, lib.COMMIT_PREFIX, fake, fake, None) == 1
    assert so.ssd_commit_pass(ctypes.byref(g), 1, fake, 15, lib.COMMIT_BLOCK, fake, fake, None) == 2
    assert so.ssd_commit_pass(ctypes.byref(g), 0, None, 32, lib.COMMIT_BLOCK, None, None, None) == 0
    assert so.ssd_stage_shift(0, 48, 24, None, None, None) == 0
    # draft predictor: shapes, null pointers, workspace
    W = so.ssd_draft_predict
    assert W(0, 64, 128, 256, fake, fake, fake, fake, fake, fake, fake, fake, 1e-6, fake, None,
             fake, 1 << 30, fake, None) == 2
    assert W(4, 60, 128, 256, fake, fake, fake, fake, fake, fake, fake, fake, 1e-6, fake, None,
             fake, 1 << 30, fake, None) == 2
    assert W(4, 64, 128, 256, fake, fake, fake, fake, fake, fake, fake, fake, 1e-6, fake, None,
             fake, 1 << 30, fake, None) == 3  # d not a multiple of 128
    assert so.ssd_draft_predict_workspace(4, 64, 128, 256) == 0
    assert W(4, 128, 256, 256, None, fake, fake, fake, fake, fake, fake, fake, 1e-6, fake, None,
             fake, 1 << 30, fake, None) == 1
    assert W(4, 128, 256, 256, fake, fake, fake, fake, fake, fake, fake, fake, -1.0, fake, None,
             fake, 1 << 30, fake, None) == 1
    need = so.ssd_draft_predict_workspace(4, 128, 256, 256)
    assert need > 0
    assert W(4, 128, 256, 256, fake, fake, fake, fake, fake, fake, fake, fake, 1e-6, fake, None,
             fake, need - 1, fake, None) == 7
    for good in (lib.STRATEGY_ACCEPT_REJECT, lib.STRATEGY_GREEDY, lib.STRATEGY_SAMPLE):
        assert so.ssd_accept_strategy(good, 0, 4096, None, None, 4096, None, 1.0,
                                      ctypes.byref(r), fake, fake, None, None, fake, None) == 0
        assert so.ssd_accept_strategy(good, 4, 4098, fake, fake, 4100, None, 1.0,
                                      ctypes.byref(r), fake, fake, None, None, fake, None) == 2
    # frontier: D_max too small for (k_v + 1) * W, end-of-line stride unsupported
    assert so.ssd_frontier(ctypes.byref(g), 1, fake, 31, fake, fake, fake, None) == 2
    g2 = lib.grid(16, 16, 32, row_stride=17)
    assert so.ssd_frontier(ctypes.byref(g2), 1, fake, 32, fake, fake, fake, None) == 3
    # workspace too small
    assert so.ssd_verify_attention(ctypes.byref(g), 1, 8, 8, 64, fake, fake, fake, 32, 288, fake,
                                   fake, fake, 0.0, fake, None, None, 0, fake, None) == 7


def test_verify_accept_and_step_host_validation(lib):
    """ssd_verify_accept / ssd_verify_step reject bad arguments on the host
    (no device memory is touched: every pointer below is a fake)."""
    so = lib.load()
    fake = 0x1000

    def args(**kw):
        a = lib.VerifyArgs()
        a.grid = lib.grid(16, 16, 32)
        a.B, a.Hq, a.Hkv, a.d, a.D_max, a.L_max, a.V = 2, 8, 8, 64, 32, 288, 4096
        a.cache_len = a.q = a.k = a.v = fake
        a.tgt_logits = a.drf_logits = fake
        a.ld = 4096
        a.temperature = 1.0
        a.rng = lib.rng(0, 0)
        for k, v in kw.items():
            setattr(a, k, v)
        return a

    def out(**kw):
        y = lib.VerifyOut()
        for name in ("n_drafts", "draft_pos", "o", "out_tok", "accepted", "ratio",
                     "accepted_count", "accepted_prefix", "next_cache_len", "status"):
            setattr(y, name, fake)
        y.next_cache_len = fake + 0x1000  # disjoint from cache_len
        for k, v in kw.items():
            setattr(y, k, v)
        return y

    def acc(a, y, ws=fake, nbytes=1 << 30):
        return so.ssd_verify_accept(ctypes.byref(a), ctypes.byref(y), ctypes.c_void_p(ws), nbytes,
                                    None)

    assert so.ssd_verify_accept(None, None, None, 0, None) == 1
    assert acc(args(B=0), out()) == 0                                # empty batch: no work
    g17 = lib.grid(16, 16, 32, row_stride=17)
    assert acc(args(grid=g17), out()) == 3                           # end-of-line slots
    assert acc(args(D_max=16), out()) == 2                           # (k_v + 1) W > D_max
    assert acc(args(cache_len=None), out()) == 1
    assert acc(args(), out(draft_pos=None)) == 1                     # the frontier is written
    assert acc(args(commit=99), out()) == 1
    assert acc(args(strategy=7), out()) == 1
    assert acc(args(V=4098, ld=4100), out()) == 2                    # V a multiple of 4
    need = so.ssd_verify_step_workspace(ctypes.byref(args()))
    assert need > 0
    assert acc(args(), out(), nbytes=0) == 7
    # the whole step: the attention's arguments too
    step = so.ssd_verify_step
    assert step(ctypes.byref(args(q=None)), ctypes.byref(out()), ctypes.c_void_p(fake), need,
                None) == 1
    assert step(ctypes.byref(args(d=96)), ctypes.byref(out()), ctypes.c_void_p(fake), need,
                None) == 3
    assert step(ctypes.byref(args()), ctypes.byref(out()), ctypes.c_void_p(fake), need - 1,
                None) == 7
    # next_cache_len overlapping cache_len (the counts advance it beside the attention)
    for at in (fake, fake + 4, fake - 4):
        assert step(ctypes.byref(args()), ctypes.byref(out(next_cache_len=at)),
                    ctypes.c_void_p(fake), need, None) == 1
    # launch counts: acceptance + attention (+ combine) + counts on the logits path,
    # and one more (the frontier) on the fused path
    n_logits = so.ssd_verify_step_launches(ctypes.byref(args()))
    assert n_logits in (3, 4)
    fused = args(tgt_logits=None, drf_logits=None, h_tgt=fake, h_drf=fake, w_tgt=fake,
                 w_drf=fake, hidden=4096)
    assert so.ssd_verify_step_launches(ctypes.byref(fused)) == n_logits + 1


def test_replay_state_file_roundtrip(tmp_path):
    import numpy as np
    from paper_2606_20543_gb300.step import ReplayState
    g = np.full((2, 16), -1, np.int32)
    g[0, :5] = [3, 1, 4, 1, 5]
    st = ReplayState(17, 5, np.array([37, 32], np.int32), g)
    st.save(tmp_path / "s.npz")
    back = ReplayState.load(tmp_path / "s.npz")
    assert (back.step, back.seed) == (17, 5)
    assert np.array_equal(back.cache_len, st.cache_len) and np.array_equal(back.grid_tok, g)
