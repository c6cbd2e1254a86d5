"""Failure detection on the GPU without a fault: a bounded device wait that
runs out.  The fused lm_head's CTAs meet at grid barriers, and the draft
predictor's CTAs wait for the previous product's tiles; with
ssd_set_barrier_shortfall(1) each barrier waits for one arrival more than the
CTAs make (a count nothing completes), so every CTA gives up after the short
poll limit set by ssd_set_wait_limit, records SSD_ERR_TIMEOUT, skips its
remaining work, releases its tensor memory and returns.  The stream then
synchronises cleanly and the next normal call on the same context is
correct."""
import numpy as np
import pytest
import torch

from oracle import lmhead as olm
from tests.helpers import FUSED_PROB_TOL, bf16_to_f64, compare_decisions
from tests.test_gpu_lmhead import make_inputs, run_fused

pytestmark = pytest.mark.gpu

SSD_ERR_TIMEOUT = 5


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def test_lmhead_grid_barrier_runs_out_and_the_context_stays_usable(ssd):
    rows, K, V = 48, 256, 2048
    ht, hd, wt, wd, u = make_inputs(rows, K, V, 21, 0.05)
    ssd.ssd_set_wait_limit(1 << 12)
    ssd.ssd_set_barrier_shortfall(1)
    try:
        tok, acc, ratio, _, st = run_fused(ssd, ht, hd, wt, wd, u)
    finally:
        ssd.ssd_set_barrier_shortfall(0)
        ssd.ssd_set_wait_limit(0)
    assert st == SSD_ERR_TIMEOUT
    # the kernel gave up before its decisions: no output row was written
    assert np.all(tok == -7) and np.all(acc == 7) and np.all(ratio == 0)
    torch.cuda.synchronize()  # the context is intact: no sticky error
    tok, acc, ratio, lse, st = run_fused(ssd, ht, hd, wt, wd, u)
    assert st == 0
    ref = olm.lmhead_accept(bf16_to_f64(ht), bf16_to_f64(hd), bf16_to_f64(wt), bf16_to_f64(wd), u)
    compare_decisions(ref, tok, acc, ratio, lse, what="after a timeout", tol=FUSED_PROB_TOL)


def test_predictor_wait_runs_out_and_the_context_stays_usable(ssd):
    from tests.test_gpu_predictor import _case, _check, _bf_dev
    rows, d, m, V = 16, 256, 512, 2048
    w, g1, g2 = _case(31, rows, d, m, V)
    dev = {k: _bf_dev(v) for k, v in w.items()}
    wsb = ssd.ssd_draft_predict_workspace(rows, d, m, V)
    ws = torch.empty(wsb, dtype=torch.uint8, device="cuda")

    def call():
        tok = torch.full((rows,), -7, dtype=torch.int32, device="cuda")
        hid = torch.zeros((rows, d), dtype=torch.float32, device="cuda")
        st = torch.zeros(1, dtype=torch.int32, device="cuda")
        ssd.ssd_draft_predict(rows, d, m, V, dev["z"], dev["w0"], dev["w1"], dev["w3"],
                              dev["w2"], torch.from_numpy(g1).cuda(), torch.from_numpy(g2).cuda(),
                              dev["wh"], 1e-6, tok, hid, ws, wsb, st)
        torch.cuda.synchronize()
        return tok.cpu().numpy(), hid.cpu().numpy(), int(st.item())

    ssd.ssd_set_wait_limit(1 << 12)
    ssd.ssd_set_barrier_shortfall(1)
    try:
        tok, _, st = call()
    finally:
        ssd.ssd_set_barrier_shortfall(0)
        ssd.ssd_set_wait_limit(0)
    assert st == SSD_ERR_TIMEOUT
    assert np.all(tok == -7)  # the products after the first never ran: no tokens
    torch.cuda.synchronize()
    tok, hid, st = call()
    assert st == 0
    _check(w, g1, g2, 1e-6, tok, hid)
