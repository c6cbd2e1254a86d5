"""Failure detection on the GPU without a fault: a bounded device wait that
runs out.  The fused lm_head's CTAs meet at grid barriers; with
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
