"""GPU replay of the whole decoding schedule of one image (Sec. 3.3; Sec. 4
"SSD Configuration"; App. "Multi-Row Anticipation Ablations") against the
oracle's replay, step by step with device state driving every frontier: the
horizontal stage on the first row, then r rounds per row (k_v = 1) or the
staged b / i schedule on two rows (k_v = 2), each group closed by commit
passes.  Kinds, cache lengths, accept flags and tokens of every step must be
equal until the replays first differ, which may only happen on near-tie
rows (after that the trajectories may part); a replay with no difference
ends with the same cache, and the step count is the oracle's, which is the
paper's formula plus the horizontal stage."""
import numpy as np
import pytest
import torch

import synth
from oracle import schedule as sch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ssd():
    import paper_2606_20543_gb300 as m
    from paper_2606_20543_gb300 import build
    build.build()
    m.load()
    return m


def _pool(D_max, V, seed):
    out = []
    for k in range(3):
        rng = np.random.default_rng(seed * 10 + k)
        tg, dr = synth._logits_zipf(rng, D_max + 1, V) if k % 2 else synth._logits_normal(
            rng, D_max + 1, V)
        out.append((tg.astype(np.float32), dr.astype(np.float32)))
    return out


@pytest.mark.parametrize("k_v,b,i,seed", [(1, 2, 0, 1), (2, 2, 1, 2), (2, 3, 2, 3)])
def test_schedule_replay_matches_oracle(ssd, k_v, b, i, seed):
    from paper_2606_20543_gb300.step import VerifySchedule, VerifyStep
    H = W = 16
    prefix, V = 32, 4096
    D_max = 2 * W
    c = synth.make_case("sched", grid_h=H, grid_w=W, prefix_len=prefix, cache_len=[prefix],
                        Hq=8, Hkv=8, d=64, V=V, seed=seed, k_v=1, with_logits=False)
    pool = _pool(D_max, V, seed)

    def o_inputs(t):
        tg, dr = pool[t % 3]
        return tg, dr, synth.philox_uniforms(seed, t, D_max + 1)

    o_steps, o_grid, o_hist = sch.replay(H, W, prefix, 5, k_v, b, i, D_max, o_inputs)

    s = VerifyStep(H, W, prefix, 1, c.Hq, c.Hkv, c.d, D_max, c.L_max, V, k_v=1)
    s.upload(cache_len=c.cache_len, q=c.q, k=c.k, v=c.v)
    dpool = [(torch.from_numpy(tg).cuda(), torch.from_numpy(dr).cuda()) for tg, dr in pool]
    sched = VerifySchedule(s, k_h=5, k_v=k_v, b=b, i=i)
    g_hist = []

    def on_step(t, kind, info):
        rec = dict(kind=kind, step=t, cache_len=info["cache_len"])
        if kind == "horizontal":
            n = int(s.n_drafts[0].item())
            nxt = int(s.next_cache_len[0].item())
            tok = s.out_tok.cpu().numpy()
            adv = nxt - info["cache_len"]
            rec.update(n_drafts=n, accepted=s.accepted.cpu().numpy()[:n].astype(bool),
                       tokens=np.concatenate([tok[:min(adv, n)], tok[n:n + 1] if adv > n else []]))
        elif kind == "round":
            n = int(s.n_drafts[0].item())
            rec.update(n_drafts=n, accepted=s.accepted.cpu().numpy()[:n].astype(bool),
                       tokens=info["tokens"].cpu().numpy()[:n])
        g_hist.append(rec)

    g_steps = sched.run(lambda t: dpool[t % 3], seed=seed, on_step=on_step)
    torch.cuda.synchronize()
    assert s.status.item() == 0

    # compare step by step until the two replays differ; a difference is excused
    # only on near-tie rows (after it the trajectories may part)
    parted = False
    compared = 0
    for o, g in zip(o_hist, g_hist):
        compared += 1
        assert (o["kind"], o["step"], o["cache_len"]) == (g["kind"], g["step"], g["cache_len"])
        if o["kind"] == "commit":
            continue
        assert o["n_drafts"] == g["n_drafts"], o["step"]
        bad_acc = o["accepted"] != g["accepted"]
        if o["kind"] == "round":
            bad = bad_acc | (np.asarray(o["tokens"]) != g["tokens"].astype(np.int64))
            if bad.any():
                assert o["tie_rows"][bad].all(), (o["step"], np.nonzero(bad & ~o["tie_rows"]))
                parted = True
                break
        else:  # horizontal: the committed tokens (drafts, first rejection's draw, bonus)
            same_tok = np.array_equal(np.asarray(o["tokens"]), g["tokens"].astype(np.int64))
            if bad_acc.any() or not same_tok:
                assert o["ties"] > 0, o["step"]
                assert not bad_acc.any() or o["tie_rows"][bad_acc].all(), o["step"]
                parted = True
                break
    print(f"schedule k_v={k_v} b={b} i={i}: {compared} of {o_steps} steps compared, "
          f"{'parted at a near-tie' if parted else 'identical'}")
    if not parted:
        assert compared == len(o_hist) == len(g_hist) == g_steps == o_steps
        assert int(s.cache_len[0].item()) == prefix + H * W
        s_h = sum(h["kind"] == "horizontal" for h in o_hist)
        assert o_steps == s_h + sch.vertical_steps(H, k_v, b, i)
