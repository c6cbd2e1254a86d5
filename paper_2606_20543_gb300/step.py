"""Device buffers for one verification problem shape and the calls that run
it through ``ssd_verify_step`` — the public API a caller uses end to end.

Marshalling only: host arrays (numpy or torch, pinned or not) are copied to
preallocated device tensors, the C-ABI entry point runs every step of the
pass, and results are copied back on request.
"""
from __future__ import annotations

import numpy as np
import torch

from . import (COMMITS, STRATEGIES, Grid, Rng, VerifyArgs, VerifyOut, grid as make_grid,
               row_addresses, ssd_commit_pass, ssd_frontier, ssd_record_commit, ssd_stage_shift,
               ssd_verify_attention, ssd_verify_attention_workspace, ssd_verify_step,
               ssd_verify_step_workspace)


def _dev(shape, dtype, device):
    return torch.empty(shape, dtype=dtype, device=device)


def _as_torch(x, dtype):
    if isinstance(x, torch.Tensor):
        return x
    x = np.ascontiguousarray(x)
    if dtype == torch.bfloat16:
        return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16)
    return torch.from_numpy(x)


class ReplayState:
    """The state of a replay of one batch between two steps: the index of the
    next step (its Philox counter offset), the seed, every sequence's cache
    length and its committed grid tokens (raster order, -1 where nothing is
    committed yet).  With the step's inputs a function of the step index, this
    is all a replay needs to resume.  ``save`` / ``load`` use one .npz file."""

    def __init__(self, step: int, seed: int, cache_len, grid_tok):
        self.step, self.seed = int(step), int(seed)
        self.cache_len = np.asarray(cache_len, np.int32)
        self.grid_tok = np.asarray(grid_tok, np.int32)

    def save(self, path) -> None:
        np.savez(path, step=self.step, seed=self.seed, cache_len=self.cache_len,
                 grid_tok=self.grid_tok)

    @classmethod
    def load(cls, path) -> "ReplayState":
        z = np.load(path)
        return cls(int(z["step"]), int(z["seed"]), z["cache_len"], z["grid_tok"])


class VerifyStep:
    """Preallocated inputs, outputs and workspace for ssd_verify_step.

    Shapes follow include/ssd.h: q [B, D_max, Hq, d], k/v [B, Hkv, L_max, d]
    (bf16), logits [B*D_max, V] (float32) or hidden [B*D_max, hidden] with
    lm_head weights [hidden, V] (bf16).

    Under strategy (C) with commit "prefix" or "prefix_bonus" a step draws only
    the tokens it commits: out_tok holds the draft token of each accepted row,
    the residual token of each sequence's first rejection and the bonus token
    when every draft is accepted; the other rejected rows (discarded by the
    prefix rule) hold -1.  accepted and ratio are written for every row."""

    def __init__(self, grid_h, grid_w, prefix_len, B, Hq, Hkv, d, D_max, L_max, V,
                 hidden=0, k_v=1, row_stride=None, device="cuda", scale=0.0, temperature=1.0,
                 strategy="accept_reject", k_h=0, commit="prefix"):
        self.g: Grid = make_grid(grid_h, grid_w, prefix_len, row_stride, k_v, k_h)
        self.B, self.Hq, self.Hkv, self.d = B, Hq, Hkv, d
        self.D_max, self.L_max, self.V, self.hidden = D_max, L_max, V, hidden
        self.device = device
        self.scale, self.temperature = scale, temperature
        self.strategy = STRATEGIES.get(strategy, strategy)
        self.commit = COMMITS.get(commit, commit)
        rows = B * D_max
        self.rows = rows
        dv = device
        self.cache_len = _dev((B,), torch.int32, dv)
        self.q = _dev((B, D_max, Hq, d), torch.bfloat16, dv)
        self.k = _dev((B, Hkv, L_max, d), torch.bfloat16, dv)
        self.v = _dev((B, Hkv, L_max, d), torch.bfloat16, dv)
        if hidden:
            self.tgt = self.drf = None
            self.h_tgt = _dev((rows, hidden), torch.bfloat16, dv)
            self.h_drf = _dev((rows, hidden), torch.bfloat16, dv)
            self.w_tgt = _dev((hidden, V), torch.bfloat16, dv)
            self.w_drf = _dev((hidden, V), torch.bfloat16, dv)
        else:
            self.tgt = _dev((rows, V), torch.float32, dv)
            self.drf = _dev((rows, V), torch.float32, dv)
            self.h_tgt = self.h_drf = self.w_tgt = self.w_drf = None
        self.uniforms = None
        self.draft_tok = None
        # outputs
        self.n_drafts = _dev((B,), torch.int32, dv)
        self.draft_pos = _dev((B, D_max), torch.int32, dv)
        self.o = torch.zeros((B, D_max, Hq, d), dtype=torch.bfloat16, device=dv)
        self.lse = _dev((B, Hq, D_max), torch.float32, dv)
        self.out_tok = _dev((rows,), torch.int32, dv)
        self.accepted = _dev((rows,), torch.uint8, dv)
        self.ratio = _dev((rows,), torch.float32, dv)
        self.accepted_count = _dev((B,), torch.int32, dv)
        self.accepted_prefix = _dev((B,), torch.int32, dv)
        self.next_cache_len = _dev((B,), torch.int32, dv)
        self.status = torch.zeros((1,), dtype=torch.int32, device=dv)
        self.rng = Rng(0, 0, None)
        self.args = self._args()
        self.ws_bytes = ssd_verify_step_workspace(self.args)
        self.workspace = _dev((max(self.ws_bytes, 256),), torch.uint8, dv)
        self.out = self._out()

    # ------------------------------------------------------------------ args
    def _args(self) -> VerifyArgs:
        a = VerifyArgs()
        a.grid = self.g
        a.B, a.Hq, a.Hkv, a.d = self.B, self.Hq, self.Hkv, self.d
        a.D_max, a.L_max, a.V = self.D_max, self.L_max, self.V
        a.cache_len = self.cache_len.data_ptr()
        a.q, a.k, a.v = self.q.data_ptr(), self.k.data_ptr(), self.v.data_ptr()
        a.scale = self.scale
        if self.hidden:
            a.tgt_logits = a.drf_logits = None
            a.ld = 0
            a.h_tgt, a.h_drf = self.h_tgt.data_ptr(), self.h_drf.data_ptr()
            a.w_tgt, a.w_drf = self.w_tgt.data_ptr(), self.w_drf.data_ptr()
            a.hidden = self.hidden
        else:
            a.tgt_logits, a.drf_logits = self.tgt.data_ptr(), self.drf.data_ptr()
            a.ld = self.V
            a.h_tgt = a.h_drf = a.w_tgt = a.w_drf = None
            a.hidden = 0
        a.draft_tok = None if self.draft_tok is None else self.draft_tok.data_ptr()
        a.temperature = self.temperature
        a.rng = self.rng
        a.strategy = self.strategy
        a.commit = self.commit
        return a

    def _out(self) -> VerifyOut:
        y = VerifyOut()
        y.n_drafts, y.draft_pos = self.n_drafts.data_ptr(), self.draft_pos.data_ptr()
        y.o, y.lse = self.o.data_ptr(), self.lse.data_ptr()
        y.out_tok, y.accepted = self.out_tok.data_ptr(), self.accepted.data_ptr()
        y.ratio = self.ratio.data_ptr()
        y.accepted_count = self.accepted_count.data_ptr()
        y.accepted_prefix = self.accepted_prefix.data_ptr()
        y.next_cache_len = self.next_cache_len.data_ptr()
        y.status = self.status.data_ptr()
        return y

    # ----------------------------------------------------------------- inputs
    def upload(self, cache_len=None, q=None, k=None, v=None, tgt_logits=None, drf_logits=None,
               h_tgt=None, h_drf=None, w_tgt=None, w_drf=None, uniforms=None, draft_tok=None,
               non_blocking=False):
        """Copy host arrays into the device buffers (bf16 given as uint16 bits
        or torch.bfloat16).  Arguments left None keep their current contents."""
        pairs = [(cache_len, self.cache_len, torch.int32), (q, self.q, torch.bfloat16),
                 (k, self.k, torch.bfloat16), (v, self.v, torch.bfloat16),
                 (tgt_logits, self.tgt, torch.float32), (drf_logits, self.drf, torch.float32),
                 (h_tgt, self.h_tgt, torch.bfloat16), (h_drf, self.h_drf, torch.bfloat16),
                 (w_tgt, self.w_tgt, torch.bfloat16), (w_drf, self.w_drf, torch.bfloat16)]
        for src, dst, dt in pairs:
            if src is not None:
                dst.copy_(_as_torch(src, dt).reshape(dst.shape), non_blocking=non_blocking)
        if uniforms is not None:
            if self.uniforms is None:
                self.uniforms = _dev((self.rows, 2), torch.float32, self.device)
            self.uniforms.copy_(_as_torch(uniforms, torch.float32).reshape(self.rows, 2),
                                non_blocking=non_blocking)
            self.rng.uniforms = self.uniforms.data_ptr()
        if draft_tok is not None:
            self.draft_tok = _dev((self.rows,), torch.int32, self.device)
            self.draft_tok.copy_(_as_torch(draft_tok, torch.int32).reshape(-1))
            self.args = self._args()
        self.args.rng = self.rng

    def set_rng(self, seed: int, offset: int, use_uniforms: bool = False):
        self.rng.seed, self.rng.offset = seed, offset
        if not use_uniforms:
            self.rng.uniforms = None
        self.args.rng = self.rng

    # -------------------------------------------------------------------- run
    def run(self, stream=None) -> None:
        ssd_verify_step(self.args, self.out, self.workspace, self.ws_bytes, stream)

    def use_cache_buffers(self, cache_len, next_cache_len) -> None:
        """Read the step's cache lengths from `cache_len` and write the next
        ones to `next_cache_len` (two distinct device int32 [B] tensors).
        Alternating two buffers chains steps with no copy of next_cache_len
        back into cache_len between them (step t reads buffer t % 2)."""
        if cache_len.data_ptr() == next_cache_len.data_ptr():
            raise ValueError("cache_len and next_cache_len must be distinct buffers")
        self.cache_len, self.next_cache_len = cache_len, next_cache_len
        self.args.cache_len = cache_len.data_ptr()
        self.out.next_cache_len = next_cache_len.data_ptr()

    # ------------------------------------------------------- replay bookkeeping
    def track_grid(self) -> None:
        """Allocate the committed-token grid [B, H*W] (-1: not committed) that
        advance() fills, for a replay that is to be dumped or resumed."""
        hw = self.g.grid_h * self.g.grid_w
        self.grid_tok = torch.full((self.B, hw), -1, dtype=torch.int32, device=self.device)

    def advance(self, stream=None) -> None:
        """After run(): write the step's committed tokens into grid_tok (if
        tracked) and make next_cache_len the next step's cache length."""
        if getattr(self, "grid_tok", None) is not None:
            ssd_record_commit(self.B, self.D_max, self.g.prefix_len, self.grid_tok.shape[1],
                              self.cache_len, self.next_cache_len, self.out_tok, self.grid_tok,
                              self.status, stream)
        self.cache_len.copy_(self.next_cache_len)

    def state(self, step: int, seed: int) -> ReplayState:
        """The replay's state before step `step` (copied to the host)."""
        return ReplayState(step, seed, self.cache_len.cpu().numpy(),
                           self.grid_tok.cpu().numpy())

    def restore(self, st: ReplayState) -> int:
        """Load a dumped state; returns the step to run next."""
        if getattr(self, "grid_tok", None) is None:
            self.track_grid()
        self.cache_len.copy_(torch.from_numpy(st.cache_len.astype(np.int32)))
        self.grid_tok.copy_(torch.from_numpy(st.grid_tok.astype(np.int32)))
        return st.step

    def results(self) -> dict:
        names = ["n_drafts", "draft_pos", "out_tok", "accepted", "ratio", "accepted_count",
                 "accepted_prefix", "next_cache_len", "status"]
        r = {n: getattr(self, n).cpu().numpy() for n in names}
        r["o"] = self.o.float().cpu().numpy()
        r["lse"] = self.lse.cpu().numpy()
        return r


class VerifyRounds:
    """r verify-and-correct rounds (Sec. 3.3) and the staged b / i schedule
    (App. multi-row drafting) over the buffers of a VerifyStep.

    Every round is one ssd_verify_step with the round's target logits, the
    rows' current reference pointers (ref_rows, redirected by the library to
    the round's target row when a row is not accepted) and the tokens the
    previous round left (two device buffers used in turn).  The caller keeps
    each round's target logits alive and unchanged until the block is
    committed: later rounds read them as references."""

    def __init__(self, step: "VerifyStep"):
        if step.hidden:
            raise ValueError("verify-and-correct rounds need the logits path")
        self.s = step
        self.ref_rows = row_addresses(step.drf)
        self.tok = [_dev((step.rows,), torch.int32, step.device) for _ in range(2)]
        self.cur = 0

    def reset(self):
        """Back to round 1 (which rewrites every reference itself)."""
        self.cur = 0

    @property
    def tokens(self):
        """Device tensor of the tokens after the last round run."""
        return self.tok[self.cur]

    def run(self, tgt_rounds, commit_last="block", uniforms_rounds=None, seed=0, offset0=0,
            first_round=True, stream=None) -> None:
        """One round per entry of tgt_rounds (device float32 [rows, V]): the
        rounds before the last commit nothing, the last commits per
        commit_last (an ssd_commit name).  Round 1 (first_round) verifies the
        draft tokens (argmax of the draft rows); later rounds the tokens the
        previous round left.  Each round draws its uniforms from Philox at
        offset offset0 + round, or from uniforms_rounds[round] if given."""
        s = self.s
        a, y = s.args, s.out
        n = len(tgt_rounds)
        for rho, tgt in enumerate(tgt_rounds):
            a.tgt_logits = tgt.data_ptr()
            a.ld = s.V
            a.ref_rows = self.ref_rows.data_ptr()
            a.ref_init = 1 if (first_round and rho == 0) else 0
            a.draft_tok = None if (first_round and rho == 0) else self.tok[self.cur].data_ptr()
            y.out_tok = self.tok[1 - self.cur].data_ptr()
            a.commit = COMMITS["none"] if rho < n - 1 else COMMITS[commit_last]
            s.rng.seed, s.rng.offset = seed, offset0 + rho
            s.rng.uniforms = None if uniforms_rounds is None else uniforms_rounds[rho].data_ptr()
            a.rng = s.rng
            ssd_verify_step(a, y, s.workspace, s.ws_bytes, stream)
            self.cur = 1 - self.cur
        # leave the VerifyStep as it was for plain steps
        a.tgt_logits, a.ref_rows, a.commit, a.ref_init = s.tgt.data_ptr(), None, s.commit, 0
        a.draft_tok = None if s.draft_tok is None else s.draft_tok.data_ptr()
        y.out_tok = s.out_tok.data_ptr()

    def run_staged(self, b, i, tgt_rounds, uniforms_rounds=None, seed=0, offset0=0,
                   stream=None) -> None:
        """The staged schedule of the paper's two-row vertical stage: from a
        row start the frontier with k_v = 1 is the two drafted rows (the
        current row and the row below).  b base rounds on both, commit the
        first row, move the trailing row to the front (ssd_stage_shift),
        advance the cache, then i rounds on the trailing row alone (k_v = 0)
        and commit it."""
        s = self.s
        if s.g.k_v != 1:
            raise ValueError("the staged schedule verifies a two-row frontier (k_v = 1)")
        W = s.g.grid_w
        u = uniforms_rounds
        self.run(tgt_rounds[:b], "first_row", None if u is None else u[:b], seed, offset0,
                 True, stream)
        ssd_stage_shift(s.B, s.D_max, W, self.tok[self.cur], self.ref_rows, stream)
        s.cache_len.copy_(s.next_cache_len)
        s.args.grid.k_v = 0
        try:
            self.run(tgt_rounds[b:], "block", None if u is None else u[b:], seed, offset0 + b,
                     False, stream)
        finally:
            s.args.grid.k_v = 1


class VerifySchedule:
    """The whole decoding schedule of one image (batch 1) over the buffers of
    a VerifyStep: Sec. 3.3 (horizontal heads until the first row is complete,
    then k_v rows drafted below at a time, verified and corrected), Sec. 4
    "SSD Configuration" (5 horizontal drafts with one round; r rounds for one
    vertical row, or staged b / i rounds for two) and App. "Multi-Row
    Anticipation Ablations" (b base rounds on both rows, commit the first row,
    i rounds on the trailing row, commit it).

    Every verification round is one ssd_verify_step; every commit pass is the
    frontier, its attention (ssd_verify_attention) and ssd_commit_pass.  Each
    is one step, a backbone forward pass in the paper's count.  The horizontal
    stage runs on the first row alone (a one-row grid, so that its bonus
    token stays in that row); the device cache length drives every frontier,
    and the host reads it after each step to know where the schedule is.

    step_inputs(t) gives step t's target and draft logits (device float32
    [>= D_max + 1, V]); the uniforms of step t are Philox(seed, t).  They
    must stay alive and unchanged for the whole run: later rounds read earlier
    rounds' rows as references."""

    def __init__(self, step: VerifyStep, k_h=5, k_v=1, b=2, i=0):
        if step.B != 1:
            raise ValueError("the schedule replays one image (batch 1)")
        if k_v not in (1, 2) or b < 1 or i < 0 or k_h < 1:
            raise ValueError("k_v in {1, 2}, b >= 1, i >= 0, k_h >= 1")
        W = step.g.grid_w
        if step.D_max < k_v * W or step.D_max < k_h + 1:
            raise ValueError("D_max must hold k_v rows and the horizontal bonus row")
        self.s, self.k_h, self.k_v, self.b, self.i = step, k_h, k_v, b, i
        self.rounds = VerifyRounds(step)
        self.att_ws_bytes = ssd_verify_attention_workspace(step.B, step.Hq, step.Hkv, step.d,
                                                           step.D_max, step.L_max)
        self.att_ws = _dev((max(self.att_ws_bytes, 256),), torch.uint8, step.device)

    def _grid(self, grid_h, k_h, k_v) -> Grid:
        g0 = self.s.g
        return make_grid(grid_h, g0.grid_w, g0.prefix_len, g0.row_stride, k_v, k_h)

    def _cache(self) -> int:
        return int(self.s.cache_len[0].item())

    def _commit_pass(self, g: Grid, mode: str, stream=None) -> None:
        s = self.s
        ssd_frontier(g, s.B, s.cache_len, s.D_max, s.n_drafts, s.draft_pos, s.status, stream)
        ssd_verify_attention(g, s.B, s.Hq, s.Hkv, s.d, s.cache_len, s.n_drafts, s.draft_pos,
                             s.D_max, s.L_max, s.q, s.k, s.v, s.scale, s.o, None, self.att_ws,
                             self.att_ws_bytes, s.status, stream)
        ssd_commit_pass(g, s.B, s.cache_len, s.D_max, mode, s.next_cache_len, s.status, stream)
        s.cache_len.copy_(s.next_cache_len)

    def run(self, step_inputs, seed=0, on_step=None, stream=None) -> int:
        """Replay to grid completion; returns the number of steps.
        on_step(t, kind, info) is called after each step (kind 'horizontal',
        'round' or 'commit'); info holds the host-side cache length before the
        step and, for rounds and horizontal steps, the device tensors of the
        decisions (valid until the next step)."""
        s = self.s
        a = s.args
        g0 = s.g
        H, W, prefix = g0.grid_h, g0.grid_w, g0.prefix_len
        saved = (a.grid, a.commit, a.strategy, a.ref_rows, a.ref_init, a.draft_tok,
                 a.tgt_logits, a.drf_logits)
        t = 0
        try:
            # ---- horizontal stage on the first row
            a.grid = self._grid(1, self.k_h, 0)
            a.commit = COMMITS["prefix_bonus"]
            a.ref_rows, a.ref_init, a.draft_tok = None, 0, None
            cache = self._cache()
            while cache - prefix < W:
                tg, dr = step_inputs(t)
                a.tgt_logits, a.drf_logits = tg.data_ptr(), dr.data_ptr()
                s.set_rng(seed, t)
                ssd_verify_step(a, s.out, s.workspace, s.ws_bytes, stream)
                if on_step is not None:
                    on_step(t, "horizontal", dict(cache_len=cache))
                s.cache_len.copy_(s.next_cache_len)
                cache = self._cache()
                t += 1
            # ---- vertical stage
            while cache - prefix < H * W:
                y0 = (cache - prefix) // W
                k = min(self.k_v, H - y0)
                g = self._grid(H, 0, k - 1)
                a.grid = g
                tg0, dr0 = step_inputs(t)
                a.drf_logits = dr0.data_ptr()
                self.rounds.reset()
                tgts = [step_inputs(t + r)[0] for r in range(self.b)]
                self._rounds(tgts, t, seed, True, on_step, cache, stream)
                t += self.b
                self._commit_pass(g, "first_row" if k > 1 else "block", stream)
                if on_step is not None:
                    on_step(t, "commit", dict(cache_len=cache))
                cache = self._cache()
                t += 1
                if k > 1:  # the trailing row: its slots move to the front
                    ssd_stage_shift(s.B, s.D_max, W, self.rounds.tokens, self.rounds.ref_rows,
                                    stream)
                    g1 = self._grid(H, 0, 0)
                    a.grid = g1
                    tgts = [step_inputs(t + r)[0] for r in range(self.i)]
                    self._rounds(tgts, t, seed, False, on_step, cache, stream)
                    t += self.i
                    self._commit_pass(g1, "block", stream)
                    if on_step is not None:
                        on_step(t, "commit", dict(cache_len=cache))
                    cache = self._cache()
                    t += 1
        finally:
            (a.grid, a.commit, a.strategy, a.ref_rows, a.ref_init, a.draft_tok, a.tgt_logits,
             a.drf_logits) = saved
        return t

    def _rounds(self, tgts, t0, seed, first_round, on_step, cache, stream):
        """Rounds t0, t0 + 1, ... of the current frontier, one at a time so
        that on_step sees each; nothing is committed."""
        for r, tg in enumerate(tgts):
            self.rounds.run([tg], "none", None, seed, t0 + r, first_round and r == 0, stream)
            if on_step is not None:
                on_step(t0 + r, "round", dict(cache_len=cache, tokens=self.rounds.tokens))
