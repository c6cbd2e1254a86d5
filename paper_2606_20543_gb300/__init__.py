"""Python binding of libssd, the GB300 (sm_103a) verification pass of
Spatially Speculative Decoding.

Argument marshalling only: every function here forwards to the entry point
of the same name in ``include/ssd.h``; every step of the pass runs in the
library's CUDA kernels.  Device buffers are torch CUDA tensors (PyTorch is
used for device memory and streams only).  There is no CPU path: if the
library has not been built, importing a function raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libssd.so")
DEBUG_LIB_PATH = os.path.join(HERE, "libssd_debug.so")

SSD_OK = 0
STATUS_NAMES = {0: "SSD_OK", 1: "SSD_ERR_INVALID_ARG", 2: "SSD_ERR_SHAPE", 3: "SSD_ERR_UNSUPPORTED",
                4: "SSD_ERR_CUDA", 5: "SSD_ERR_TIMEOUT", 6: "SSD_ERR_DEVICE_BOUNDS",
                7: "SSD_ERR_WORKSPACE"}

EXPORTED = ["ssd_abi_version", "ssd_status_string", "ssd_set_wait_limit",
            "ssd_set_barrier_shortfall", "ssd_frontier", "ssd_verify_attention_workspace",
            "ssd_verify_attention", "ssd_verify_attention_noalloc", "ssd_accept", "ssd_accept_strategy",
            "ssd_accept_round", "ssd_stage_shift", "ssd_commit_pass", "ssd_record_commit",
            "ssd_draft_predict_workspace",
            "ssd_draft_predict",
            "ssd_lmhead_accept_workspace", "ssd_lmhead_accept",
            "ssd_verify_step_workspace", "ssd_verify_step_launches", "ssd_verify_step",
            "ssd_verify_accept"]


STRATEGY_ACCEPT_REJECT, STRATEGY_GREEDY, STRATEGY_SAMPLE = 0, 1, 2
COMMIT_PREFIX, COMMIT_NONE, COMMIT_BLOCK, COMMIT_FIRST_ROW, COMMIT_PREFIX_BONUS = 0, 1, 2, 3, 4
COMMITS = {"prefix": COMMIT_PREFIX, "none": COMMIT_NONE, "block": COMMIT_BLOCK,
           "first_row": COMMIT_FIRST_ROW, "prefix_bonus": COMMIT_PREFIX_BONUS}
STRATEGIES = {"accept_reject": STRATEGY_ACCEPT_REJECT, "greedy": STRATEGY_GREEDY,
              "sample": STRATEGY_SAMPLE}


class SsdError(RuntimeError):
    def __init__(self, fn: str, code: int):
        super().__init__(f"{fn} returned {STATUS_NAMES.get(code, code)}")
        self.code = code


class Grid(ctypes.Structure):
    _fields_ = [("grid_h", ctypes.c_int32), ("grid_w", ctypes.c_int32),
                ("row_stride", ctypes.c_int32), ("prefix_len", ctypes.c_int32),
                ("k_v", ctypes.c_int32), ("k_h", ctypes.c_int32)]


class Rng(ctypes.Structure):
    _fields_ = [("seed", ctypes.c_uint64), ("offset", ctypes.c_uint64),
                ("uniforms", ctypes.c_void_p)]


class VerifyArgs(ctypes.Structure):
    _fields_ = [("grid", Grid),
                ("B", ctypes.c_int32), ("Hq", ctypes.c_int32), ("Hkv", ctypes.c_int32),
                ("d", ctypes.c_int32), ("D_max", ctypes.c_int32), ("L_max", ctypes.c_int32),
                ("V", ctypes.c_int32),
                ("cache_len", ctypes.c_void_p), ("q", ctypes.c_void_p), ("k", ctypes.c_void_p),
                ("v", ctypes.c_void_p), ("scale", ctypes.c_float),
                ("tgt_logits", ctypes.c_void_p), ("drf_logits", ctypes.c_void_p),
                ("ld", ctypes.c_int64),
                ("h_tgt", ctypes.c_void_p), ("h_drf", ctypes.c_void_p),
                ("w_tgt", ctypes.c_void_p), ("w_drf", ctypes.c_void_p),
                ("hidden", ctypes.c_int32),
                ("draft_tok", ctypes.c_void_p), ("temperature", ctypes.c_float),
                ("rng", Rng), ("strategy", ctypes.c_int32), ("ref_rows", ctypes.c_void_p),
                ("ref_init", ctypes.c_int32), ("commit", ctypes.c_int32)]


class VerifyOut(ctypes.Structure):
    _fields_ = [("n_drafts", ctypes.c_void_p), ("draft_pos", ctypes.c_void_p),
                ("o", ctypes.c_void_p), ("lse", ctypes.c_void_p),
                ("out_tok", ctypes.c_void_p), ("accepted", ctypes.c_void_p),
                ("ratio", ctypes.c_void_p), ("accepted_count", ctypes.c_void_p),
                ("accepted_prefix", ctypes.c_void_p), ("next_cache_len", ctypes.c_void_p),
                ("status", ctypes.c_void_p)]


_LIB: Optional[ctypes.CDLL] = None


def load(path: Optional[str] = None) -> ctypes.CDLL:
    """Load libssd.so (built by ``paper_2606_20543_gb300.build``); raise if
    absent.  With SSD_LIBRARY=debug in the environment the default is the
    bounds-checking build libssd_debug.so (``build --debug-bounds``)."""
    global _LIB
    if _LIB is not None:
        return _LIB
    if path is None:
        path = DEBUG_LIB_PATH if os.environ.get("SSD_LIBRARY") == "debug" else LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"libssd.so not built ({path} missing): run "
                           "`python -m paper_2606_20543_gb300.build` (needs nvcc)")
    lib = ctypes.CDLL(path)
    P, I32, I64, F, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_float, ctypes.c_size_t
    sig = {
        "ssd_abi_version": (I32, []),
        "ssd_status_string": (ctypes.c_char_p, [I32]),
        "ssd_set_wait_limit": (None, [ctypes.c_uint32]),
        "ssd_set_barrier_shortfall": (None, [ctypes.c_uint32]),
        "ssd_frontier": (I32, [ctypes.POINTER(Grid), I32, P, I32, P, P, P, P]),
        "ssd_verify_attention_workspace": (SZ, [I32, I32, I32, I32, I32, I32]),
        "ssd_verify_attention": (I32, [ctypes.POINTER(Grid), I32, I32, I32, I32, P, P, P, I32, I32,
                                       P, P, P, F, P, P, P, SZ, P, P]),
        "ssd_verify_attention_noalloc": (I32, [ctypes.POINTER(Grid), I32, I32, I32, I32, P, P, P,
                                               I32, I32, P, P, P, F, P, P, P, P]),
        "ssd_accept": (I32, [I32, I32, P, P, I64, P, F, ctypes.POINTER(Rng), P, P, P, P, P, P]),
        "ssd_accept_strategy": (I32, [I32, I32, I32, P, P, I64, P, F, ctypes.POINTER(Rng), P, P, P,
                                      P, P, P]),
        "ssd_accept_round": (I32, [I32, I32, I32, P, I64, P, P, F, ctypes.POINTER(Rng), P, P, P, P,
                                   P, P]),
        "ssd_stage_shift": (I32, [I32, I32, I32, P, P, P]),
        "ssd_commit_pass": (I32, [ctypes.POINTER(Grid), I32, P, I32, I32, P, P, P]),
        "ssd_record_commit": (I32, [I32, I32, I32, I32, P, P, P, P, P, P]),
        "ssd_draft_predict_workspace": (SZ, [I32, I32, I32, I32]),
        "ssd_draft_predict": (I32, [I32, I32, I32, I32, P, P, P, P, P, P, P, P, F, P, P, P, SZ,
                                    P, P]),
        "ssd_lmhead_accept_workspace": (SZ, [I32, I32]),
        "ssd_lmhead_accept": (I32, [I32, I32, I32, P, P, P, P, P, F, ctypes.POINTER(Rng), P, P, P,
                                    P, P, SZ, P, P]),
        "ssd_verify_step_workspace": (SZ, [ctypes.POINTER(VerifyArgs)]),
        "ssd_verify_step_launches": (I32, [ctypes.POINTER(VerifyArgs)]),
        "ssd_verify_step": (I32, [ctypes.POINTER(VerifyArgs), ctypes.POINTER(VerifyOut), P, SZ, P]),
        "ssd_verify_accept": (I32, [ctypes.POINTER(VerifyArgs), ctypes.POINTER(VerifyOut), P, SZ, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _LIB = lib
    return lib


def _ptr(t) -> Optional[int]:
    """Device address of a torch tensor (None stays None)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libssd takes device (CUDA) tensors")
    return t.data_ptr()


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


def _check(fn: str, code: int) -> None:
    if code != SSD_OK:
        raise SsdError(fn, code)


def grid(grid_h: int, grid_w: int, prefix_len: int, row_stride: Optional[int] = None,
         k_v: int = 1, k_h: int = 0) -> Grid:
    return Grid(grid_h, grid_w, grid_w if row_stride is None else row_stride, prefix_len, k_v, k_h)


def rng(seed: int = 0, offset: int = 0, uniforms=None) -> Rng:
    return Rng(seed, offset, _ptr(uniforms))


def ssd_abi_version() -> int:
    return load().ssd_abi_version()


def ssd_set_wait_limit(max_polls: int) -> None:
    """Poll limit of the bounded device waits of later launches (0: default)."""
    load().ssd_set_wait_limit(int(max_polls))


def ssd_set_barrier_shortfall(arrivals: int) -> None:
    """Extra arrivals the fused lm_head's grid barriers wait for (0: off)."""
    load().ssd_set_barrier_shortfall(int(arrivals))


def ssd_status_string(code: int) -> str:
    return load().ssd_status_string(code).decode()


def ssd_frontier(g: Grid, B: int, cache_len, D_max: int, n_drafts, draft_pos, status,
                 stream=None) -> None:
    _check("ssd_frontier", load().ssd_frontier(ctypes.byref(g), B, _ptr(cache_len), D_max,
                                               _ptr(n_drafts), _ptr(draft_pos), _ptr(status),
                                               _stream(stream)))


def ssd_verify_attention_workspace(B, Hq, Hkv, d, D_max, L_max) -> int:
    return load().ssd_verify_attention_workspace(B, Hq, Hkv, d, D_max, L_max)


def ssd_verify_attention(g: Grid, B, Hq, Hkv, d, cache_len, n_drafts, draft_pos, D_max, L_max,
                         q, k, v, scale, o, lse, workspace, workspace_bytes, status,
                         stream=None) -> None:
    _check("ssd_verify_attention", load().ssd_verify_attention(
        ctypes.byref(g), B, Hq, Hkv, d, _ptr(cache_len), _ptr(n_drafts), _ptr(draft_pos), D_max,
        L_max, _ptr(q), _ptr(k), _ptr(v), scale, _ptr(o), _ptr(lse), _ptr(workspace),
        workspace_bytes, _ptr(status), _stream(stream)))


def ssd_verify_attention_noalloc(g: Grid, B, Hq, Hkv, d, cache_len, n_drafts, draft_pos, D_max,
                                 L_max, q, k, v, scale, o, lse, status, stream=None) -> None:
    """ssd_verify_attention() for callers that cannot allocate device memory:
    the library's own static device scratch replaces the workspace (limit
    SSD_NOALLOC_SCRATCH_BYTES = 64 MiB; calls that overlap on the GPU race on
    that scratch and must be serialised by the caller)."""
    _check("ssd_verify_attention_noalloc", load().ssd_verify_attention_noalloc(
        ctypes.byref(g), B, Hq, Hkv, d, _ptr(cache_len), _ptr(n_drafts), _ptr(draft_pos), D_max,
        L_max, _ptr(q), _ptr(k), _ptr(v), scale, _ptr(o), _ptr(lse), _ptr(status),
        _stream(stream)))


def ssd_accept(rows, V, tgt_logits, drf_logits, ld, draft_tok, temperature, r: Rng, out_tok,
               accepted, ratio, lse, status, stream=None) -> None:
    _check("ssd_accept", load().ssd_accept(
        rows, V, _ptr(tgt_logits), _ptr(drf_logits), ld, _ptr(draft_tok), temperature,
        ctypes.byref(r), _ptr(out_tok), _ptr(accepted), _ptr(ratio), _ptr(lse), _ptr(status),
        _stream(stream)))


def ssd_accept_strategy(strategy, rows, V, tgt_logits, drf_logits, ld, draft_tok, temperature,
                        r: Rng, out_tok, accepted, ratio, lse, status, stream=None) -> None:
    """ssd_accept() under one of the strategies of Sec. 3.3: STRATEGY_ACCEPT_REJECT
    (C), STRATEGY_GREEDY (A) or STRATEGY_SAMPLE (B); also accepts their names."""
    strategy = STRATEGIES.get(strategy, strategy)
    _check("ssd_accept_strategy", load().ssd_accept_strategy(
        strategy, rows, V, _ptr(tgt_logits), _ptr(drf_logits), ld, _ptr(draft_tok), temperature,
        ctypes.byref(r), _ptr(out_tok), _ptr(accepted), _ptr(ratio), _ptr(lse), _ptr(status),
        _stream(stream)))


def ssd_accept_round(strategy, rows, V, tgt_logits, ld, ref_rows, tok, temperature, r: Rng,
                     out_tok, accepted, ratio, lse, status, stream=None) -> None:
    """One verify-and-correct round: ref_rows is a device int64 tensor of row
    addresses (updated in place for rows the round does not accept)."""
    strategy = STRATEGIES.get(strategy, strategy)
    _check("ssd_accept_round", load().ssd_accept_round(
        strategy, rows, V, _ptr(tgt_logits), ld, _ptr(ref_rows), _ptr(tok), temperature,
        ctypes.byref(r), _ptr(out_tok), _ptr(accepted), _ptr(ratio), _ptr(lse), _ptr(status),
        _stream(stream)))


def ssd_commit_pass(g: Grid, B, cache_len, D_max, commit, next_cache_len, status,
                    stream=None) -> None:
    c = COMMITS.get(commit, commit)
    _check("ssd_commit_pass", load().ssd_commit_pass(ctypes.byref(g), B, _ptr(cache_len), D_max,
                                                     c, _ptr(next_cache_len), _ptr(status),
                                                     _stream(stream)))


def ssd_stage_shift(B, D_max, W, tok, ref_rows, stream=None) -> None:
    _check("ssd_stage_shift", load().ssd_stage_shift(B, D_max, W, _ptr(tok), _ptr(ref_rows),
                                                     _stream(stream)))


def ssd_record_commit(B, D_max, prefix_len, hw, cache_len, next_cache_len, out_tok, grid_tok,
                      status, stream=None) -> None:
    _check("ssd_record_commit",
           load().ssd_record_commit(B, D_max, prefix_len, hw, _ptr(cache_len),
                                    _ptr(next_cache_len), _ptr(out_tok), _ptr(grid_tok),
                                    _ptr(status), _stream(stream)))


def ssd_draft_predict_workspace(rows, d, m, V) -> int:
    return load().ssd_draft_predict_workspace(rows, d, m, V)


def ssd_draft_predict(rows, d, m, V, z, w0, w1, w3, w2, gamma1, gamma2, w_head, eps, out_tok,
                      out_hidden, workspace, workspace_bytes, status, stream=None) -> None:
    """Eq. 2's spatial draft predictor and argmax GenHead(RMSNorm(h_hat))."""
    _check("ssd_draft_predict", load().ssd_draft_predict(
        rows, d, m, V, _ptr(z), _ptr(w0), _ptr(w1), _ptr(w3), _ptr(w2), _ptr(gamma1),
        _ptr(gamma2), _ptr(w_head), eps, _ptr(out_tok), _ptr(out_hidden), _ptr(workspace),
        workspace_bytes, _ptr(status), _stream(stream)))


def row_addresses(t, ld=None):
    """Device int64 tensor of the addresses of the rows of a 2D float32 tensor
    (the reference pointers of round 1)."""
    import torch
    ld = t.shape[1] if ld is None else ld
    return t.data_ptr() + torch.arange(t.shape[0], device=t.device, dtype=torch.int64) * (ld * 4)


def ssd_lmhead_accept_workspace(rows, V) -> int:
    return load().ssd_lmhead_accept_workspace(rows, V)


def ssd_lmhead_accept(rows, V, K, h_tgt, h_drf, w_tgt, w_drf, draft_tok, temperature, r: Rng,
                      out_tok, accepted, ratio, lse, workspace, workspace_bytes, status,
                      stream=None) -> None:
    _check("ssd_lmhead_accept", load().ssd_lmhead_accept(
        rows, V, K, _ptr(h_tgt), _ptr(h_drf), _ptr(w_tgt), _ptr(w_drf), _ptr(draft_tok),
        temperature, ctypes.byref(r), _ptr(out_tok), _ptr(accepted), _ptr(ratio), _ptr(lse),
        _ptr(workspace), workspace_bytes, _ptr(status), _stream(stream)))


def ssd_verify_step_workspace(args: VerifyArgs) -> int:
    return load().ssd_verify_step_workspace(ctypes.byref(args))


def ssd_verify_step_launches(args: VerifyArgs) -> int:
    return load().ssd_verify_step_launches(ctypes.byref(args))


def ssd_verify_step(args: VerifyArgs, out: VerifyOut, workspace, workspace_bytes,
                    stream=None) -> None:
    _check("ssd_verify_step", load().ssd_verify_step(
        ctypes.byref(args), ctypes.byref(out), _ptr(workspace), workspace_bytes, _stream(stream)))


def ssd_verify_accept(args: VerifyArgs, out: VerifyOut, workspace, workspace_bytes,
                      stream=None) -> None:
    _check("ssd_verify_accept", load().ssd_verify_accept(
        ctypes.byref(args), ctypes.byref(out), _ptr(workspace), workspace_bytes, _stream(stream)))
