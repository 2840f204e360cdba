"""Python binding of libeti, the sm_103a kernels of the entropic-time decode step.

Argument marshalling only: every function below checks tensor dtypes,
devices and shapes, then calls the C entry point of the same name in
``_build/libeti.so`` (declared in ``include/eti.h``) on the current CUDA
stream.  There is no Python or CPU implementation of any step: if the
library is missing or CUDA is unavailable, the calls raise.
"""
from __future__ import annotations

import ctypes
import math
import os
import threading

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libeti.so")
_lock = threading.Lock()
_lib = None

ETI_OK = 0
STATUS = {0: "ok", -1: "null pointer", -2: "bad shape", -3: "unsupported shape",
          -4: "workspace too small", -5: "CUDA launch failed", -6: "device wait gave up (reserved)",
          -7: "too large for the fixed scratch", -8: "misaligned tensor"}
ERRF_BAD_PAGE, ERRF_BAD_CTX, ERRF_NONFINITE, ERRF_ALL_NEG_INF, ERRF_BAD_TEMP = 1, 2, 4, 8, 16
ERRF_TIMEOUT, ERRF_DRAIN = 32, 64

# C-ABI symbols declared in include/eti.h
SYMBOLS = ("eti_ctrl_defaults", "eti_entropy_temp_sample", "eti_entropy_temp_sample_workspace_size",
           "eti_score_prune_workspace_size",
           "eti_score_prune_blocks", "eti_score_blocks", "eti_prune_blocks",
           "eti_paged_decode_workspace_size", "eti_paged_decode", "eti_version",
           "eti_status_string", "eti_entropy_temp_sample_noalloc",
           "eti_entropy_temp_sample_noalloc_max_bytes", "eti_topk_entropy", "eti_sched_defaults",
           "eti_schedule", "eti_set_wait_limit")


class EtiError(RuntimeError):
    pass


class CtrlParams(ctypes.Structure):
    """eti_ctrl_params (include/eti.h)."""
    _fields_ = [(n, ctypes.c_float) for n in
                ("eta", "sign", "T_min", "T_max", "eps_H", "H_min", "theta_user", "theta_hi",
                 "T_cal", "rho_T", "dtheta")]


def build(force: bool = False) -> str:
    from . import buildlib as _b
    return _b.build(force=force)


def load(path: str | None = None):
    """Load libeti.so and declare its signatures (raises if it is not built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise EtiError(f"libeti is not built ({p} missing); run __graft_entry__.build()")
        lib = ctypes.CDLL(p)
        P, i32, i64, u64, f32, sz = (ctypes.c_void_p, ctypes.c_int, ctypes.c_int64,
                                     ctypes.c_uint64, ctypes.c_float, ctypes.c_size_t)
        lib.eti_ctrl_defaults.argtypes = [P]
        lib.eti_ctrl_defaults.restype = None
        lib.eti_version.restype = ctypes.c_char_p
        lib.eti_status_string.argtypes = [i32]
        lib.eti_status_string.restype = ctypes.c_char_p
        lib.eti_entropy_temp_sample_workspace_size.argtypes = [i32, i32]
        lib.eti_entropy_temp_sample_workspace_size.restype = sz
        lib.eti_entropy_temp_sample.argtypes = [P, i32, i32, i64, P, P, P, P, P, u64, u64, P,
                                                P, P, P, P, P, P, P, P, P, sz, P]
        lib.eti_entropy_temp_sample_noalloc.argtypes = [P, i32, i32, i64, P, P, P, P, P, u64, u64, P,
                                                        P, P, P, P, P, P, P, P, P]
        lib.eti_set_wait_limit.argtypes = [i64]
        lib.eti_set_wait_limit.restype = i64
        lib.eti_entropy_temp_sample_noalloc.restype = i32
        lib.eti_entropy_temp_sample_noalloc_max_bytes.restype = sz
        lib.eti_entropy_temp_sample.restype = i32
        lib.eti_sched_defaults.argtypes = [P]
        lib.eti_sched_defaults.restype = None
        lib.eti_schedule.argtypes = [P, P, P, i32, i32, P, P, P, i32, i32, P, P, P]
        lib.eti_schedule.restype = i32
        lib.eti_topk_entropy.argtypes = [P, i32, i32, i64, P, i32, P, P, P, P, P]
        lib.eti_topk_entropy.restype = i32
        lib.eti_score_prune_workspace_size.argtypes = [i32] * 6
        lib.eti_score_prune_workspace_size.restype = sz
        lib.eti_score_prune_blocks.argtypes = ([P, P, P, P] + [i32] * 6 + [i64, f32, P, i32, i32, P]
                                               + [P] * 7 + [P, sz, P])
        lib.eti_score_prune_blocks.restype = i32
        lib.eti_score_blocks.argtypes = [P, P, P, P] + [i32] * 6 + [i64, f32, P, P, P, P]
        lib.eti_score_blocks.restype = i32
        lib.eti_prune_blocks.argtypes = [P, P, P] + [i32] * 6 + [i64, P, i32, i32] + [P] * 7
        lib.eti_prune_blocks.restype = i32
        lib.eti_paged_decode_workspace_size.argtypes = [i32] * 7
        lib.eti_paged_decode_workspace_size.restype = sz
        lib.eti_paged_decode.argtypes = ([P, P, P, P, P] + [i32] * 6 + [i64, f32]
                                         + [P] * 7 + [P, sz, P])
        lib.eti_paged_decode.restype = i32
        _lib = lib
    return _lib


def version() -> str:
    return load().eti_version().decode()


def set_wait_limit(polls: int) -> int:
    """Diagnostic: polls before a device-side tile wait gives up (< 0: the
    default); applies to later calls of this process.  Returns the previous
    limit (see eti_set_wait_limit in include/eti.h)."""
    return int(load().eti_set_wait_limit(int(polls)))


def ctrl_params(**kw) -> CtrlParams:
    """Controller parameters: the library defaults, overridden by keywords."""
    p = CtrlParams()
    load().eti_ctrl_defaults(ctypes.byref(p))
    for k, v in kw.items():
        setattr(p, k, float(v))
    return p


def _check(status: int, what: str):
    if status != ETI_OK:
        msg = load().eti_status_string(status).decode()
        raise EtiError(f"{what}: {msg} (status {status})")


def _dev(t: torch.Tensor | None, name: str, dtype=None, numel=None):
    if t is None:
        return None
    if not t.is_cuda:
        raise EtiError(f"{name} must be a CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise EtiError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise EtiError(f"{name} must be contiguous")
    if numel is not None and t.numel() < numel:
        raise EtiError(f"{name} has {t.numel()} elements, needs {numel}")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


# ---------------------------------------------------------------------------
def entropy_temp_sample_workspace_size(B: int, V: int) -> int:
    return int(load().eti_entropy_temp_sample_workspace_size(B, V))


class SurpStore(ctypes.Structure):
    """eti_surp_store (include/eti.h)."""
    _fields_ = [("store", ctypes.c_void_p), ("slot_mapping", ctypes.c_void_p),
                ("num_slots", ctypes.c_int64)]


def _surp_store(surp_store, slot_mapping, B):
    """(surp_store fp32 tensor, slot_mapping int64 [B]) -> SurpStore by reference, or None."""
    if surp_store is None and slot_mapping is None:
        return None
    if surp_store is None or slot_mapping is None:
        raise EtiError("surp_store and slot_mapping go together")
    st = SurpStore(_dev(surp_store, "surp_store", torch.float32),
                   _dev(slot_mapping, "slot_mapping", torch.int64, B), surp_store.numel())
    return ctypes.byref(st)


def eti_entropy_temp_sample(logits, T_in, H_prev, tau, H_target, tok, H, T_out, err_flags, ws,
                            params: CtrlParams | None = None, seed: int = 0, offset: int = 0,
                            dH=None, theta_next=None, tok_surprisal=None, V: int | None = None,
                            surp_store=None, slot_mapping=None, offset_dev=None, stream=None):
    """Half (a) of the step; see include/eti.h.  logits fp32 [B, ld]; offset_dev:
    an int64 CUDA tensor of one element that replaces `offset` and is advanced
    by one after the call's draws."""
    B, ld = logits.shape
    V = ld if V is None else int(V)
    if logits.stride(1) != 1 or logits.stride(0) != ld:
        raise EtiError("logits must be a row-major [B, ld] tensor")
    f32, i32 = torch.float32, torch.int32
    params = params or ctrl_params()
    st = load().eti_entropy_temp_sample(
        _dev(logits, "logits", f32), B, V, ld, _dev(T_in, "T_in", f32, B),
        _dev(H_prev, "H_prev", f32, B), _dev(tau, "tau", f32, B), _dev(H_target, "H_target", f32, B),
        ctypes.byref(params), int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1),
        _dev(offset_dev, "offset_dev", torch.int64, 1),
        _dev(tok, "tok", i32, B), _dev(H, "H", f32, B), _dev(T_out, "T_out", f32, B),
        _dev(dH, "dH", f32, B), _dev(theta_next, "theta_next", f32, B),
        _dev(tok_surprisal, "tok_surprisal", f32, B), _surp_store(surp_store, slot_mapping, B),
        _dev(err_flags, "err_flags", torch.int32, B),
        _dev(ws, "ws", torch.uint8), ws.numel() if ws is not None else 0, _stream(stream))
    _check(st, "eti_entropy_temp_sample")


def eti_entropy_temp_sample_noalloc(logits, T_in, H_prev, tau, H_target, tok, H, T_out, err_flags,
                                    params: CtrlParams | None = None, seed: int = 0,
                                    offset: int = 0, dH=None, theta_next=None, tok_surprisal=None,
                                    V: int | None = None, surp_store=None, slot_mapping=None,
                                    offset_dev=None, stream=None):
    """eti_entropy_temp_sample without a workspace (fixed library scratch); see include/eti.h."""
    B, ld = logits.shape
    V = ld if V is None else int(V)
    if logits.stride(1) != 1 or logits.stride(0) != ld:
        raise EtiError("logits must be a row-major [B, ld] tensor")
    f32, i32 = torch.float32, torch.int32
    params = params or ctrl_params()
    st = load().eti_entropy_temp_sample_noalloc(
        _dev(logits, "logits", f32), B, V, ld, _dev(T_in, "T_in", f32, B),
        _dev(H_prev, "H_prev", f32, B), _dev(tau, "tau", f32, B), _dev(H_target, "H_target", f32, B),
        ctypes.byref(params), int(seed) & (2 ** 64 - 1), int(offset) & (2 ** 64 - 1),
        _dev(offset_dev, "offset_dev", torch.int64, 1),
        _dev(tok, "tok", i32, B), _dev(H, "H", f32, B), _dev(T_out, "T_out", f32, B),
        _dev(dH, "dH", f32, B), _dev(theta_next, "theta_next", f32, B),
        _dev(tok_surprisal, "tok_surprisal", f32, B), _surp_store(surp_store, slot_mapping, B),
        _dev(err_flags, "err_flags", torch.int32, B), _stream(stream))
    _check(st, "eti_entropy_temp_sample_noalloc")


class SchedParams(ctypes.Structure):
    """eti_sched_params (include/eti.h)."""
    _fields_ = [(n, ctypes.c_float) for n in ("lambda_", "alpha", "beta", "gamma", "den_min")]


def sched_params(**kw) -> SchedParams:
    """Scheduling parameters: the library defaults, overridden by keywords."""
    p = SchedParams()
    load().eti_sched_defaults(ctypes.byref(p))
    for k, v in kw.items():
        setattr(p, k, float(v))
    return p


def eti_schedule(dH, ema, budget: int, priority, admit_mask, kept_cnt=None, P: int = 16,
                 ctx_lens=None, urgency=None, params: SchedParams | None = None, stream=None):
    """Entropy-aware priority and admission (Section 3.1); see include/eti.h."""
    B = dH.shape[0]
    params = params or sched_params()
    Hkv = kept_cnt.shape[1] if kept_cnt is not None else 1
    f32, i32 = torch.float32, torch.int32
    st = load().eti_schedule(
        _dev(dH, "dH", f32, B), _dev(ema, "ema", f32, B), _dev(kept_cnt, "kept_cnt", i32, B * Hkv),
        Hkv, int(P), _dev(ctx_lens, "ctx_lens", i32, B), _dev(urgency, "urgency", f32, B),
        ctypes.byref(params), B, int(budget), _dev(priority, "priority", f32, B),
        _dev(admit_mask, "admit_mask", torch.uint8, B), _stream(stream))
    _check(st, "eti_schedule")


def eti_topk_entropy(logits, T_in, k: int, H_tilde, H_hat, err_flags, tail_mass=None,
                     V: int | None = None, stream=None):
    """Top-k entropy H~, tail-corrected H^ and tail mass (Section 2.1); see include/eti.h."""
    B, ld = logits.shape
    V = ld if V is None else int(V)
    if logits.stride(1) != 1 or logits.stride(0) != ld:
        raise EtiError("logits must be a row-major [B, ld] tensor")
    f32 = torch.float32
    st = load().eti_topk_entropy(
        _dev(logits, "logits", f32), B, V, ld, _dev(T_in, "T_in", f32, B), int(k),
        _dev(H_tilde, "H_tilde", f32, B), _dev(H_hat, "H_hat", f32, B),
        _dev(tail_mass, "tail_mass", f32, B), _dev(err_flags, "err_flags", torch.int32, B),
        _stream(stream))
    _check(st, "eti_topk_entropy")


def _attn_shapes(q, k_cache, block_table):
    B, Hq, D = q.shape
    num_pages, Hkv, P, D2 = k_cache.shape
    if D2 != D:
        raise EtiError("q and k_cache head dims differ")
    if block_table.dim() != 2 or block_table.shape[0] != B:
        raise EtiError("block_table must be [B, max_blocks]")
    return B, Hq, Hkv, D, P, block_table.shape[1], num_pages


def score_prune_workspace_size(B, Hq, Hkv, D, P, max_blocks) -> int:
    return int(load().eti_score_prune_workspace_size(B, Hq, Hkv, D, P, max_blocks))


def paged_decode_workspace_size(B, Hq, Hkv, D, P, max_blocks, have_scores: bool) -> int:
    return int(load().eti_paged_decode_workspace_size(B, Hq, Hkv, D, P, max_blocks, int(have_scores)))


def eti_score_prune_blocks(q, k_cache, block_table, ctx_lens, scale: float, theta, B_min: int,
                           keep_mask, kept_idx, kept_cnt, err_flags, ws,
                           block_score=None, token_scores=None, kept_norm=None,
                           num_pages: int | None = None, score_mode: int = 0, tok_surp=None,
                           stream=None):
    """Entropic keep set of half (b); see include/eti.h.  score_mode 0 (A), 1 (E,
    with the token-surprisal store tok_surp fp32 [num_pages, P]) or 2 (M)."""
    B, Hq, Hkv, D, P, mb, npg = _attn_shapes(q, k_cache, block_table)
    num_pages = npg if num_pages is None else num_pages
    bf, i32, f32, u8 = torch.bfloat16, torch.int32, torch.float32, torch.uint8
    g = Hq // Hkv
    st = load().eti_score_prune_blocks(
        _dev(q, "q", bf), _dev(k_cache, "k_cache", bf), _dev(block_table, "block_table", i32),
        _dev(ctx_lens, "ctx_lens", i32, B), B, Hq, Hkv, D, P, mb, int(num_pages), float(scale),
        _dev(theta, "theta", f32, B), int(B_min), int(score_mode),
        _dev(tok_surp, "tok_surp", f32, npg * P),
        _dev(keep_mask, "keep_mask", u8, B * Hkv * mb), _dev(kept_idx, "kept_idx", i32, B * Hkv * mb),
        _dev(kept_cnt, "kept_cnt", i32, B * Hkv), _dev(block_score, "block_score", f32, B * Hkv * mb),
        _dev(token_scores, "token_scores", f32, B * Hkv * mb * P * g),
        _dev(kept_norm, "kept_norm", f32, B * Hq * 2), _dev(err_flags, "err_flags", i32, B),
        _dev(ws, "ws", torch.uint8), ws.numel() if ws is not None else 0, _stream(stream))
    _check(st, "eti_score_prune_blocks")


def eti_score_blocks(q, k_cache, block_table, ctx_lens, scale: float, block_stats,
                     token_scores=None, num_pages: int | None = None, tok_surp=None, stream=None):
    """The scoring pass alone (block stats and, optionally, token scores)."""
    B, Hq, Hkv, D, P, mb, npg = _attn_shapes(q, k_cache, block_table)
    num_pages = npg if num_pages is None else num_pages
    g = Hq // Hkv
    st = load().eti_score_blocks(
        _dev(q, "q", torch.bfloat16), _dev(k_cache, "k_cache", torch.bfloat16),
        _dev(block_table, "block_table", torch.int32), _dev(ctx_lens, "ctx_lens", torch.int32, B),
        B, Hq, Hkv, D, P, mb, int(num_pages), float(scale),
        _dev(tok_surp, "tok_surp", torch.float32, npg * P),
        _dev(token_scores, "token_scores", torch.float32, B * Hkv * mb * P * g),
        _dev(block_stats, "block_stats", torch.float32, B * Hq * mb * 4), _stream(stream))
    _check(st, "eti_score_blocks")


def eti_prune_blocks(block_stats, block_table, ctx_lens, shape, theta, B_min: int, keep_mask,
                     kept_idx, kept_cnt, err_flags, block_score=None, kept_norm=None,
                     num_pages: int = 0, score_mode: int = 0, stream=None):
    """The keep set from block stats; shape = (B, Hq, Hkv, D, P, max_blocks)."""
    B, Hq, Hkv, D, P, mb = shape
    i32, f32, u8 = torch.int32, torch.float32, torch.uint8
    st = load().eti_prune_blocks(
        _dev(block_stats, "block_stats", f32, B * Hq * mb * 4), _dev(block_table, "block_table", i32),
        _dev(ctx_lens, "ctx_lens", i32, B), B, Hq, Hkv, D, P, mb, int(num_pages),
        _dev(theta, "theta", f32, B), int(B_min), int(score_mode),
        _dev(keep_mask, "keep_mask", u8, B * Hkv * mb),
        _dev(kept_idx, "kept_idx", i32, B * Hkv * mb), _dev(kept_cnt, "kept_cnt", i32, B * Hkv),
        _dev(block_score, "block_score", f32, B * Hkv * mb), _dev(kept_norm, "kept_norm", f32, B * Hq * 2),
        _dev(err_flags, "err_flags", i32, B), _stream(stream))
    _check(st, "eti_prune_blocks")


def eti_paged_decode(q, k_cache, v_cache, block_table, ctx_lens, scale: float, out, err_flags, ws,
                     keep_mask=None, kept_idx=None, kept_cnt=None, token_scores=None,
                     kept_norm=None, num_pages: int | None = None, stream=None):
    """GQA paged decode over the kept blocks; see include/eti.h."""
    B, Hq, Hkv, D, P, mb, npg = _attn_shapes(q, k_cache, block_table)
    num_pages = npg if num_pages is None else num_pages
    bf, i32, f32, u8 = torch.bfloat16, torch.int32, torch.float32, torch.uint8
    g = Hq // Hkv
    st = load().eti_paged_decode(
        _dev(q, "q", bf), _dev(k_cache, "k_cache", bf), _dev(v_cache, "v_cache", bf),
        _dev(block_table, "block_table", i32), _dev(ctx_lens, "ctx_lens", i32, B),
        B, Hq, Hkv, D, P, mb, int(num_pages), float(scale),
        _dev(keep_mask, "keep_mask", u8, B * Hkv * mb), _dev(kept_idx, "kept_idx", i32, B * Hkv * mb),
        _dev(kept_cnt, "kept_cnt", i32, B * Hkv),
        _dev(token_scores, "token_scores", f32, B * Hkv * mb * P * g),
        _dev(kept_norm, "kept_norm", f32, B * Hq * 2), _dev(out, "out", bf, B * Hq * D),
        _dev(err_flags, "err_flags", i32, B), _dev(ws, "ws", torch.uint8),
        ws.numel() if ws is not None else 0, _stream(stream))
    _check(st, "eti_paged_decode")


# ---------------------------------------------------------------------------
class DecodeStep:
    """Device buffers for one batched decode step of a given shape, and the
    three calls of the step in order (score + prune, decode, entropy + sample).

    All state lives in caller-visible tensors; nothing is cached between calls
    except these preallocated buffers.
    """

    def __init__(self, B, Hq, Hkv, D, P, max_blocks, V, device="cuda", ld=None):
        self.B, self.Hq, self.Hkv, self.D, self.P, self.mb, self.V = B, Hq, Hkv, D, P, max_blocks, V
        g = Hq // Hkv
        dev = torch.device(device)
        i32, f32, u8 = torch.int32, torch.float32, torch.uint8
        self.keep_mask = torch.empty((B, Hkv, max_blocks), dtype=u8, device=dev)
        self.kept_idx = torch.empty((B, Hkv, max_blocks), dtype=i32, device=dev)
        self.kept_cnt = torch.empty((B, Hkv), dtype=i32, device=dev)
        self.block_score = torch.empty((B, Hkv, max_blocks), dtype=f32, device=dev)
        self.token_scores = torch.empty((B, Hkv, max_blocks, P, g), dtype=f32, device=dev)
        self.kept_norm = torch.empty((B, Hq, 2), dtype=f32, device=dev)
        self.err_attn = torch.empty(B, dtype=i32, device=dev)
        self.err_dec = torch.empty(B, dtype=i32, device=dev)
        self.err_ets = torch.empty(B, dtype=i32, device=dev)
        self.out = torch.empty((B, Hq, D), dtype=torch.bfloat16, device=dev)
        self.tok = torch.empty(B, dtype=i32, device=dev)
        self.H = torch.empty(B, dtype=f32, device=dev)
        self.T_out = torch.empty(B, dtype=f32, device=dev)
        self.dH = torch.empty(B, dtype=f32, device=dev)
        self.theta_next = torch.empty(B, dtype=f32, device=dev)
        self.surprisal = torch.empty(B, dtype=f32, device=dev)
        self.ws_score = torch.empty(score_prune_workspace_size(B, Hq, Hkv, D, P, max_blocks),
                                    dtype=u8, device=dev)
        self.ws_dec = torch.empty(paged_decode_workspace_size(B, Hq, Hkv, D, P, max_blocks, True),
                                  dtype=u8, device=dev)
        self.ws_ets = torch.empty(entropy_temp_sample_workspace_size(B, V), dtype=u8, device=dev)

    def attention(self, q, k_cache, v_cache, block_table, ctx_lens, scale, theta, B_min,
                  num_pages=None, stream=None):
        eti_score_prune_blocks(q, k_cache, block_table, ctx_lens, scale, theta, B_min,
                               self.keep_mask, self.kept_idx, self.kept_cnt, self.err_attn,
                               self.ws_score, block_score=self.block_score,
                               token_scores=self.token_scores, kept_norm=self.kept_norm,
                               num_pages=num_pages, stream=stream)
        eti_paged_decode(q, k_cache, v_cache, block_table, ctx_lens, scale, self.out,
                         self.err_dec, self.ws_dec, kept_idx=self.kept_idx,
                         kept_cnt=self.kept_cnt, token_scores=self.token_scores,
                         kept_norm=self.kept_norm, num_pages=num_pages, stream=stream)

    def sample(self, logits, T_in, H_prev, tau, H_target, params=None, seed=0, offset=0, V=None,
               offset_dev=None, stream=None):
        eti_entropy_temp_sample(logits, T_in, H_prev, tau, H_target, self.tok, self.H, self.T_out,
                                self.err_ets, self.ws_ets, params=params, seed=seed, offset=offset,
                                dH=self.dH,
                                theta_next=self.theta_next, tok_surprisal=self.surprisal,
                                V=V, offset_dev=offset_dev, stream=stream)


def default_scale(D: int) -> float:
    return 1.0 / math.sqrt(D)
