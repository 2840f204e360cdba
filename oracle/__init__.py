"""Plain fp64 CPU oracle of the entropic-time decode step.

TEST INFRASTRUCTURE ONLY: the test suite, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline / reference leg are the only callers.  The product
package never imports this module, and this module never imports the product
package; the two share nothing but the seeded input generators in
``workloads``.

The arithmetic lives in ``eti_oracle.c`` (plain C, double precision, direct
two-pass loops written from the paper's definitions).  This file only builds
that library with gcc and marshals numpy arrays into it.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "eti_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

ERR_BAD_PAGE = 0x1
ERR_BAD_CTX = 0x2
ERR_NONFINITE = 0x4
ERR_ALL_NEG_INF = 0x8
ERR_BAD_TEMP = 0x10


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (OpenMP when the compiler has it)."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    base = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", _SRC, "-o", tmp, "-lm"]
    try:
        subprocess.run(base[:1] + ["-fopenmp"] + base[1:], check=True,
                       capture_output=True, text=True)
    except subprocess.CalledProcessError:
        subprocess.run(base, check=True, capture_output=True, text=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


class _Ctrl(ctypes.Structure):
    _fields_ = [("eta", ctypes.c_double), ("sign", ctypes.c_double),
                ("T_min", ctypes.c_double), ("T_max", ctypes.c_double),
                ("eps_H", ctypes.c_double), ("H_min", ctypes.c_double),
                ("theta_user", ctypes.c_double), ("theta_hi", ctypes.c_double),
                ("T_cal", ctypes.c_double), ("rho_T", ctypes.c_double),
                ("dtheta", ctypes.c_double)]


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            P = ctypes.c_void_p
            i32, i64, u64, f64 = ctypes.c_int, ctypes.c_int64, ctypes.c_uint64, ctypes.c_double
            lib.oracle_num_threads.restype = i32
            lib.oracle_philox4x32_10.argtypes = [P, P, P]
            lib.oracle_words.argtypes = [P, P, i64, P]
            lib.oracle_uniforms.argtypes = [u64, u64, i64, i64, i64, P]
            lib.oracle_sample_key.argtypes = [P, f64, u64, u64, i64, i64]
            lib.oracle_sample_key.restype = f64
            lib.oracle_entropy_row.argtypes = [P, i64, f64]
            lib.oracle_entropy_row.restype = f64
            lib.oracle_entropy_temp_sample.argtypes = (
                [P, i32, i64, i64, P, P, P, P, P, u64, u64] + [P] * 10)
            lib.oracle_topk_entropy.argtypes = [P, i32, i64, i64, P, i64, P, P, P, P]
            lib.oracle_schedule.argtypes = [P, P, P, i32, i32, P, P, P, i32, i32, P, P, P]
            lib.oracle_score_prune.argtypes = (
                [P, P, P, P, i32, i32, i32, i32, i32, i32, i64, f64, P, i32, i32, P] + [P] * 8)
            lib.oracle_paged_attention.argtypes = (
                [P, P, P, P, P, i32, i32, i32, i32, i32, i32, i64, f64, P, P, P])
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _c(a, dtype):
    return np.ascontiguousarray(a, dtype=dtype)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


# ---------------------------------------------------------------------------
# Controller parameters (defaults are the readings stated in the design notes:
# eta 0.1, restoring sign, T in [0.05, 5], no estimator slack, no entropy
# floor, no user threshold, theta_max scale 1).
DEFAULT_CTRL = dict(eta=0.1, sign=-1.0, T_min=0.05, T_max=5.0, eps_H=0.0, H_min=0.0,
                    theta_user=float("inf"), theta_hi=1.0, T_cal=1.0, rho_T=0.0, dtheta=0.0)


def ctrl(**kw) -> dict:
    c = dict(DEFAULT_CTRL)
    c.update(kw)
    return c


def philox4x32_10(ctr, key) -> np.ndarray:
    """Philox4x32-10 blocks: ctr uint32 [n,4], key uint32 [n,2] -> uint32 [n,4]."""
    ctr = _c(np.atleast_2d(ctr), np.uint32)
    key = _c(np.atleast_2d(key), np.uint32)
    out = np.empty_like(ctr)
    _load().oracle_words(_ptr(ctr), _ptr(key), ctr.shape[0], _ptr(out))
    return out


def uniforms(seed: int, offset: int, row: int, x0: int, n: int) -> np.ndarray:
    """The sampler's uniforms u_x for tokens x0..x0+n-1 of one row."""
    out = np.empty(n, np.float64)
    _load().oracle_uniforms(seed, offset, row, x0, n, _ptr(out))
    return out


def sample_key(logits_row, T: float, seed: int, offset: int, row: int, x: int) -> float:
    z = _c(logits_row, np.float32)
    return float(_load().oracle_sample_key(_ptr(z), float(T), seed, offset, row, x))


def entropy_row(z, T: float = 1.0) -> float:
    z = _c(z, np.float32)
    return float(_load().oracle_entropy_row(_ptr(z), z.shape[0], float(T)))


class _Sched(ctypes.Structure):
    _fields_ = [(n, ctypes.c_double) for n in ("lambda_", "alpha", "beta", "gamma", "den_min")]


DEFAULT_SCHED = dict(lambda_=0.9, alpha=1e-3, beta=1e-3, gamma=1.0, den_min=1e-6)


def schedule(dH, ema_in, budget: int, kept_cnt=None, P: int = 16, ctx_lens=None, urgency=None,
             params=None) -> dict:
    """Entropy-aware priority pi(s) and the admitted set (Section 3.1, reading R14).

    dH, ema_in, urgency float32 [B]; kept_cnt int32 [B, Hkv]; ctx_lens int32 [B].
    """
    lib = _load()
    dH = _c(dH, np.float32)
    B = dH.shape[0]
    ema_in = _c(ema_in, np.float32)
    kc = None if kept_cnt is None else _c(kept_cnt, np.int32)
    Hkv = 1 if kc is None else kc.shape[1]
    cl = None if ctx_lens is None else _c(ctx_lens, np.int32)
    ur = None if urgency is None else _c(urgency, np.float32)
    sp = _Sched(**{**DEFAULT_SCHED, **(params or {})})
    out = dict(ema=np.empty(B), priority=np.empty(B), admit=np.empty(B, np.uint8))
    lib.oracle_schedule(_ptr(dH), _ptr(ema_in), _ptr(kc), Hkv, int(P), _ptr(cl), _ptr(ur),
                        ctypes.byref(sp), B, int(budget), _ptr(out["ema"]), _ptr(out["priority"]),
                        _ptr(out["admit"]))
    return out


def topk_entropy(logits, T_in, k: int, V: int | None = None) -> dict:
    """Top-k entropy H~, tail-corrected H^ and the tail mass of every row.

    logits float32 [B, ld] (the first V columns are the vocabulary); T_in [B].
    """
    lib = _load()
    z = _c(logits, np.float32)
    B, ld = z.shape
    V = ld if V is None else int(V)
    T_in = _c(T_in, np.float32)
    out = {n: np.empty(B, np.float64) for n in ("H_tilde", "H_hat", "tail_mass")}
    err = np.empty(B, np.uint32)
    lib.oracle_topk_entropy(_ptr(z), B, V, ld, _ptr(T_in), int(k), _ptr(out["H_tilde"]),
                            _ptr(out["H_hat"]), _ptr(out["tail_mass"]), _ptr(err))
    out["err"] = err
    return out


def entropy_temp_sample(logits, T_in, H_prev, tau_in, H_target, ctrl_params=None,
                        seed: int = 0, offset: int = 0, V: int | None = None, theta_prev=None):
    """Entropy / entropic time / temperature / threshold / Gumbel-max sample.

    logits: float32 [B, ld] (the first V columns are the vocabulary);
    theta_prev float32 [B]: the previous thresholds (used by the dtheta guard).
    Returns a dict of numpy arrays (double outputs, int32 tok, uint32 err).
    """
    lib = _load()
    z = _c(logits, np.float32)
    B, ld = z.shape
    V = ld if V is None else V
    cp = _Ctrl(**{**DEFAULT_CTRL, **(ctrl_params or {})})
    T_in, H_prev, tau_in, H_target = (_c(a, np.float32) for a in (T_in, H_prev, tau_in, H_target))
    theta_prev = None if theta_prev is None else _c(theta_prev, np.float32)
    out = {k: np.empty(B, np.float64) for k in
           ("H", "T_out", "dH", "tau", "theta_next", "surprisal", "margin")}
    tok = np.empty(B, np.int32)
    err = np.empty(B, np.uint32)
    lib.oracle_entropy_temp_sample(
        _ptr(z), B, V, ld, _ptr(T_in), _ptr(H_prev), _ptr(tau_in), _ptr(H_target),
        ctypes.byref(cp), seed, offset, _ptr(theta_prev), _ptr(tok), _ptr(out["H"]), _ptr(out["T_out"]),
        _ptr(out["dH"]), _ptr(out["tau"]), _ptr(out["theta_next"]), _ptr(out["surprisal"]),
        _ptr(out["margin"]), _ptr(err))
    out["tok"] = tok
    out["err"] = err
    return out


SCORE_A, SCORE_E, SCORE_M = 0, 1, 2


def score_prune(q, k_cache, block_table, ctx_lens, scale: float, theta, B_min: int,
                num_pages: int | None = None, want_heads: bool = False,
                score_mode: int = SCORE_A, surp=None):
    """Entropic block scores, keep mask and compacted kept lists.

    q: bf16 bit patterns uint16 [B, Hq, D]; k_cache uint16 [pages, Hkv, P, D];
    block_table int32 [B, max_blocks]; ctx_lens int32 [B]; theta float32 [B];
    score_mode 0 (A: -log a_i), 1 (E: stored token surprisal surp float32
    [pages, P]) or 2 (M: attention mass).
    """
    lib = _load()
    q = _c(q, np.uint16)
    k_cache = _c(k_cache, np.uint16)
    bt = _c(block_table, np.int32)
    cl = _c(ctx_lens, np.int32)
    th = _c(theta, np.float32)
    B, Hq, D = q.shape
    pages, Hkv, P, D2 = k_cache.shape
    assert D2 == D and Hq % Hkv == 0
    mb = bt.shape[1]
    num_pages = pages if num_pages is None else num_pages
    keep = np.empty((B, Hkv, mb), np.uint8)
    kidx = np.empty((B, Hkv, mb), np.int32)
    kcnt = np.empty((B, Hkv), np.int32)
    score = np.empty((B, Hkv, mb), np.float64)
    head_I = np.empty((B, Hq, mb), np.float64) if want_heads else None
    head_A = np.empty((B, Hq, mb), np.float64) if want_heads else None
    head_H = np.empty((B, Hq), np.float64) if want_heads else None
    err = np.empty(B, np.uint32)
    if score_mode == SCORE_E:
        surp = _c(surp, np.float32)
        assert surp.shape == (pages, P)
    else:
        surp = None
    lib.oracle_score_prune(_ptr(q), _ptr(k_cache), _ptr(bt), _ptr(cl), B, Hq, Hkv, D, P, mb,
                           num_pages, float(scale), _ptr(th), int(B_min), int(score_mode),
                           _ptr(surp), _ptr(keep), _ptr(kidx),
                           _ptr(kcnt), _ptr(score), _ptr(head_I), _ptr(head_A), _ptr(head_H),
                           _ptr(err))
    res = dict(keep_mask=keep, kept_idx=kidx, kept_cnt=kcnt, block_score=score, err=err)
    if want_heads:
        res["head_I"] = head_I
        res["head_A"] = head_A
        res["head_H"] = head_H
    return res


def paged_attention(q, k_cache, v_cache, block_table, ctx_lens, scale: float,
                    keep_mask=None, num_pages: int | None = None):
    """Exact paged GQA decode over the kept blocks (all blocks if keep_mask is None).

    Returns (out float64 [B, Hq, D], err uint32 [B]).
    """
    lib = _load()
    q = _c(q, np.uint16)
    k_cache = _c(k_cache, np.uint16)
    v_cache = _c(v_cache, np.uint16)
    bt = _c(block_table, np.int32)
    cl = _c(ctx_lens, np.int32)
    km = None if keep_mask is None else _c(keep_mask, np.uint8)
    B, Hq, D = q.shape
    pages, Hkv, P, _ = k_cache.shape
    mb = bt.shape[1]
    num_pages = pages if num_pages is None else num_pages
    out = np.empty((B, Hq, D), np.float64)
    err = np.empty(B, np.uint32)
    lib.oracle_paged_attention(_ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(bt), _ptr(cl),
                               B, Hq, Hkv, D, P, mb, num_pages, float(scale), _ptr(km),
                               _ptr(out), _ptr(err))
    return out, err
