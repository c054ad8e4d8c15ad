"""fp64 CPU oracle for the CompressKV compression step -- TEST INFRASTRUCTURE ONLY.

Only the tests, the package smoke check and the benchmark's CPU-baseline leg load this module.
The CUDA library never imports, links or calls it.  ``build()`` compiles ``ckv_oracle.c`` with
gcc (OpenMP, no fast-math, no FMA contraction) next to this file; the functions below marshal
numpy arrays into it.  See ``ckv_oracle.c`` for the definitions and the paper passages they
follow.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ckv_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libckv_oracle.so")
_lib = None

POOL_MAX, POOL_AVG = 0, 1
POOL_THEN_SUM, SUM_THEN_POOL = 0, 1


def build(force: bool = False) -> str:
    """Compiles the oracle shared library (gcc, C11, OpenMP)."""
    if force or not os.path.exists(_LIB_PATH) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC):
        tmp = _LIB_PATH + f".{os.getpid()}.tmp"
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp",
                               "-ffp-contract=off", "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is None:
        build()
        lib = C.CDLL(_LIB_PATH)
        P = C.c_void_p
        lib.ckv_oracle_window_scores.argtypes = [C.c_int, C.c_int, C.c_int, C.c_double, P, C.c_long,
                                                 P, C.c_long, P, P, P]
        lib.ckv_oracle_pool.argtypes = [P, C.c_int, C.c_int, C.c_int, P]
        lib.ckv_oracle_topk.argtypes = [P, C.c_int, C.c_int, P]
        lib.ckv_oracle_keep_lengths.argtypes = [C.c_int, P, C.c_int, P]
        lib.ckv_oracle_window_scores_lse.argtypes = [C.c_int, C.c_int, C.c_int, C.c_double, P,
                                                     C.c_long, P, C.c_long, P, P]
        lib.ckv_oracle_compress_layer.argtypes = [
            C.c_int, P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_double, P, C.c_int,
            C.c_int, C.c_int, C.c_int, C.c_int, P, P, P, P, C.c_long, P, P, P, P, P, P, P, C.c_int]
        lib.ckv_oracle_srs.argtypes = [C.c_int, P, C.c_int, C.c_int, C.c_int, C.c_int, C.c_double,
                                       P, P, P, P, P, P]
        lib.ckv_oracle_threads.argtypes = [C.c_int]
        _lib = lib
    return _lib


def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _check(rc):
    if rc != 0:
        raise ValueError(f"oracle rejected its arguments (code {rc})")


def threads(n: int = 0) -> int:
    return _load().ckv_oracle_threads(n)


def window_scores(q_rows: np.ndarray, k_rows: np.ndarray, scale: float | None = None):
    """Window attention of one head: q_rows [w, d], k_rows [L, d] (bf16 bits, uint16).

    Returns (a [L], lse [w], mass [w]) in float64.
    """
    q = np.ascontiguousarray(q_rows, dtype=np.uint16)
    k = np.ascontiguousarray(k_rows, dtype=np.uint16)
    w, d = q.shape
    L = k.shape[0]
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    a = np.empty(L, np.float64)
    lse = np.empty(w, np.float64)
    mass = np.empty(w, np.float64)
    _check(_load().ckv_oracle_window_scores(L, w, d, float(scale), _p(q), d, _p(k), d,
                                            _p(a), _p(lse), _p(mass)))
    return a, lse, mass


def window_scores_lse(q_rows: np.ndarray, k_rows: np.ndarray, lse: np.ndarray,
                      scale: float | None = None) -> np.ndarray:
    """Window scores of one head with the rows' normalisers given (lse [w], natural log):
    a [L] = sum over the rows that see key j of exp(s - lse_r)."""
    q = np.ascontiguousarray(q_rows, dtype=np.uint16)
    k = np.ascontiguousarray(k_rows, dtype=np.uint16)
    lse = np.ascontiguousarray(lse, dtype=np.float64)
    w, d = q.shape
    L = k.shape[0]
    assert lse.shape == (w,)
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    a = np.empty(L, np.float64)
    _check(_load().ckv_oracle_window_scores_lse(L, w, d, float(scale), _p(q), d, _p(k), d, _p(lse), _p(a)))
    return a


def pool(x: np.ndarray, kernel: int, pool_type: int) -> np.ndarray:
    x = np.ascontiguousarray(x, dtype=np.float64)
    y = np.empty_like(x)
    _check(_load().ckv_oracle_pool(_p(x), x.size, kernel, pool_type, _p(y)))
    return y


def topk(c: np.ndarray, k: int) -> np.ndarray:
    c = np.ascontiguousarray(c, dtype=np.float64)
    out = np.empty(max(k, 0), np.int32)
    _check(_load().ckv_oracle_topk(_p(c), c.size, k, _p(out)))
    return out


def keep_lengths(cu_seqlens: np.ndarray, budget: int) -> np.ndarray:
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    out = np.empty_like(cu)
    _check(_load().ckv_oracle_keep_lengths(cu.size - 1, _p(cu), budget, _p(out)))
    return out


SCOPE_KV_HEAD, SCOPE_LAYER = 0, 1


def compress_layer(q_win, k, v, cu_seqlens, head_mask, budget, window, pool_kernel, pool_type,
                   head_order, scale=None, want_scores=True, want_kv=True, groups=None,
                   num_threads=0, scope=SCOPE_KV_HEAD, lse=None):
    """One layer of the compression step.  Arrays are bf16 bits (uint16), packed.

    q_win [S, w, Hq, d], k/v [T, Hkv, d], cu_seqlens [S+1], head_mask [Hq] (uint8).
    Returns a dict with scores [n_sel, T] (float64), pooled [Hkv, T] (float64; [1, T] with
    scope=SCOPE_LAYER), cu_keep [S+1], idx [Hkv, T_keep] (int32), k_out / v_out
    [T_keep, Hkv, d] (uint16).  ``groups`` (optional iterable of KV heads, KV-head scope only)
    restricts the work to those groups; rows of the other groups are left as NaN / -1.
    ``lse`` (optional, [Hq, S*w] float64, natural log): the window rows' normalisers, used
    instead of computing them.
    """
    q_win = np.ascontiguousarray(q_win, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    v = np.ascontiguousarray(v, dtype=np.uint16)
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    mask = np.ascontiguousarray(head_mask, dtype=np.uint8)
    S = cu.size - 1
    T, Hkv, d = k.shape
    Hq = q_win.shape[2]
    assert q_win.shape == (S, window, Hq, d) and int(cu[-1]) == T
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    cu_keep = keep_lengths(cu, budget)
    Tk = int(cu_keep[-1])
    n_sel = int(mask.astype(bool).sum())
    scores = np.full((n_sel, T), np.nan) if want_scores else None
    pooled = np.full((Hkv if scope == SCOPE_KV_HEAD else 1, T), np.nan)
    idx = np.full((Hkv, Tk), -1, np.int32)
    k_out = np.zeros((Tk, Hkv, d), np.uint16) if want_kv else None
    v_out = np.zeros((Tk, Hkv, d), np.uint16) if want_kv else None
    gf = None
    if groups is not None:
        gf = np.zeros(Hkv, np.uint8)
        gf[list(groups)] = 1
    lse_arr, lse_stride = None, 0
    if lse is not None:
        lse_arr = np.ascontiguousarray(lse, dtype=np.float64)
        assert lse_arr.ndim == 2 and lse_arr.shape[0] == Hq and lse_arr.shape[1] >= S * window
        lse_stride = lse_arr.shape[1]
    _check(_load().ckv_oracle_compress_layer(
        S, _p(cu), Hq, Hkv, d, window, float(scale), _p(mask), int(budget), int(pool_kernel),
        int(pool_type), int(head_order), int(scope), _p(q_win), _p(k), _p(v), _p(lse_arr),
        int(lse_stride), _p(scores), _p(pooled), None, _p(idx), _p(k_out), _p(v_out), _p(gf),
        int(num_threads)))
    return dict(scores=scores, pooled=pooled, cu_keep=cu_keep, idx=idx, k_out=k_out, v_out=v_out)


def semantic_retrieval_scores(q_dec, k, cu_seqlens, head_mask, window, in_answer, span, scale=None):
    """Eq. 5 per selected head, summed over the batch's sequences: float64 [Hq] (0 for heads
    that are not selected).  q_dec [S, w, Hq, d], k [T, Hkv, d] (bf16 bits), in_answer [S*w],
    span [S, 2] (sequence-local [a0, a1))."""
    q = np.ascontiguousarray(q_dec, dtype=np.uint16)
    k = np.ascontiguousarray(k, dtype=np.uint16)
    cu = np.ascontiguousarray(cu_seqlens, dtype=np.int32)
    mask = np.ascontiguousarray(head_mask, dtype=np.uint8)
    flags = np.ascontiguousarray(in_answer, dtype=np.uint8)
    sp = np.ascontiguousarray(span, dtype=np.int32)
    S = cu.size - 1
    T, Hkv, d = k.shape
    Hq = q.shape[2]
    assert q.shape == (S, window, Hq, d) and flags.size == S * window and sp.shape == (S, 2)
    scale = 1.0 / np.sqrt(d) if scale is None else scale
    out = np.zeros(Hq, np.float64)
    _check(_load().ckv_oracle_srs(S, _p(cu), Hq, Hkv, d, window, float(scale), _p(mask), _p(q), _p(k),
                                  _p(flags), _p(sp), _p(out)))
    return out
