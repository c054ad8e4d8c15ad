"""Independent statements of the compression step, used only to pin the oracle.

They share no code or structure with ``oracle/ckv_oracle.c``:
  * ``window_attention_exact`` builds each window row's causal softmax with exactly rounded
    sums (``math.fsum``) and divides by the partition function;
  * ``window_attention_matrix`` forms the full L x L causal attention matrix with numpy and
    ``scipy.special.softmax`` and slices the window rows out of it;
  * ``compress_layer_reference`` runs the whole step on top of the matrix form, pooling with
    ``scipy.ndimage`` filters and ranking with ``numpy.lexsort``.
"""
from __future__ import annotations

import math

import numpy as np
from scipy.ndimage import maximum_filter1d, uniform_filter1d
from scipy.special import softmax


def widen(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns -> float64, via a float32 view of the high half-word."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) * np.uint32(65536)
    return u.view(np.float32).astype(np.float64)


def window_attention_exact(q_rows, k_rows, scale):
    """q_rows [w, d], k_rows [L, d] as float64 lists/arrays.  Returns (a, lse, mass)."""
    q = [list(map(float, r)) for r in np.asarray(q_rows)]
    k = [list(map(float, r)) for r in np.asarray(k_rows)]
    w, L = len(q), len(k)
    P = L - w
    per_key = [[] for _ in range(L)]
    lse, mass = [], []
    for r in range(w):
        pos = P + r
        if pos < 0:
            lse.append(float("nan"))
            mass.append(0.0)
            continue
        logits = [scale * math.fsum(qc * kc for qc, kc in zip(q[r], k[j])) for j in range(pos + 1)]
        top = max(logits)
        z = math.fsum(math.exp(x - top) for x in logits)
        probs = [math.exp(x - top) / z for x in logits]
        for j, p in enumerate(probs):
            per_key[j].append(p)
        lse.append(top + math.log(z))
        mass.append(math.fsum(probs[max(P, 0):]))
    a = np.array([math.fsum(v) for v in per_key])
    return a, np.array(lse), np.array(mass)


def window_attention_matrix(q_rows, k_rows, scale, filler_seed=0):
    """Full causal attention over all L query positions; returns the window-row sum per key.

    Query positions before the window get arbitrary filler rows (they are sliced away).
    Requires L >= w.
    """
    q_rows = np.asarray(q_rows, np.float64)
    k_rows = np.asarray(k_rows, np.float64)
    w, d = q_rows.shape
    L = k_rows.shape[0]
    assert L >= w
    rng = np.random.default_rng(filler_seed)
    q_all = np.concatenate([rng.standard_normal((L - w, d)), q_rows], axis=0)
    logits = scale * (q_all @ k_rows.T)
    causal = np.tril(np.ones((L, L), dtype=bool))
    logits = np.where(causal, logits, -np.inf)
    probs = softmax(logits, axis=1)
    return probs[L - w:].sum(axis=0)


def _pool(x, kernel, pool_type):
    if x.size == 0:
        return x.copy()
    if pool_type == 0:
        return maximum_filter1d(x, size=kernel, mode="constant", cval=0.0)
    return uniform_filter1d(x, size=kernel, mode="constant", cval=0.0)


def compress_layer_reference(q_win, k, v, cu_seqlens, head_mask, budget, window, pool_kernel,
                             pool_type, head_order, scale=None, scope=0):
    """Whole step for inputs where every sequence has L >= window.  bf16 bits in.

    scope 0: one vector and selection per KV head g from the selected heads of group g;
    scope 1: one per sequence from all selected heads (kept[(s, 0)], pooled row 0)."""
    qf, kf = widen(q_win), widen(k)
    S = len(cu_seqlens) - 1
    T, Hkv, d = k.shape
    Hq = q_win.shape[2]
    G = Hq // Hkv
    scale = 1.0 / math.sqrt(d) if scale is None else scale
    n_vec = Hkv if scope == 0 else 1
    pooled = np.zeros((n_vec, T))
    kept = {}
    for s in range(S):
        t0, t1 = int(cu_seqlens[s]), int(cu_seqlens[s + 1])
        L = t1 - t0
        P = L - window
        for g in range(n_vec):
            span = range(g * G, (g + 1) * G) if scope == 0 else range(Hq)
            heads = [h for h in span if head_mask[h]]
            vecs = [window_attention_matrix(qf[s, :, h, :], kf[t0:t1, h // G, :], scale)[:P]
                    for h in heads]
            if head_order == 0:
                c = np.sum([_pool(a, pool_kernel, pool_type) for a in vecs], axis=0)
            else:
                c = _pool(np.sum(vecs, axis=0), pool_kernel, pool_type)
            pooled[g, t0:t0 + P] = c
            if L <= budget:
                kept[(s, g)] = np.arange(L)
            else:
                order = np.lexsort((np.arange(P), -c))
                kept[(s, g)] = np.concatenate([np.sort(order[:budget - window]),
                                               np.arange(P, L)])
    return pooled, kept
