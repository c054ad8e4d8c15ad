"""Pins for the oracle's given-lse path (the window rows' normalisers supplied by the caller, as
a prefill attention kernel returns them; Sec. 3.3 with the attention of Eq. 2).

With the true normalisers the scores are the window attention summed over the rows, so the
given-lse scores must equal the ones computed from scratch when the lse is obtained by an
independent routine (scipy's logsumexp over numpy's own logits); a shifted lse must scale a
row's contribution by exp(-shift); rows whose query position is before the sequence start are
never read.
"""
import math

import numpy as np
import pytest
from scipy.special import logsumexp

import ckv_synth as cs
from tests import independent as ind


def _bits(shape, key):
    return cs.bf16_bits(cs.normals(key, int(np.prod(shape))).reshape(shape))


def _independent_lse(q_bits, k_bits, scale):
    """log sum_{j <= P + r} exp(scale q_r . k_j) per window row, by numpy and scipy."""
    q, k = ind.widen(q_bits), ind.widen(k_bits)
    w, L = q.shape[0], k.shape[0]
    P = L - w
    s = scale * (q @ k.T)
    out = np.full(w, np.nan)
    for r in range(w):
        if P + r >= 0:
            out[r] = logsumexp(s[r, :P + r + 1])
    return out


@pytest.mark.parametrize("L,w,d", [(1, 1, 8), (7, 3, 8), (40, 8, 16), (129, 32, 128), (5, 8, 8)])
def test_given_true_lse_reproduces_the_scores(oracle_lib, L, w, d):
    q = _bits((w, d), 5000 + L)
    k = _bits((L, d), 6000 + L)
    scale = 1.0 / math.sqrt(d)
    a, _, _ = oracle_lib.window_scores(q, k)
    lse = _independent_lse(q, k, scale)
    b = oracle_lib.window_scores_lse(q, k, lse)  # NaN rows (L < w) must not be read
    assert np.all(np.isfinite(b))
    np.testing.assert_allclose(b, a, rtol=1e-11, atol=1e-300)


@pytest.mark.parametrize("delta", [-3.0, 0.5, 7.25])
def test_shifted_lse_scales_a_single_row(oracle_lib, delta):
    q = _bits((1, 16), 7001)
    k = _bits((50, 16), 7002)
    lse = _independent_lse(q, k, 0.25)
    a0 = oracle_lib.window_scores_lse(q, k, lse, scale=0.25)
    a1 = oracle_lib.window_scores_lse(q, k, lse + delta, scale=0.25)
    np.testing.assert_allclose(a1, a0 * math.exp(-delta), rtol=1e-12)
    np.testing.assert_allclose(a0.sum(), 1.0, rtol=1e-12)  # one row: a probability distribution


def test_shift_of_one_row_changes_only_that_rows_share(oracle_lib):
    w, L, d = 4, 30, 8
    q = _bits((w, d), 7101)
    k = _bits((L, d), 7102)
    scale = 1.0 / math.sqrt(d)
    lse = _independent_lse(q, k, scale)
    base = oracle_lib.window_scores_lse(q, k, lse)
    shifted = lse.copy()
    shifted[2] += 1.5
    b = oracle_lib.window_scores_lse(q, k, shifted)
    # row 2's probabilities alone, by numpy
    s = scale * (ind.widen(q) @ ind.widen(k).T)
    P = L - w
    p2 = np.zeros(L)
    p2[:P + 3] = np.exp(s[2, :P + 3] - lse[2])
    np.testing.assert_allclose(b, base + (math.exp(-1.5) - 1.0) * p2, rtol=1e-11, atol=1e-15)


@pytest.mark.parametrize("scope", [0, 1])
def test_compress_layer_with_the_lse_it_would_compute(oracle_lib, scope):
    """The layer function's lse input ([Hq, S*w], natural log) gives the same result as letting
    it compute the normalisers, when fed the independently computed ones."""
    wl = cs.Workload(name="lse_pin", num_layers=1, num_q_heads=8, num_kv_heads=2,
                     seqlens=(300, 5, 700), window=8, heads_per_group=2, budget_mean=40,
                     budget_uniform=True, pool_kernel=5, seed=17,
                     **({"scope": "layer", "heads_per_layer": 3} if scope else {}))
    li = wl.layer(0)
    cu = wl.cu_seqlens()
    S, w, Hq = wl.num_seqs, wl.window, wl.num_q_heads
    G = Hq // wl.num_kv_heads
    scale = 1.0 / math.sqrt(wl.head_dim)
    lse = np.full((Hq, S * w + 3), np.nan)  # a padded row stride
    for s in range(S):
        t0, t1 = int(cu[s]), int(cu[s + 1])
        for h in range(Hq):
            lse[h, s * w:(s + 1) * w] = _independent_lse(li.q_win[s, :, h], li.k[t0:t1, h // G], scale)
    mask = wl.head_mask()[0]
    args = (li.q_win, li.k, li.v, cu, mask, int(wl.budgets()[0]), w, wl.pool_kernel, 0, 0)
    ref = oracle_lib.compress_layer(*args, scope=scope)
    got = oracle_lib.compress_layer(*args, scope=scope, lse=lse)
    np.testing.assert_allclose(got["scores"], ref["scores"], rtol=1e-11, atol=1e-300)
    np.testing.assert_allclose(got["pooled"], ref["pooled"], rtol=1e-11, atol=1e-300)
    np.testing.assert_array_equal(got["idx"], ref["idx"])
    np.testing.assert_array_equal(got["k_out"], ref["k_out"])
