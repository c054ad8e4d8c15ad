"""Pins for the oracle's Semantic Retrieval Score (Sec. 3.2, Eq. 5), CPU only.

SRS(h) = sum over decode steps t whose generated token is in the answer span A of head h's
attention on A.  Independent facts: a span that covers every key gives each flagged step its
whole probability mass (SRS = the number of flagged steps); no flagged step gives 0; the score
is additive over disjoint spans and over disjoint sets of steps; and on tiny inputs it equals a
softmax computed by scipy from numpy's own logits.
"""
import math

import numpy as np
import pytest
from scipy.special import softmax

import ckv_synth as cs
from tests import independent as ind


def _bits(shape, key):
    return cs.bf16_bits(cs.normals(key, int(np.prod(shape))).reshape(shape))


def _case(seqlens=(40, 23), w=4, Hq=4, Hkv=2, d=16, key=900):
    S = len(seqlens)
    cu = np.concatenate([[0], np.cumsum(seqlens)]).astype(np.int32)
    q = _bits((S, w, Hq, d), key)
    k = _bits((int(cu[-1]), Hkv, d), key + 1)
    return cu, q, k


def test_span_over_every_key_counts_the_flagged_steps(oracle_lib):
    cu, q, k = _case()
    w, S = 4, 2
    flags = np.array([1, 0, 1, 1, 0, 1, 1, 1], np.uint8)
    span = np.array([[0, 40], [0, 23]], np.int32)
    srs = oracle_lib.semantic_retrieval_scores(q, k, cu, np.ones(4, np.uint8), w, flags, span)
    np.testing.assert_allclose(srs, np.full(4, flags.sum(), np.float64), rtol=1e-12)


def test_no_flagged_step_and_unselected_heads_give_zero(oracle_lib):
    cu, q, k = _case()
    span = np.array([[3, 20], [0, 10]], np.int32)
    srs = oracle_lib.semantic_retrieval_scores(q, k, cu, np.ones(4, np.uint8), 4, np.zeros(8, np.uint8), span)
    assert np.all(srs == 0)
    srs = oracle_lib.semantic_retrieval_scores(q, k, cu, np.array([1, 0, 0, 1], np.uint8), 4,
                                               np.ones(8, np.uint8), span)
    assert srs[1] == 0 and srs[2] == 0 and srs[0] > 0 and srs[3] > 0


def test_additive_over_spans_and_steps(oracle_lib):
    cu, q, k = _case()
    m = np.ones(4, np.uint8)
    f1 = np.array([1, 0, 1, 0, 0, 1, 0, 0], np.uint8)
    f2 = np.array([0, 1, 0, 1, 1, 0, 1, 1], np.uint8)
    sp = np.array([[5, 30], [2, 19]], np.int32)
    a = oracle_lib.semantic_retrieval_scores(q, k, cu, m, 4, f1, sp)
    b = oracle_lib.semantic_retrieval_scores(q, k, cu, m, 4, f2, sp)
    ab = oracle_lib.semantic_retrieval_scores(q, k, cu, m, 4, f1 | f2, sp)
    np.testing.assert_allclose(a + b, ab, rtol=1e-12)
    lo = oracle_lib.semantic_retrieval_scores(q, k, cu, m, 4, f1 | f2, np.array([[5, 12], [2, 7]], np.int32))
    hi = oracle_lib.semantic_retrieval_scores(q, k, cu, m, 4, f1 | f2, np.array([[12, 30], [7, 19]], np.int32))
    np.testing.assert_allclose(lo + hi, ab, rtol=1e-12)


@pytest.mark.parametrize("seqlens,w", [((9,), 3), ((12, 5), 2), ((4,), 4)])
def test_matches_scipy_softmax_on_tiny_inputs(oracle_lib, seqlens, w):
    Hq, Hkv, d = 2, 1, 8
    cu, q, k = _case(seqlens, w, Hq, Hkv, d, key=1234 + w)
    S = len(seqlens)
    flags = (np.arange(S * w) % 2 == 0).astype(np.uint8)
    span = np.array([[1, max(2, L - 1)] for L in seqlens], np.int32)
    got = oracle_lib.semantic_retrieval_scores(q, k, cu, np.ones(Hq, np.uint8), w, flags, span)
    want = np.zeros(Hq)
    for s, L in enumerate(seqlens):
        t0 = int(cu[s])
        for h in range(Hq):
            for t in range(w):
                last = L - w + t
                if not flags[s * w + t] or last < 0:
                    continue
                logits = ind.widen(k[t0:t0 + last + 1, h // (Hq // Hkv)]) @ ind.widen(q[s, t, h]) / math.sqrt(d)
                p = softmax(logits)
                a0, a1 = span[s]
                want[h] += p[a0:min(a1, last + 1)].sum()
    np.testing.assert_allclose(got, want, rtol=1e-12)


def test_planted_answer_span_ranks_the_planted_heads_first(oracle_lib):
    """Keys of a planted span aligned with the selected heads' queries (the input recipe's
    planting): those heads' attention on the span, hence their SRS, exceeds every other head's
    of the same group."""
    wl = cs.Workload(name="srs", num_layers=1, num_q_heads=8, num_kv_heads=2, seqlens=(400,),
                     window=8, heads_per_group=1, plant="span", plant_count=16, plant_beta=4.0,
                     budget_mean=64, budget_uniform=True, seed=41)
    li = wl.layer(0)
    mask = wl.head_mask()[0]
    span0 = int(li.planted[0].min())
    span = np.array([[span0, span0 + 16]], np.int32)
    srs = oracle_lib.semantic_retrieval_scores(li.q_win, li.k, wl.cu_seqlens(), np.ones(8, np.uint8),
                                               wl.window, np.ones(wl.window, np.uint8), span)
    G = 4
    for g in range(2):
        heads = list(range(g * G, (g + 1) * G))
        planted = [h for h in heads if mask[h]]
        assert len(planted) == 1
        assert srs[planted[0]] == max(srs[h] for h in heads)
