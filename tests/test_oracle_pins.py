"""Pins for the fp64 oracle against things other than itself (CPU only).

Each test ties one part of the oracle to an independent fact: exact brute force on tiny inputs,
a closed form, a library routine, an exhaustive search, or an invariant of the method
(Sec. 3.3 of the paper; Eq. 2 for the attention; App. A for the pooling).
"""
import itertools
import math

import numpy as np
import pytest

import ckv_synth as cs
from tests import independent as ind

pytestmark = pytest.mark.filterwarnings("ignore::RuntimeWarning")


def _bits(shape, key):
    return cs.bf16_bits(cs.normals(key, int(np.prod(shape))).reshape(shape))


# ---------------------------------------------------------------- window attention (Eq. 2)
@pytest.mark.parametrize("L,w,d", [(1, 1, 8), (5, 1, 8), (5, 3, 8), (17, 8, 16), (40, 8, 8),
                                   (9, 9, 16), (10, 9, 8), (3, 8, 8), (33, 32, 8)])
def test_window_scores_match_exact_bruteforce(oracle_lib, L, w, d):
    q = _bits((w, d), 1000 + L * 7 + w)
    k = _bits((L, d), 2000 + L * 7 + w)
    scale = 1.0 / math.sqrt(d)
    a, lse, mass = oracle_lib.window_scores(q, k)
    ea, else_, emass = ind.window_attention_exact(ind.widen(q), ind.widen(k), scale)
    np.testing.assert_allclose(a, ea, rtol=1e-12, atol=1e-300)
    np.testing.assert_allclose(lse, else_, rtol=1e-12, equal_nan=True)
    np.testing.assert_allclose(mass, emass, rtol=1e-12, atol=1e-300)


@pytest.mark.parametrize("L,w,d", [(64, 8, 128), (100, 32, 128), (33, 32, 16)])
def test_window_scores_match_full_attention_matrix(oracle_lib, L, w, d):
    q = _bits((w, d), 3000 + L)
    k = _bits((L, d), 4000 + L)
    a, _, _ = oracle_lib.window_scores(q, k)
    ref = ind.window_attention_matrix(ind.widen(q), ind.widen(k), 1.0 / math.sqrt(d))
    np.testing.assert_allclose(a, ref, rtol=1e-12)


def test_window_scores_equal_keys_closed_form(oracle_lib):
    """All keys equal: row r spreads 1/(P+r+1) over its visible keys."""
    L, w, d = 50, 8, 128
    q = _bits((w, d), 11)
    k = np.tile(_bits((1, d), 12), (L, 1))
    a, lse, mass = oracle_lib.window_scores(q, k)
    P = L - w
    expect = np.array([sum(1.0 / (P + r + 1) for r in range(w) if j <= P + r) for j in range(L)])
    np.testing.assert_allclose(a, expect, rtol=1e-13)
    # and with q = 0 every logit is 0: the same closed form, lse = log(P + r + 1)
    a0, lse0, _ = oracle_lib.window_scores(np.zeros((w, d), np.uint16), _bits((L, d), 13))
    np.testing.assert_allclose(a0, expect, rtol=1e-13)
    np.testing.assert_allclose(lse0, np.log(P + np.arange(w) + 1.0), rtol=1e-14)


@pytest.mark.parametrize("L,w", [(32, 32), (33, 32), (300, 32), (129, 8)])
def test_window_rows_sum_to_one(oracle_lib, L, w):
    """Every window row is a distribution: candidates + window mass = w in total."""
    q = _bits((w, 128), 21 + L)
    k = _bits((L, 128), 22 + L)
    a, lse, mass = oracle_lib.window_scores(q, k)
    P = L - w
    assert np.all(np.isfinite(lse))
    assert math.isclose(math.fsum(a[:P]) + math.fsum(mass), w, rel_tol=1e-12)
    assert math.isclose(math.fsum(a), w, rel_tol=1e-12)
    assert np.all(mass > 0) and np.all(mass <= 1 + 1e-15)


def test_window_scores_scale_argument(oracle_lib):
    """A scale of 0 makes every visible key equally likely (pins the use of the scale)."""
    L, w, d = 20, 4, 8
    a, _, _ = oracle_lib.window_scores(_bits((w, d), 5), _bits((L, d), 6), scale=0.0)
    P = L - w
    expect = np.array([sum(1.0 / (P + r + 1) for r in range(w) if j <= P + r) for j in range(L)])
    np.testing.assert_allclose(a, expect, rtol=1e-13)


# ---------------------------------------------------------------- pooling (Sec. 3.3, App. A)
@pytest.mark.parametrize("n", [1, 2, 3, 6, 10, 101])
@pytest.mark.parametrize("kernel", [1, 3, 5, 7, 9])
@pytest.mark.parametrize("pool_type", [0, 1])
def test_pool_matches_scipy_filters(oracle_lib, n, kernel, pool_type):
    rng = np.random.default_rng(n * 100 + kernel)
    x = rng.random(n) ** 3
    y = oracle_lib.pool(x, kernel, pool_type)
    if pool_type == 0:
        from scipy.ndimage import maximum_filter1d
        ref = maximum_filter1d(x, size=kernel, mode="constant", cval=0.0)
    else:
        from scipy.ndimage import uniform_filter1d
        ref = uniform_filter1d(x, size=kernel, mode="constant", cval=0.0)
    # scipy's running-sum filter carries absolute (not relative) rounding error
    np.testing.assert_allclose(y, ref, rtol=1e-13, atol=1e-14 * max(x.max(), 1e-300))


@pytest.mark.parametrize("kernel", [3, 5, 7])
def test_pool_closed_forms(oracle_lib, kernel):
    half, n, a = kernel // 2, 40, 0.375
    y = oracle_lib.pool(np.full(n, a), kernel, 1)
    for j in range(n):
        cnt = min(j, half) + min(n - 1 - j, half) + 1
        assert y[j] == pytest.approx(a * cnt / kernel, rel=1e-15)
    spike = np.zeros(n)
    spike[17] = 2.5
    ym = oracle_lib.pool(spike, kernel, 0)
    assert np.array_equal(np.nonzero(ym)[0], np.arange(17 - half, 17 + half + 1))
    assert np.all(ym[17 - half:17 + half + 1] == 2.5)


# ---------------------------------------------------------------- top-N selection (Sec. 3.3)
@pytest.mark.parametrize("P", [0, 1, 2, 5, 9, 12])
def test_topk_matches_exhaustive_search(oracle_lib, P):
    rng = np.random.default_rng(P)
    c = rng.integers(0, 4, size=P).astype(np.float64)  # many ties, exact sums
    for k in range(P + 1):
        got = tuple(oracle_lib.topk(c, k))
        best = max(itertools.combinations(range(P), k),
                   key=lambda sub: (sum(c[list(sub)]), tuple(-i for i in sub)))
        assert got == best, (c, k, got, best)


def test_topk_uniform_input_takes_first_positions(oracle_lib):
    assert list(oracle_lib.topk(np.ones(20), 6)) == list(range(6))


# ---------------------------------------------------------------- the whole layer
def _tiny(name="tiny", **kw):
    base = dict(name=name, num_layers=2, num_q_heads=8, num_kv_heads=2, seqlens=(96,), window=8,
                heads_per_group=2, budget_mean=24, budget_uniform=True, pool_kernel=5, seed=7)
    base.update(kw)
    return cs.Workload(**base)


def _run(oracle_lib, wl, layer=0, mask=None, q=None, **kw):
    li = wl.layer(layer)
    m = wl.head_mask()[layer] if mask is None else mask
    return oracle_lib.compress_layer(
        li.q_win if q is None else q, li.k, li.v, wl.cu_seqlens(), m, int(wl.budgets()[layer]),
        wl.window, wl.pool_kernel, 0 if wl.pool_type == "max" else 1,
        0 if wl.head_order == "pool_then_sum" else 1, **kw), li, m


@pytest.mark.parametrize("pool_type", ["max", "avg"])
@pytest.mark.parametrize("head_order", ["pool_then_sum", "sum_then_pool"])
@pytest.mark.parametrize("hpg", [1, 2, 4])
def test_layer_matches_independent_pipeline(oracle_lib, pool_type, head_order, hpg):
    wl = _tiny(pool_type=pool_type, head_order=head_order, heads_per_group=hpg,
               seqlens=(96, 40, 120), budget_mean=30)
    out, li, m = _run(oracle_lib, wl)
    pooled, kept = ind.compress_layer_reference(
        li.q_win, li.k, li.v, wl.cu_seqlens(), m, 30, wl.window, wl.pool_kernel,
        0 if pool_type == "max" else 1, 0 if head_order == "pool_then_sum" else 1)
    cu, ck = wl.cu_seqlens(), out["cu_keep"]
    for s in range(wl.num_seqs):
        P = wl.seqlens[s] - wl.window
        for g in range(wl.num_kv_heads):
            np.testing.assert_allclose(out["pooled"][g, cu[s]:cu[s] + P],
                                       pooled[g, cu[s]:cu[s] + P], rtol=1e-11)
            np.testing.assert_array_equal(out["idx"][g, ck[s]:ck[s + 1]], kept[(s, g)])


def test_all_heads_selected_is_snapkv_group_aggregation(oracle_lib):
    """With every head selected the step is SnapKV's per-group aggregation (Sec. 2.1.1)."""
    wl = _tiny(heads_per_group=4)
    out, li, m = _run(oracle_lib, wl, mask=np.ones(8, np.uint8))
    pooled, kept = ind.compress_layer_reference(li.q_win, li.k, li.v, wl.cu_seqlens(),
                                                np.ones(8, np.uint8), 24, 8, 5, 0, 0)
    for g in range(2):
        np.testing.assert_array_equal(out["idx"][g], kept[(0, g)])


def test_budget_at_least_length_keeps_everything(oracle_lib):
    wl = _tiny(seqlens=(96, 24, 8, 3), budget_mean=96)
    out, li, _ = _run(oracle_lib, wl)
    cu = wl.cu_seqlens()
    np.testing.assert_array_equal(out["cu_keep"], cu)
    for s in range(wl.num_seqs):
        for g in range(2):
            np.testing.assert_array_equal(out["idx"][g, cu[s]:cu[s + 1]], np.arange(wl.seqlens[s]))
    np.testing.assert_array_equal(out["k_out"], li.k)
    np.testing.assert_array_equal(out["v_out"], li.v)


def test_window_always_kept_and_sizes(oracle_lib):
    wl = _tiny(seqlens=(96, 33, 8, 9), budget_mean=8)  # k = 0 candidates: only the window
    out, _, _ = _run(oracle_lib, wl)
    ck = out["cu_keep"]
    assert list(np.diff(ck)) == [8, 8, 8, 8]
    for s, L in enumerate(wl.seqlens):
        for g in range(2):
            np.testing.assert_array_equal(out["idx"][g, ck[s]:ck[s + 1]], np.arange(L - 8, L))
    wl = _tiny(seqlens=(200, 57), budget_mean=20)
    out, _, _ = _run(oracle_lib, wl)
    ck = out["cu_keep"]
    for s, L in enumerate(wl.seqlens):
        for g in range(2):
            ix = out["idx"][g, ck[s]:ck[s + 1]]
            assert len(ix) == 20 and np.all(np.diff(ix) > 0)
            assert set(range(L - 8, L)) <= set(ix.tolist())


def test_kept_rows_are_the_input_rows(oracle_lib):
    wl = _tiny(seqlens=(96, 50), budget_mean=20)
    out, li, _ = _run(oracle_lib, wl)
    cu, ck = wl.cu_seqlens(), out["cu_keep"]
    for s in range(2):
        for g in range(2):
            rows = cu[s] + out["idx"][g, ck[s]:ck[s + 1]]
            np.testing.assert_array_equal(out["k_out"][ck[s]:ck[s + 1], g], li.k[rows, g])
            np.testing.assert_array_equal(out["v_out"][ck[s]:ck[s + 1], g], li.v[rows, g])


def test_planted_span_is_recovered(oracle_lib):
    """Keys aligned with the selected heads' window queries must survive compression."""
    wl = _tiny(seqlens=(512,), budget_mean=40, plant="span", plant_count=16, plant_beta=4.0,
               plant_noise=True, outlier_channels=2, num_layers=3)
    for layer in range(3):
        out, li, _ = _run(oracle_lib, wl, layer=layer)
        span = set(li.planted[0].tolist())
        for g in range(2):
            assert span <= set(out["idx"][g].tolist())


def test_unselected_heads_do_not_matter(oracle_lib):
    wl = _tiny(seqlens=(96, 61))
    out, li, m = _run(oracle_lib, wl)
    q = li.q_win.copy()
    q[:, :, m == 0, :] = 0x7FC0  # NaN
    out2, _, _ = _run(oracle_lib, wl, q=q)
    for key in ("scores", "pooled", "idx", "k_out", "v_out"):
        np.testing.assert_array_equal(out[key], out2[key])


def test_permuting_heads_within_a_group(oracle_lib):
    wl = _tiny(seqlens=(96,), heads_per_group=2)
    out, li, m = _run(oracle_lib, wl)
    perm = np.array([2, 0, 3, 1, 5, 7, 4, 6])  # stays inside groups {0..3}, {4..7}
    out2, _, _ = _run(oracle_lib, wl, mask=m[perm], q=li.q_win[:, :, perm, :])
    np.testing.assert_allclose(out2["pooled"], out["pooled"], rtol=1e-14)
    np.testing.assert_array_equal(out2["idx"], out["idx"])


def test_head_orders_agree_for_average_pool_and_single_heads(oracle_lib):
    wl = _tiny(pool_type="avg", seqlens=(96, 70))
    a, _, _ = _run(oracle_lib, wl)
    b, _, _ = _run(oracle_lib, wl.with_(head_order="sum_then_pool"))
    np.testing.assert_allclose(a["pooled"], b["pooled"], rtol=1e-13)
    wl = _tiny(heads_per_group=1, seqlens=(96, 70))
    a, _, _ = _run(oracle_lib, wl)
    b, _, _ = _run(oracle_lib, wl.with_(head_order="sum_then_pool"))
    np.testing.assert_array_equal(a["pooled"], b["pooled"])
    np.testing.assert_array_equal(a["idx"], b["idx"])


def test_varlen_batch_equals_separate_sequences(oracle_lib):
    wl = _tiny(seqlens=(96, 40, 8, 3, 120), budget_mean=20)
    out, li, m = _run(oracle_lib, wl)
    cu, ck = wl.cu_seqlens(), out["cu_keep"]
    for s in range(wl.num_seqs):
        one = oracle_lib.compress_layer(li.q_win[s:s + 1], li.k[cu[s]:cu[s + 1]],
                                        li.v[cu[s]:cu[s + 1]], np.array([0, wl.seqlens[s]]),
                                        m, 20, 8, 5, 0, 0)
        np.testing.assert_array_equal(one["idx"], out["idx"][:, ck[s]:ck[s + 1]])
        np.testing.assert_array_equal(one["scores"], out["scores"][:, cu[s]:cu[s + 1]])


def test_rejects_bad_arguments(oracle_lib):
    wl = _tiny()
    li = wl.layer(0)
    m = wl.head_mask()[0]
    with pytest.raises(ValueError):  # budget below the window
        oracle_lib.compress_layer(li.q_win, li.k, li.v, wl.cu_seqlens(), m, 4, 8, 5, 0, 0)
    with pytest.raises(ValueError):  # even pool kernel
        oracle_lib.compress_layer(li.q_win, li.k, li.v, wl.cu_seqlens(), m, 24, 8, 4, 0, 0)
    bad = m.copy()
    bad[:4] = 0                      # a group without a selected head
    with pytest.raises(ValueError):
        oracle_lib.compress_layer(li.q_win, li.k, li.v, wl.cu_seqlens(), bad, 24, 8, 5, 0, 0)


# ---------------------------------------------------------------- layer scope (Sec. 3.3 as printed)
@pytest.mark.parametrize("pool_type", ["max", "avg"])
@pytest.mark.parametrize("head_order", ["pool_then_sum", "sum_then_pool"])
def test_layer_scope_matches_independent_pipeline(oracle_lib, pool_type, head_order):
    """One vector per sequence from every selected head, each against its own group's keys."""
    wl = _tiny(pool_type=pool_type, head_order=head_order, seqlens=(96, 40, 120), budget_mean=30)
    mask = np.array([0, 1, 1, 0, 0, 0, 1, 1], np.uint8)  # 4 heads over the two groups
    out, li, m = _run(oracle_lib, wl, mask=mask, scope=oracle_lib.SCOPE_LAYER)
    pooled, kept = ind.compress_layer_reference(
        li.q_win, li.k, li.v, wl.cu_seqlens(), mask, 30, wl.window, wl.pool_kernel,
        0 if pool_type == "max" else 1, 0 if head_order == "pool_then_sum" else 1, scope=1)
    cu, ck = wl.cu_seqlens(), out["cu_keep"]
    assert out["pooled"].shape[0] == 1
    for s in range(wl.num_seqs):
        P = wl.seqlens[s] - wl.window
        np.testing.assert_allclose(out["pooled"][0, cu[s]:cu[s] + P], pooled[0, cu[s]:cu[s] + P],
                                   rtol=1e-11)
        for g in range(wl.num_kv_heads):  # the same positions for every KV head
            np.testing.assert_array_equal(out["idx"][g, ck[s]:ck[s + 1]], kept[(s, 0)])
    for g in range(wl.num_kv_heads):  # each KV head's own rows at those positions
        for s in range(wl.num_seqs):
            rows = cu[s] + out["idx"][g, ck[s]:ck[s + 1]]
            np.testing.assert_array_equal(out["k_out"][ck[s]:ck[s + 1], g], li.k[rows, g])
            np.testing.assert_array_equal(out["v_out"][ck[s]:ck[s + 1], g], li.v[rows, g])


def test_layer_scope_vector_is_the_sum_of_the_groups_vectors(oracle_lib):
    wl = _tiny(seqlens=(150, 70), budget_mean=40)
    mask = np.array([1, 0, 1, 0, 0, 1, 0, 1], np.uint8)  # both groups have selected heads
    per_group, _, _ = _run(oracle_lib, wl, mask=mask)
    layer, _, _ = _run(oracle_lib, wl, mask=mask, scope=oracle_lib.SCOPE_LAYER)
    cu = wl.cu_seqlens()
    for s in range(wl.num_seqs):
        P = wl.seqlens[s] - wl.window
        a = per_group["pooled"][:, cu[s]:cu[s] + P].sum(axis=0)
        np.testing.assert_allclose(layer["pooled"][0, cu[s]:cu[s] + P], a, rtol=1e-12)


def test_layer_scope_with_one_kv_head_is_the_kv_head_scope(oracle_lib):
    wl = _tiny(num_q_heads=4, num_kv_heads=1, heads_per_group=2, seqlens=(120, 60), budget_mean=30)
    a, _, m = _run(oracle_lib, wl)
    b, _, _ = _run(oracle_lib, wl, mask=m, scope=oracle_lib.SCOPE_LAYER)
    for key in ("pooled", "idx", "k_out", "v_out", "cu_keep"):
        np.testing.assert_array_equal(a[key], b[key])


def test_layer_scope_allows_groups_without_selected_heads(oracle_lib):
    wl = _tiny(seqlens=(100,), budget_mean=30)
    mask = np.array([1, 1, 1, 0, 0, 0, 0, 0], np.uint8)  # every selected head in group 0
    with pytest.raises(ValueError):
        _run(oracle_lib, wl, mask=mask)  # the KV-head scope needs a head in every group
    out, li, _ = _run(oracle_lib, wl, mask=mask, scope=oracle_lib.SCOPE_LAYER)
    np.testing.assert_array_equal(out["idx"][0], out["idx"][1])
    assert len(set(out["idx"][0].tolist())) == 30
