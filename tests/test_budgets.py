"""ckv_layer_error_scores and ckv_allocate_budgets (host entry points, no GPU) against the
oracle in oracle/budgets.py: budgets bit-exact, scores to a few ulps."""
import random

import numpy as np
import pytest

import paper_2508_02401_gb300 as ckv
from oracle import budgets as ob


@pytest.fixture(scope="module", autouse=True)
def _lib():
    ckv.load()


def _random_case(rng):
    L = rng.randint(1, 80)
    raw = [rng.random() ** rng.choice([1, 3, 6]) for _ in range(L)]
    if rng.random() < 0.3:  # equal scores, exact ties
        raw = [rng.choice([1.0, 2.0, 4.0]) for _ in range(L)]
    s = sum(raw)
    scores = [x / s for x in raw]
    mean = rng.choice([32, 64, 128, 256, 512, 1024, 3000])
    m = rng.choice([0, 8, 32])
    M = rng.choice([3 * mean, 2 * mean, mean + 1, 100000])
    M = max(M, m)
    total = L * mean + rng.randint(-2 * L, 2 * L) * rng.choice([1, 7, 50])
    return scores, total, m, M


def test_budgets_match_the_oracle_exactly():
    rng = random.Random(2025)
    for _ in range(2000):
        scores, total, m, M = _random_case(rng)
        got = ckv.ckv_allocate_budgets(scores, total, m, M)
        assert got.tolist() == ob.allocate_budgets(scores, total, m, M), (scores, total, m, M)


@pytest.mark.parametrize("case", [
    ([0.5, 0.25, 0.25], 100, 10, 60),
    ([0.7, 0.2, 0.1], 90, 10, 40),
    ([0.5, 0.5], 65, 32, 96),
    ([0.9, 0.1], 50, 32, 96),
    ([0.6, 0.4], 1000, 32, 96),
])
def test_budgets_on_the_pinned_cases(case):
    assert ckv.ckv_allocate_budgets(*case).tolist() == ob.allocate_budgets(*case)


def test_default_maximum_is_three_times_the_mean():
    s = np.full(32, 1 / 32)
    s[0] = 0.9
    s /= s.sum()
    b = ckv.ckv_allocate_budgets(s, 32 * 256)
    assert b.max() == 3 * 256 and b.min() >= 32 and b.sum() == 32 * 256


def test_error_scores_match_the_oracle():
    rng = random.Random(11)
    for _ in range(200):
        D, L = rng.randint(1, 6), rng.randint(1, 48)
        e = [[rng.random() * 10 ** rng.randint(-3, 3) for _ in range(L)] for _ in range(D)]
        got = ckv.ckv_layer_error_scores(np.array(e))
        ref = np.array(ob.layer_error_scores(e))
        np.testing.assert_allclose(got, ref, rtol=1e-14, atol=0)


@pytest.mark.parametrize("bad", [np.zeros((1, 3)), np.array([[1.0, -2.0]]), np.array([[np.inf, 1.0]])])
def test_error_scores_reject_unusable_inputs(bad):
    with pytest.raises(ckv.CkvError):
        ckv.ckv_layer_error_scores(bad)


@pytest.mark.parametrize("args", [([float("nan"), 0.5], 100, 32, 96), ([0.5, 0.5], 100, 40, 32),
                                  ([-0.1, 1.1], 100, 32, 96)])
def test_budgets_reject_unusable_inputs(args):
    with pytest.raises(ckv.CkvError):
        ckv.ckv_allocate_budgets(*args)
