"""Pins of the budget oracle (oracle/budgets.py) against values worked out by hand from
Algorithm 1 and Eq. 11-13 of App. B, and against properties the algorithm guarantees."""
import random

import pytest

from oracle import budgets as ob


def test_proportional_share_with_a_rounding_tie_then_one_token_back():
    # m=10 each, R = 100 - 30 = 70: 35, 17.5 -> 18 (ties to even), 17.5 -> 18; sum 101, so one
    # token comes back from the lowest score above m, the lower index of the two 0.25s.
    assert ob.allocate_budgets([0.5, 0.25, 0.25], 100, 10, 60) == [45, 27, 28]


def test_clipped_layer_passes_its_excess_to_the_next_highest_score():
    # R = 60: 42, 12, 6 -> [52 -> 40 (clip at M), 22, 16] = 78; the 12 left go one at a time
    # to the highest score still below M, layer 1.
    assert ob.allocate_budgets([0.7, 0.2, 0.1], 90, 10, 40) == [40, 34, 16]


def test_round_half_to_even_reading():
    # R = 1: round(0.5) = 0 for both, so one token is left and goes to the argmax with the
    # lower index.  (Ties away from zero would give [32, 33].)
    assert ob.allocate_budgets([0.5, 0.5], 65, 32, 96) == [33, 32]


def test_total_below_the_minimums_keeps_every_layer_at_m():
    assert ob.allocate_budgets([0.9, 0.1], 50, 32, 96) == [32, 32]


def test_total_above_the_maximums_stops_at_m_capital():
    assert ob.allocate_budgets([0.6, 0.4], 1000, 32, 96) == [96, 96]


def test_uniform_scores_split_evenly():
    assert ob.allocate_budgets([0.25] * 4, 4 * 256, 32, 768) == [256] * 4


def test_properties_on_random_scores():
    rng = random.Random(7)
    for _ in range(300):
        L = rng.randint(1, 40)
        raw = [rng.random() ** 3 for _ in range(L)]
        s = sum(raw)
        scores = [x / s for x in raw]
        mean = rng.choice([32, 64, 256, 1024])
        m, M = 32, 3 * mean
        total = L * mean + rng.randint(-L, L)
        B = ob.allocate_budgets(scores, total, m, M)
        assert all(m <= b <= M for b in B)
        if L * m <= total <= L * M:
            assert sum(B) == total
        for i in range(L):  # a higher score never gets a smaller budget
            for j in range(L):
                if scores[i] > scores[j]:
                    assert B[i] >= B[j]


def test_error_scores_worked_example():
    # Eq. 11: [1, 3] -> [0.25, 0.75]; [2, 2] -> [0.5, 0.5]; Eq. 12: mean [0.375, 0.625];
    # Eq. 13: already sums to 1.
    assert ob.layer_error_scores([[1.0, 3.0], [2.0, 2.0]]) == [0.375, 0.625]


def test_error_scores_ignore_each_datasets_scale_and_sum_to_one():
    rng = random.Random(3)
    errors = [[rng.random() for _ in range(12)] for _ in range(5)]
    a = ob.layer_error_scores(errors)
    scaled = [[x * (d + 1) * 10.0 for x in row] for d, row in enumerate(errors)]
    b = ob.layer_error_scores(scaled)
    assert abs(sum(a) - 1.0) < 1e-12
    assert all(abs(x - y) <= 1e-12 * max(abs(x), 1e-300) for x, y in zip(a, b))


def test_error_scores_single_dataset_is_its_l1_normalisation():
    e = [2.0, 6.0, 0.0, 12.0]
    assert ob.layer_error_scores([e]) == [0.1, 0.3, 0.0, 0.6]


@pytest.mark.parametrize("bad", [[[0.0, 0.0]], [[1.0, -1.0]], [[1.0, float("nan")]]])
def test_error_scores_reject_unusable_inputs(bad):
    with pytest.raises(ValueError):
        ob.layer_error_scores(bad)
