"""Layer budgets of the paper's error-aware allocation -- TEST INFRASTRUCTURE ONLY.

Plain Python, one step of the definition per line, for the tests to check the library's
``ckv_layer_error_scores`` and ``ckv_allocate_budgets`` against.  Nothing in the product
imports this module.

* ``layer_error_scores``: App. B, Eq. 11-13 -- each dataset's per-layer errors are
  L1-normalised over the layers, the normalised errors are averaged over the datasets, and the
  average is L1-normalised again.
* ``allocate_budgets``: Algorithm 1 (App. B) -- every layer starts at the minimum m, the rest of
  the total is handed out in proportion to the scores (rounded, then clipped to [m, M]), and the
  difference left by rounding and clipping is settled one token at a time: added to the
  highest-scoring layer still below M, or taken from the lowest-scoring layer still above m.

Readings (the paper does not say):
* round() takes ties to the even integer, as numpy and PyTorch do;
* argmax / argmin take the lowest layer index among equal scores, as numpy does;
* a dataset whose errors sum to 0, negative or non-finite errors, or scores that sum to 0 are
  rejected (ValueError) instead of dividing by zero.
"""
from __future__ import annotations

import math


def layer_error_scores(errors):
    """errors[d][l] = e_d^(l) (Eq. 10); returns the scores e~^(l) of Eq. 13 as a list."""
    D = len(errors)
    if D == 0:
        raise ValueError("no datasets")
    L = len(errors[0])
    for row in errors:
        if len(row) != L:
            raise ValueError("ragged errors")
        for x in row:
            if not math.isfinite(x) or x < 0:
                raise ValueError("errors must be finite and non-negative")
    # Eq. 11: per dataset, divide by the sum over layers
    normalised = []
    for row in errors:
        total = 0.0
        for x in row:
            total += x
        if total == 0.0:
            raise ValueError("a dataset's errors sum to 0")
        normalised.append([x / total for x in row])
    # Eq. 12: mean over datasets
    mean = []
    for l in range(L):
        acc = 0.0
        for d in range(D):
            acc += normalised[d][l]
        mean.append(acc / D)
    # Eq. 13: divide by the sum over layers
    total = 0.0
    for x in mean:
        total += x
    if total == 0.0:
        raise ValueError("scores sum to 0")
    return [x / total for x in mean]


def _round_half_even(x: float) -> int:
    return int(round(x))  # Python's round() takes ties to even


def allocate_budgets(scores, total_budget: int, m: int, M: int):
    """Algorithm 1: per-layer budgets (list of int) from the scores e~ (non-negative)."""
    L = len(scores)
    for s in scores:
        if not math.isfinite(s) or s < 0:
            raise ValueError("scores must be finite and non-negative")
    if m < 0 or M < m:
        raise ValueError("need 0 <= m <= M")
    B = [m] * L                                   # B_i <- m
    R = total_budget - sum(B)                     # R <- B_total - sum_i B_i
    for i in range(L):                            # B_i <- clip(B_i + round(e_i R), m, M)
        B[i] = min(max(B[i] + _round_half_even(scores[i] * R), m), M)
    delta = total_budget - sum(B)                 # Delta <- B_total - sum_i B_i
    while delta != 0:
        if delta > 0:
            eligible = [i for i in range(L) if B[i] < M]
            if not eligible:
                break
            j = eligible[0]
            for i in eligible:                    # argmax, lowest index on ties
                if scores[i] > scores[j]:
                    j = i
            B[j] += 1
            delta -= 1
        else:
            eligible = [i for i in range(L) if B[i] > m]
            if not eligible:
                break
            j = eligible[0]
            for i in eligible:                    # argmin, lowest index on ties
                if scores[i] < scores[j]:
                    j = i
            B[j] -= 1
            delta += 1
    return B
