"""Pins of the oracle's fill-clamp-refill allocation (CPU only).

Section 3.2.2 allocates a budget of resources among co-running experts: seed
each with its minimum, share out the rest in proportion to work coefficients,
clamp the saturated ones and share out what they gave up again.  Its fixed
point has a closed form: with lambda >= 0 such that the shares sum to the
budget, every expert with work gets min(saturation, minimum + lambda * work)
(an expert with no work keeps its minimum).  The tests find lambda by bisection
-- a different algorithm from the oracle's iteration -- and check the oracle
against it, against a hand-worked example, against its sums and bounds, and the
rounded shares against brute-force enumeration on small cases.
"""
import itertools
import json
import os
import random

import numpy as np
import pytest

from oracle import planner

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "shares_example.json")


def closed_form(work, minimum, saturation, budget):
    """min(sat, min + lam * w) with lam by bisection so that the total is the budget,
    or every expert with work saturated when the saturations do not reach it."""
    w = np.asarray(work, float)
    mn = np.asarray(minimum, float)
    sat = np.asarray(saturation, float)

    def shares(lam):
        return np.where(w > 0, np.minimum(sat, mn + lam * w), mn)
    if shares(1e18).sum() <= budget:
        return shares(1e18)
    lo, hi = 0.0, 1.0
    while shares(hi).sum() < budget:
        hi *= 2
    for _ in range(200):
        mid = 0.5 * (lo + hi)
        if shares(mid).sum() < budget:
            lo = mid
        else:
            hi = mid
    return shares(hi)


def test_hand_worked_example():
    g = json.load(open(GOLDEN))
    x, left = planner.fill_clamp_refill(g["work"], g["minimum"], g["saturation"], g["budget"])
    np.testing.assert_allclose(x, g["shares"], rtol=0, atol=1e-12)
    assert left == 0.0
    assert planner.integer_shares(g["work"], g["minimum"], g["saturation"], g["budget"]) == \
        g["integer_shares"]


def _random_case(rng):
    n = rng.randint(1, 12)
    work = [rng.choice([0.0, rng.random() * 10, float(rng.randint(1, 5))]) for _ in range(n)]
    minimum = [rng.randint(0, 3) for _ in range(n)]
    saturation = [m + rng.randint(0, 9) for m in minimum]
    budget = sum(minimum) + rng.randint(0, 40)
    return work, minimum, saturation, budget


@pytest.mark.parametrize("seed", range(200))
def test_matches_closed_form(seed):
    rng = random.Random(seed)
    work, minimum, saturation, budget = _random_case(rng)
    x, left = planner.fill_clamp_refill(work, minimum, saturation, budget)
    ref = closed_form(work, minimum, saturation, budget)
    np.testing.assert_allclose(x, ref, rtol=0, atol=1e-9)
    # sums and bounds
    cap = sum(s if w > 0 else m for w, m, s in zip(work, minimum, saturation))
    assert abs(sum(x) - min(budget, cap)) < 1e-9
    assert abs(left - (budget - min(budget, cap))) < 1e-9
    assert all(m - 1e-12 <= v <= s + 1e-12 for v, m, s in zip(x, minimum, saturation))


def test_proportional_when_nothing_saturates():
    x, _ = planner.fill_clamp_refill([3, 1, 2], [1, 2, 0], [100, 100, 100], 15)
    np.testing.assert_allclose(x, [1 + 6, 2 + 2, 0 + 4], atol=1e-12)  # 12 left, shared 3:1:2


def test_equal_work_equal_shares_and_refused_budget():
    x, _ = planner.fill_clamp_refill([2, 2, 2, 2], [1, 1, 1, 1], [9, 9, 9, 9], 10)
    np.testing.assert_allclose(x, [2.5] * 4, atol=1e-12)
    with pytest.raises(ValueError):
        planner.fill_clamp_refill([1, 1], [3, 3], [5, 5], 5)  # minima above the budget


@pytest.mark.parametrize("seed", range(60))
def test_integer_shares_brute_force(seed):
    """Rounded shares: within one unit of the real ones, the same total, inside
    [minimum, saturation], and nearest to the real shares (least squares) among
    all integer vectors with that total and those bounds."""
    rng = random.Random(1000 + seed)
    n = rng.randint(1, 5)
    work = [rng.choice([0.0, rng.random() * 5]) for _ in range(n)]
    minimum = [rng.randint(0, 2) for _ in range(n)]
    saturation = [m + rng.randint(0, 4) for m in minimum]
    budget = sum(minimum) + rng.randint(0, 12)
    x, _ = planner.fill_clamp_refill(work, minimum, saturation, budget)
    a = planner.integer_shares(work, minimum, saturation, budget)
    total = int(round(sum(x)))
    assert sum(a) == total
    assert all(m <= v <= s for v, m, s in zip(a, minimum, saturation))
    assert all(abs(v - r) < 1 for v, r in zip(a, x))
    best = min(sum((c - r) ** 2 for c, r in zip(cand, x))
               for cand in itertools.product(*[range(m, s + 1) for m, s in zip(minimum, saturation)])
               if sum(cand) == total)
    assert sum((c - r) ** 2 for c, r in zip(a, x)) <= best + 1e-9
