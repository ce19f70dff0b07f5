"""Pins of the oracle's cross-task slice planner (CPU only).

The planner (Section 3.2.1) is a 0/1-knapsack DP iterated over the remaining
experts.  It is checked against brute-force enumeration of every subset on small
instances, a textbook knapsack instance with a known optimum, and the closed
forms of degenerate cases (equal weights: slices of floor(cap / w) experts, the
shortest jobs first when the lifespan term is on).
"""
import itertools
import random

import pytest

from oracle import planner


def _check_partition(slices, n, w, cap):
    seen = sorted(i for s in slices for i in s)
    assert seen == list(range(n))
    for s in slices:
        assert sum(w[i] for i in s) <= cap


@pytest.mark.parametrize("seed", range(40))
def test_first_slice_is_the_brute_force_optimum(seed):
    rng = random.Random(seed)
    n = rng.randint(1, 9)
    w = [rng.randint(0, 12) for _ in range(n)]
    r = [rng.choice([rng.random(), float(rng.randint(0, 3))]) for _ in range(n)]
    cap = max(w) + rng.randint(0, 20)
    eta = rng.choice([0.0, 0.05, 0.3])
    slices = planner.plan_slices(w, r, cap, eta)
    _check_partition(slices, n, w, cap)
    pos = [i for i in range(n) if w[i] > 0]
    best = -1.0
    for m in range(len(pos) + 1):
        for sub in itertools.combinations(pos, m):
            if sum(w[i] for i in sub) <= cap:
                best = max(best, planner.slice_value(sub, w, r, cap, eta))
    first = [i for i in slices[0] if w[i] > 0]
    got = planner.slice_value(first, w, r, cap, eta)
    if best > 1e-12:
        assert got == pytest.approx(best, rel=1e-12, abs=1e-12)
    else:  # nothing has positive value: the shortest remaining job alone
        order = planner.sjf_order(r)
        assert first == [next(i for i in order if w[i] > 0)] or not pos


def test_textbook_knapsack():
    # weights 1, 3, 4, 5 and values 1, 4, 5, 7 under capacity 7: optimum 9 = {3, 4}.
    # Values enter as -eta * lifespan with eta = -1 and a budget so large that the
    # utilisation term vanishes.
    w, vals = [1, 3, 4, 5], [1.0, 4.0, 5.0, 7.0]
    slices = planner.plan_slices(w, vals, 7, eta=-1.0, budget=1e300)
    assert sorted(slices[0]) == [1, 2]
    assert planner.slice_value(slices[0], w, vals, 7, -1.0, 1e300) == pytest.approx(9.0)
    _check_partition(slices, 4, w, 7)


def test_equal_weights_pack_full_slices_shortest_first():
    n, w0, cap = 23, 5, 21
    r = [float((7 * i) % n) for i in range(n)]  # a permutation of 0..22
    w = [w0] * n
    for eta in (0.0, 0.01):
        slices = planner.plan_slices(w, r, cap, eta)
        _check_partition(slices, n, w, cap)
        k = cap // w0
        assert [len(s) for s in slices] == [k] * (n // k) + ([n % k] if n % k else [])
    # with the lifespan term the slices come out in SJF order
    slices = planner.plan_slices(w, r, cap, 0.01)
    flat = [i for s in slices for i in s]
    assert [r[i] for i in flat] == sorted(r)


def test_zero_weights_join_the_first_slice_and_oversize_is_refused():
    slices = planner.plan_slices([0, 4, 0, 4], [3.0, 1.0, 0.0, 2.0], 4)
    assert slices == [[2, 0, 1], [3]]
    with pytest.raises(ValueError):
        planner.plan_slices([5], [1.0], 4)
