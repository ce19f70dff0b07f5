"""Oracle of the cross-task slice planner -- TEST INFRASTRUCTURE, NOT PRODUCT CODE.

Only the test suite, the smoke check and the benchmark's CPU-baseline leg may
import this module.  It shares no code with the CUDA library.

Section 3.2.1 (fragmentation-aware expert grouping) groups the experts pooled
across tasks into ordered time slices.  Each expert i has a temporary memory
footprint w_i (the knapsack weight), a lifespan r_i, and the value
v_i = w_i / M_c - eta * r_i.  A 0/1 knapsack by dynamic programming,

    dp[i][j] = max(dp[i-1][j], dp[i-1][j - w_i] + v_i),

picks the slice that fits the budget M_c - M_s; the chosen experts leave the
candidate set and the DP runs again, until every expert is in a slice.

Readings (the paper prints the recurrence but not these details):
  * the items enter the DP in shortest-job-first order (lifespan ascending,
    index ascending), the paper's SJF bias; within a slice the experts keep
    that order;
  * dp[0][j] = 0 for every j ("at most j units used"), so dp[N][cap] is the
    optimum; an item is taken only when that is strictly better, so ties keep
    the smaller set;
  * if the DP picks nothing while experts remain (every remaining value <= 0),
    the first remaining expert in SJF order forms a slice of its own;
  * zero-footprint experts need no memory and join the first slice;
  * an expert heavier than the budget cannot be placed: the planner refuses
    (the caller treats it as unsupported).
The arithmetic of the values and of the DP sums is float64, in the order above.
"""
from __future__ import annotations

import numpy as np


def sjf_order(lifespan):
    return sorted(range(len(lifespan)), key=lambda i: (lifespan[i], i))


def plan_slices(weight, lifespan, capacity: int, eta: float = 0.0, budget: float | None = None):
    """Ordered slices (lists of item indices) of the items under `capacity`.

    weight: non-negative ints (memory units); lifespan: floats; capacity: the
    budget M_c - M_s in the same units; budget: M_c for the value term
    (defaults to capacity, i.e. M_s = 0)."""
    n = len(weight)
    w = [int(x) for x in weight]
    r = [float(x) for x in lifespan]
    cap = int(capacity)
    if any(x < 0 for x in w) or cap < 0:
        raise ValueError("negative weight or capacity")
    if any(x > cap for x in w):
        raise ValueError("an item does not fit the budget")
    mc = float(cap if budget is None else budget)
    v = [(w[i] / mc if mc > 0 else 0.0) - eta * r[i] for i in range(n)]
    order = sjf_order(r)
    zero = [i for i in order if w[i] == 0]
    remaining = [i for i in order if w[i] > 0]
    slices = []
    while remaining:
        m = len(remaining)
        dp = np.zeros(cap + 1, dtype=np.float64)
        take = np.zeros((m, cap + 1), dtype=bool)
        for a, i in enumerate(remaining):
            wi = w[i]
            cand = np.full(cap + 1, -np.inf)
            cand[wi:] = dp[:cap + 1 - wi] + v[i]
            t = cand > dp
            take[a] = t
            dp = np.where(t, cand, dp)
        chosen = []
        j = cap
        for a in range(m - 1, -1, -1):
            if take[a, j]:
                chosen.append(remaining[a])
                j -= w[remaining[a]]
        if not chosen:
            chosen = [remaining[0]]
        chosen_set = set(chosen)
        slices.append([i for i in remaining if i in chosen_set])
        remaining = [i for i in remaining if i not in chosen_set]
    if zero:
        if slices:
            slices[0] = zero + slices[0]
        else:
            slices = [zero]
    return slices


def slice_value(slice_items, weight, lifespan, capacity, eta=0.0, budget=None):
    mc = float(capacity if budget is None else budget)
    return sum((weight[i] / mc if mc > 0 else 0.0) - eta * lifespan[i] for i in slice_items)


def fill_clamp_refill(work, minimum, saturation, budget):
    """Resource shares of co-running experts (Section 3.2.2, lifespan-aware
    aligning): the controller's fill-clamp-refill allocation, real-valued.

      1. seed: every expert gets its minimum;
      2. fill: the budget left is shared out in proportion to the work
         coefficients of the experts not yet saturated;
      3. clamp: an expert above its saturation point is cut back to it, and what
         it gave up is shared out again over the others (step 2), until nothing
         is left or every expert with work is saturated.

    Readings (the paper gives the three steps, not their arithmetic):
      * an expert with no work (coefficient 0) keeps its minimum;
      * an expert whose share reaches its saturation exactly counts as clamped;
      * a budget below the sum of the minima is an error;
      * what is left when every expert with work is saturated stays unallocated.
    float64 throughout, sums in index order.  Returns (shares, unallocated)."""
    n = len(work)
    w = [float(x) for x in work]
    sat = [float(x) for x in saturation]
    a = [float(x) for x in minimum]
    if any(x < 0 for x in w) or any(a[i] < 0 or sat[i] < a[i] for i in range(n)):
        raise ValueError("negative work or minimum, or saturation below minimum")
    left = float(budget) - sum(a)
    if left < 0:
        raise ValueError("the minima exceed the budget")
    active = [i for i in range(n) if w[i] > 0 and a[i] < sat[i]]
    while left > 0 and active:
        wsum = 0.0
        for i in active:
            wsum += w[i]
        for i in active:
            a[i] += left * w[i] / wsum
        left = 0.0
        still = []
        for i in active:
            if a[i] >= sat[i]:
                left += a[i] - sat[i]
                a[i] = sat[i]
            else:
                still.append(i)
        active = still
    return a, left


def integer_shares(work, minimum, saturation, budget):
    """fill_clamp_refill rounded to whole units (CTAs): every share is floored,
    then the units still missing from the real-valued total go one each to the
    largest fractional parts (ties to the lower index).  A real share lies in
    [minimum, saturation], both integers, so the rounded one does too."""
    x, _ = fill_clamp_refill(work, minimum, saturation, budget)
    fl = [int(np.floor(v)) for v in x]
    total = int(round(sum(x)))
    missing = total - sum(fl)
    frac = sorted(range(len(x)), key=lambda i: (-(x[i] - fl[i]), i))
    for i in frac[:missing]:
        fl[i] += 1
    return fl
