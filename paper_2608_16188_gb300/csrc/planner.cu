// planner.cu -- the cross-task slice planner (host code): Section 3.2.1
// groups the experts pooled across tasks into ordered time slices that fit a
// memory budget, by a 0/1-knapsack dynamic programme over each expert's
// temporary footprint w_i (the weight) and the value
//     v_i = w_i / M_c - eta * r_i          (r_i: the expert's lifespan),
//     dp[i][j] = max(dp[i-1][j], dp[i-1][j - w_i] + v_i),
// run again over the experts left until all are placed.  The library uses it to
// run the expert backward in slices whose dH fits a caller's workspace.
//
// Readings: the experts enter the DP in shortest-job-first order (lifespan,
// then index), the paper's SJF bias, and keep that order inside a slice;
// dp[0][j] = 0 for all j (capacity used at most j), an expert is taken only
// when that is strictly better; an empty choice while experts remain places
// the first remaining expert alone; zero-footprint experts join the first
// slice; an expert heavier than the budget is refused.
#include <stdint.h>

#include <math.h>

#include <algorithm>
#include <memory>
#include <numeric>
#include <vector>

#include "vmoe.h"

namespace vmoe {

int plan_slices(int n, const int64_t *weight, const double *lifespan, int64_t capacity, double eta,
                double budget, int32_t *order, int32_t *slice_start) {
    if (n < 0 || capacity < 0 || (n > 0 && (!weight || !lifespan || !order || !slice_start)))
        return VMOE_ERR_INVALID;
    if (!slice_start) return VMOE_ERR_INVALID;
    for (int i = 0; i < n; ++i) {
        if (weight[i] < 0 || !(lifespan[i] == lifespan[i])) return VMOE_ERR_INVALID;
        if (weight[i] > capacity) return VMOE_ERR_UNSUPPORTED;
    }
    if (capacity >= (1 << 24) || (int64_t)n * (capacity + 1) > ((int64_t)1 << 30))
        return VMOE_ERR_UNSUPPORTED;  // DP table too large
    const int cap = (int)capacity;
    const double mc = budget > 0.0 ? budget : (double)capacity;
    std::vector<double> v(n);
    for (int i = 0; i < n; ++i) v[i] = (mc > 0.0 ? (double)weight[i] / mc : 0.0) - eta * lifespan[i];
    std::vector<int> sjf(n);
    std::iota(sjf.begin(), sjf.end(), 0);
    std::stable_sort(sjf.begin(), sjf.end(), [&](int a, int b) { return lifespan[a] < lifespan[b]; });
    std::vector<int> zero, remaining;
    for (int i : sjf) (weight[i] == 0 ? zero : remaining).push_back(i);

    std::vector<std::vector<int>> slices;
    // Two DP rows, row a-1 (cur) -> row a (nxt): every entry of row a depends on
    // row a-1 only, so the update is branch-free and vectorises; the decision
    // table gets every entry written, so it needs no clearing.
    std::vector<double> cur(cap + 1), nxt(cap + 1);
    std::unique_ptr<uint8_t[]> take(new uint8_t[(size_t)n * (cap + 1)]);
    while (!remaining.empty()) {
        const int m = (int)remaining.size();
        std::fill(cur.begin(), cur.end(), 0.0);
        for (int a = 0; a < m; ++a) {
            const int i = remaining[a];
            const int wi = (int)weight[i];
            const double vi = v[i];
            uint8_t *__restrict__ t = take.get() + (size_t)a * (cap + 1);
            const double *__restrict__ o = cur.data();
            double *__restrict__ nw = nxt.data();
            for (int j = 0; j < wi; ++j) {
                nw[j] = o[j];
                t[j] = 0;
            }
            for (int j = wi; j <= cap; ++j) {  // taken only when strictly better
                const double cand = o[j - wi] + vi;
                const bool tk = cand > o[j];
                nw[j] = tk ? cand : o[j];
                t[j] = tk;
            }
            cur.swap(nxt);
        }
        std::vector<uint8_t> chosen(n, 0);
        int nchosen = 0;
        for (int a = m - 1, j = cap; a >= 0; --a)
            if (take[(size_t)a * (cap + 1) + j]) {
                chosen[remaining[a]] = 1;
                ++nchosen;
                j -= (int)weight[remaining[a]];
            }
        if (nchosen == 0) chosen[remaining[0]] = 1;
        std::vector<int> slice, rest;
        for (int i : remaining) (chosen[i] ? slice : rest).push_back(i);
        slices.push_back(std::move(slice));
        remaining.swap(rest);
    }
    if (!zero.empty()) {
        if (slices.empty()) slices.push_back({});
        slices[0].insert(slices[0].begin(), zero.begin(), zero.end());
    }
    int pos = 0;
    for (size_t s = 0; s < slices.size(); ++s) {
        slice_start[s] = pos;
        for (int i : slices[s]) order[pos++] = i;
    }
    slice_start[slices.size()] = pos;
    return (int)slices.size();
}

// Section 3.2.2 (lifespan-aware aligning): the fill-clamp-refill allocation of a
// budget of resources among co-running experts -- seed each with its minimum,
// share the rest out in proportion to the work coefficients of the experts not
// yet saturated, clamp those above their saturation and share out again what
// they gave up -- then rounded to whole units: shares floored, the units still
// missing from the real-valued total to the largest fractional parts (ties to
// the lower index).  Readings: an expert with no work keeps its minimum; one
// that reaches its saturation exactly counts as clamped; what is left once
// every expert with work is saturated stays unallocated.  float64, sums in
// index order.  Returns the number of units allocated.
int plan_shares(int n, const double *work, const int32_t *minimum, const int32_t *saturation,
                int32_t budget, int32_t *shares) {
    if (n < 0 || budget < 0 || (n > 0 && (!work || !minimum || !saturation || !shares)))
        return VMOE_ERR_INVALID;
    std::vector<double> a(n);
    double msum = 0.0;
    for (int i = 0; i < n; ++i) {
        if (!(work[i] >= 0.0) || minimum[i] < 0 || saturation[i] < minimum[i]) return VMOE_ERR_INVALID;
        a[i] = (double)minimum[i];
        msum += a[i];
    }
    double left = (double)budget - msum;
    if (left < 0.0) return VMOE_ERR_UNSUPPORTED;  // the minima exceed the budget
    std::vector<int> active, still;
    for (int i = 0; i < n; ++i)
        if (work[i] > 0.0 && a[i] < (double)saturation[i]) active.push_back(i);
    while (left > 0.0 && !active.empty()) {
        double wsum = 0.0;
        for (int i : active) wsum += work[i];
        for (int i : active) a[i] += left * work[i] / wsum;
        left = 0.0;
        still.clear();
        for (int i : active) {
            const double s = (double)saturation[i];
            if (a[i] >= s) {
                left += a[i] - s;
                a[i] = s;
            } else {
                still.push_back(i);
            }
        }
        active.swap(still);
    }
    double xsum = 0.0;
    int64_t fsum = 0;
    std::vector<int> idx(n);
    for (int i = 0; i < n; ++i) {
        xsum += a[i];
        shares[i] = (int32_t)std::floor(a[i]);
        fsum += shares[i];
        idx[i] = i;
    }
    const int64_t total = std::llround(xsum);
    std::stable_sort(idx.begin(), idx.end(),
                     [&](int p, int q) { return a[p] - shares[p] > a[q] - shares[q]; });
    for (int64_t r = 0; r < total - fsum && r < n; ++r) shares[idx[r]] += 1;
    return (int)total;
}

}  // namespace vmoe

extern "C" int vmoe_plan_shares(int n, const double *work, const int32_t *minimum,
                                const int32_t *saturation, int32_t budget, int32_t *shares) {
    return vmoe::plan_shares(n, work, minimum, saturation, budget, shares);
}

extern "C" int vmoe_plan_slices(int n, const int64_t *weight, const double *lifespan,
                                int64_t capacity, double eta, double budget, int32_t *order,
                                int32_t *slice_start) {
    return vmoe::plan_slices(n, weight, lifespan, capacity, eta, budget, order, slice_start);
}
