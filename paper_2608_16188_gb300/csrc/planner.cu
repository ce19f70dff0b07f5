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

#include "planner.cuh"
#include "vmoe.h"

namespace vmoe {

int SlicePlanner::init(int n, const int64_t *weight, const double *lifespan, int64_t capacity, double eta,
                       double budget) {
    if (n < 0 || capacity < 0 || (n > 0 && (!weight || !lifespan))) return VMOE_ERR_INVALID;
    for (int i = 0; i < n; ++i) {
        if (weight[i] < 0 || !(lifespan[i] == lifespan[i])) return VMOE_ERR_INVALID;
        if (weight[i] > capacity) return VMOE_ERR_UNSUPPORTED;
    }
    if (capacity >= (1 << 24) || (int64_t)n * (capacity + 1) > ((int64_t)1 << 30))
        return VMOE_ERR_UNSUPPORTED;  // DP table too large
    weight_ = weight;
    n_ = n;
    cap_ = (int)capacity;
    first_ = true;
    const double mc = budget > 0.0 ? budget : (double)capacity;
    v_.assign(n, 0.0);
    for (int i = 0; i < n; ++i) v_[i] = (mc > 0.0 ? (double)weight[i] / mc : 0.0) - eta * lifespan[i];
    std::vector<int> sjf(n);
    std::iota(sjf.begin(), sjf.end(), 0);
    std::stable_sort(sjf.begin(), sjf.end(), [&](int a, int b) { return lifespan[a] < lifespan[b]; });
    zero_.clear();
    remaining_.clear();
    for (int i : sjf) (weight[i] == 0 ? zero_ : remaining_).push_back(i);
    // Two DP rows, row a-1 (cur) -> row a (nxt): every entry of row a depends on
    // row a-1 only, so the update is branch-free and vectorises; the decision
    // table gets every entry written, so it needs no clearing.
    cur_.assign(cap_ + 1, 0.0);
    nxt_.assign(cap_ + 1, 0.0);
    chosen_.assign(n, 0);
    take_.reset(new uint8_t[(size_t)(remaining_.size() > 0 ? remaining_.size() : 1) * (cap_ + 1)]);
    return VMOE_OK;
}

bool SlicePlanner::next(std::vector<int> &slice) {
    slice.clear();
    const bool first = first_;
    first_ = false;
    if (first) slice = zero_;  // zero-footprint experts join the first slice
    if (remaining_.empty()) return first && n_ > 0;
    const int m = (int)remaining_.size(), cap = cap_;
    std::fill(cur_.begin(), cur_.end(), 0.0);
    for (int a = 0; a < m; ++a) {
        const int i = remaining_[a];
        const int wi = (int)weight_[i];
        const double vi = v_[i];
        uint8_t *__restrict__ t = take_.get() + (size_t)a * (cap + 1);
        const double *__restrict__ o = cur_.data();
        double *__restrict__ nw = nxt_.data();
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
        cur_.swap(nxt_);
    }
    int nchosen = 0;
    for (int a = m - 1, j = cap; a >= 0; --a)
        if (take_[(size_t)a * (cap + 1) + j]) {
            chosen_[remaining_[a]] = 1;
            ++nchosen;
            j -= (int)weight_[remaining_[a]];
        }
    if (nchosen == 0) chosen_[remaining_[0]] = 1;  // an empty choice: the first expert alone
    std::vector<int> rest;
    for (int i : remaining_) {
        if (chosen_[i]) {
            slice.push_back(i);
            chosen_[i] = 0;
        } else {
            rest.push_back(i);
        }
    }
    remaining_.swap(rest);
    return true;
}

int plan_slices(int n, const int64_t *weight, const double *lifespan, int64_t capacity, double eta,
                double budget, int32_t *order, int32_t *slice_start) {
    if (n < 0 || (n > 0 && !order) || !slice_start) return VMOE_ERR_INVALID;
    SlicePlanner planner;
    const int st = planner.init(n, weight, lifespan, capacity, eta, budget);
    if (st != VMOE_OK) return st;
    std::vector<int> slice;
    int pos = 0, ns = 0;
    while (planner.next(slice)) {
        slice_start[ns++] = pos;
        for (int i : slice) order[pos++] = i;
    }
    slice_start[ns] = pos;
    return ns;
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
