// planner.cuh -- the cross-task slice planner of Section 3.2.1 in incremental
// form (host code, internal): next() hands out the slices one at a time, in the
// order plan_slices gives them, so that a caller can run slice s on the GPU
// while the DP places the experts left for slice s + 1.
#pragma once

#include <stdint.h>

#include <memory>
#include <vector>

namespace vmoe {

class SlicePlanner {
public:
    // Checks the inputs and sorts the experts (VMOE_OK or an error status; see
    // plan_slices).  The arrays must stay valid until the last next().
    int init(int n, const int64_t *weight, const double *lifespan, int64_t capacity, double eta,
             double budget);
    // The next slice's experts, in SJF order (zero-footprint experts first in
    // the first slice); false once every expert is placed.
    bool next(std::vector<int> &slice);

private:
    const int64_t *weight_ = nullptr;
    int n_ = 0, cap_ = 0;
    bool first_ = true;
    std::vector<double> v_, cur_, nxt_;
    std::vector<int> zero_, remaining_;
    std::vector<uint8_t> chosen_;
    std::unique_ptr<uint8_t[]> take_;
};

int plan_slices(int n, const int64_t *weight, const double *lifespan, int64_t capacity, double eta,
                double budget, int32_t *order, int32_t *slice_start);

}  // namespace vmoe
