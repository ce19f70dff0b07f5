// topk.cuh -- softmax + top-k gating of one token's logit row (Section 2.1
// routing), shared by the router kernels (internal).
#pragma once

#include <math.h>

#include "common.cuh"

namespace vmoe {

// One token: the max, the softmax denominator, then k picks, each the best
// expert that comes after the previous pick in the order (larger logit first,
// equal logits by lower index).  NaN is treated as -inf so the chosen indices
// stay in range.  Writes idx and gate of token `tok` (= t * N + n); the gates
// are renormalised over the k picks unless VMOE_NO_RENORM.
__device__ __forceinline__ void topk_row(const Dims &p, const float *row, long long tok,
                                         int32_t *__restrict__ out_idx,
                                         float *__restrict__ out_gate) {
    const int E = p.E;
    const bool renorm = !(p.flags & VMOE_NO_RENORM);
    float mx = -INFINITY;
    for (int e = 0; e < E; ++e) {
        float v = row[e];
        mx = fmaxf(mx, isnan(v) ? -INFINITY : v);
    }
    float sum = 0.0f;
    for (int e = 0; e < E; ++e) {
        float v = row[e];
        sum += expf((isnan(v) ? -INFINITY : v) - mx);
    }
    float ev[8];
    int ei[8];
    float pv = INFINITY;  // previous pick: (pv, pe); the next pick comes after it
    int pe = -1;
    float kept = 0.0f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        ev[j] = 0.0f;
        ei[j] = 0;
        if (j >= p.k) continue;
        float bv = -INFINITY;
        int be = -1;
        for (int e = 0; e < E; ++e) {
            float v = row[e];
            v = isnan(v) ? -INFINITY : v;
            const bool after = v < pv || (v == pv && e > pe);
            if (after && (be < 0 || v > bv)) {  // strict '>' keeps the lower index on ties
                bv = v;
                be = e;
            }
        }
        ei[j] = be;
        ev[j] = expf(bv - mx);
        kept += ev[j];
        pv = bv;
        pe = be;
    }
    const long long base = tok * p.k;
#pragma unroll
    for (int j = 0; j < 8; ++j)
        if (j < p.k) {
            out_idx[base + j] = ei[j];
            out_gate[base + j] = renorm ? ev[j] / kept : ev[j] / sum;
        }
}

}  // namespace vmoe
