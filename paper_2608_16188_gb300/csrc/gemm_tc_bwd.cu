// gemm_tc_bwd.cu -- backward launches of the tcgen05 grouped GEMM:
//   dA + GELU': dH = (dYe W2^T) * GELU'(H)  (A: dYe K-major; B: W2 [f,d] read K-major)
//   dX:         dXe = dH W1^T               (A: dH K-major;  B: W1 [d,f] read K-major)
//   dW1:        dW1 = Xe^T dH               (both MN-major, K = load)
//   dW2:        dW2 = A^T dYe               (both MN-major, K = load)
#include "gemm_tc.cuh"

namespace vmoe {

using namespace tc;

int launch_expert_bwd_bf16(const Dims &p, const __nv_bfloat16 *xe, const __nv_bfloat16 *h,
                           const __nv_bfloat16 *act, const __nv_bfloat16 *w1,
                           const __nv_bfloat16 *w2, const __nv_bfloat16 *dye,
                           const int32_t *load, __nv_bfloat16 *dxe, __nv_bfloat16 *dw1,
                           __nv_bfloat16 *dw2, __nv_bfloat16 *dh, cudaStream_t s) {
    // dH is kept as a bf16 pair: the workspace holds, per group, dH_hi in rows
    // [0, C) and the residual dH_lo = dH - dH_hi in rows [C, 2C).  dX uses dH_hi;
    // dW1 = Xe^T dH_hi + Xe^T dH_lo, which keeps short weight-gradient sums
    // (groups with a few rows, where terms cancel) at fp32-like accuracy.
    const long long C = p.C, f = p.f;
    __nv_bfloat16 *dh_hi = dh, *dh_lo = dh + C * f;
    int st = row_gemm<EPI_DGELU, false>(p, dye, p.d, w2, p.f, load, dh_hi, dh_lo, h, s,
                                        "tc_da_dgelu", 2 * C * f, C * f);
    if (st != VMOE_OK) return st;
    if ((st = row_gemm<EPI_STORE, false>(p, dh_hi, p.f, w1, p.d, load, dxe, nullptr, nullptr, s,
                                         "tc_dx", 0, 0, 2 * C * f)) != VMOE_OK)
        return st;
    if ((st = wgrad_gemm(p, xe, p.d, dh, p.f, load, dw1, s, "tc_dw1", true)) != VMOE_OK) return st;
    return wgrad_gemm(p, act, p.f, dye, p.d, load, dw2, s, "tc_dw2");
}

}  // namespace vmoe
