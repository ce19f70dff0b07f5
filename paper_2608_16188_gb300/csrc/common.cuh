// common.cuh -- shared declarations of the libvmoe CUDA sources (internal).
#pragma once

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>
#include <mutex>

#include <utility>

#include "vmoe.h"

namespace vmoe {

// Validated problem sizes, as the kernels see them.
struct Dims {
    int T, N, d, f, E, k, C;
    unsigned flags;
    bool bf16;
    int G() const { return T * E; }
};

// Host-side hooks (abi.cu).
void trace_before(cudaStream_t s, const char *kernel_name);
void trace_after(cudaStream_t s);
int *device_status_word();  // device address of the current device's status word, or NULL
int num_sms();              // SM count of the current device

// Returns VMOE_OK or VMOE_ERR_CUDA after a launch.
inline int launch_result() {
    cudaError_t e = cudaGetLastError();
    return e == cudaSuccess ? VMOE_OK : VMOE_ERR_CUDA;
}

// Programmatic dependent launch for the kernels of a step: each launches with
// programmatic stream serialisation and waits for its predecessor's results
// (pdl_wait) only after its own set-up -- barriers, TMEM, tensor-map prefetch.
// The grouped GEMMs let their successor launch once every CTA has reached its
// last tile (pdl_launch_dependents); the other kernels at exit.  Letting it
// launch at the start measured slower: the waiting CTAs of the successor hold
// warp slots and registers on every SM while the predecessor runs.
// On by default; the environment variable VMOE_PDL=0 turns it off.
bool pdl_enabled();  // abi.cu

// The SM-pair (cta_group::2) grouped GEMMs (abi.cu): the weight-gradient
// kernel, on unless VMOE_PAIR=0 in the environment; the row-mode kernel for
// groups above 128 rows, off unless VMOE_ROW_PAIR=1.
bool pair_enabled();
bool row_pair_enabled();
// The fill-clamp-refill pair shares of the memory-budgeted backward's dW1,
// off unless VMOE_SHARES=1 (abi.cu).
bool shares_enabled();
// The tcgen05 router for bf16 tokens (route_tc.cu), off unless
// VMOE_ROUTE_TC=1; problems it does not take use the mma.sync router.
bool route_tc_enabled();

template <typename... KArgs, typename... Args>
int launch_kernel(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                  Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 1 : 0;
    return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...) == cudaSuccess ? VMOE_OK
                                                                                    : VMOE_ERR_CUDA;
}

// Launchers (one file each).
int route_tc_width(const Dims &p);  // 0: the tcgen05 router does not take p
int launch_route_tc(const Dims &p, const __nv_bfloat16 *x, const float *wr, const float *bias, float *logits,
                    int32_t *idx, float *gate, cudaStream_t s);
int launch_route(const Dims &p, const void *x, const float *w_router, const float *bias,
                 float *logits, int32_t *idx, float *gate, int32_t *slot, int32_t *load,
                 cudaStream_t s);
int launch_dispatch(const Dims &p, const void *src, const float *weight, const int32_t *idx,
                    const int32_t *slot, const int32_t *load, void *dst, cudaStream_t s);
int launch_combine(const Dims &p, const void *src, const float *weight, const int32_t *idx,
                   const int32_t *slot, void *dst, cudaStream_t s);
int launch_expert_fwd_f32(const Dims &p, const float *xe, const float *w1, const float *w2,
                          const int32_t *load, float *h, float *a, float *ye, cudaStream_t s);
int launch_expert_bwd_f32(const Dims &p, const float *xe, const float *h, const float *a,
                          const float *w1, const float *w2, const float *dye,
                          const int32_t *load, float *dxe, float *dw1, float *dw2, float *dh,
                          cudaStream_t s);
int launch_expert_fwd_bf16(const Dims &p, const __nv_bfloat16 *xe, const __nv_bfloat16 *w1,
                           const __nv_bfloat16 *w2, const int32_t *load, __nv_bfloat16 *h,
                           __nv_bfloat16 *a, __nv_bfloat16 *ye, cudaStream_t s);
int launch_expert_bwd_bf16(const Dims &p, const __nv_bfloat16 *xe, const __nv_bfloat16 *h,
                           const __nv_bfloat16 *a, const __nv_bfloat16 *w1,
                           const __nv_bfloat16 *w2, const __nv_bfloat16 *dye,
                           const int32_t *load, __nv_bfloat16 *dxe, __nv_bfloat16 *dw1,
                           __nv_bfloat16 *dw2, __nv_bfloat16 *dh, cudaStream_t s);
// The expert backward under a dH budget (gemm_tc_bwd.cu): slices planned by
// the cross-task DP; `workspace` holds the plan, then the slices' dH.
size_t bwd_plan_bytes(const Dims &p);
size_t bwd_min_workspace(const Dims &p);
int launch_expert_bwd_bf16_sliced(const Dims &p, const __nv_bfloat16 *xe, const __nv_bfloat16 *h,
                                  const __nv_bfloat16 *act, const __nv_bfloat16 *w1,
                                  const __nv_bfloat16 *w2, const __nv_bfloat16 *dye,
                                  const int32_t *load, __nv_bfloat16 *dxe, __nv_bfloat16 *dw1,
                                  __nv_bfloat16 *dw2, void *workspace, size_t workspace_bytes,
                                  cudaStream_t s, int *nslices_out);
int launch_router_bwd(const Dims &p, const void *x, const float *w_router, const float *logits,
                      const int32_t *idx, const float *gate, const int32_t *slot, const void *dy,
                      const void *ye, float *dgate, float *dlogits, float *dw_router, float *dbias,
                      void *dx, cudaStream_t s);

// Attention experts (attention.cu: the attention core; gemm_tc_fwd.cu /
// gemm_tc_bwd.cu: the projections and their gradients).  Head dimension 64.
bool attn_core_supported(int C, int head_dim);
int launch_attn_core_fwd(int G, int C, int H, const int32_t *load, const __nv_bfloat16 *qkv,
                         __nv_bfloat16 *o, float *lse, cudaStream_t s);
int launch_attn_core_bwd(int G, int C, int H, const int32_t *load, const __nv_bfloat16 *qkv,
                         const __nv_bfloat16 *o, const float *lse, const __nv_bfloat16 *dout, float *dsum,
                         __nv_bfloat16 *dqkv, cudaStream_t s);
int launch_attn_expert_fwd(const Dims &p, int H, const __nv_bfloat16 *xe, const __nv_bfloat16 *wqkv,
                           const __nv_bfloat16 *wo, const int32_t *load, __nv_bfloat16 *qkv,
                           __nv_bfloat16 *o, float *lse, __nv_bfloat16 *ye, cudaStream_t s);
size_t attn_bwd_workspace(const Dims &p, int H);
int launch_attn_expert_bwd(const Dims &p, int H, const __nv_bfloat16 *xe, const __nv_bfloat16 *qkv,
                           const __nv_bfloat16 *o, const float *lse, const __nv_bfloat16 *wqkv,
                           const __nv_bfloat16 *wo, const __nv_bfloat16 *dye, const int32_t *load,
                           __nv_bfloat16 *dxe, __nv_bfloat16 *dwqkv, __nv_bfloat16 *dwo, void *workspace,
                           cudaStream_t s);

// ---------------------------------------------------------------------------
// Device helpers.

// Raises `kern`'s dynamic shared-memory limit on the current device to at
// least `bytes`, never lowering it, so that concurrent host threads launching
// it with different sizes all stay within the limit.  `limit` caches the value
// set per device (up to 64 devices).
inline int raise_smem_limit(const void *kern, std::atomic<int> (&limit)[64], int bytes) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return VMOE_ERR_CUDA;
    if (limit[dev].load(std::memory_order_acquire) >= bytes) return VMOE_OK;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    if (limit[dev].load(std::memory_order_relaxed) >= bytes) return VMOE_OK;
    if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) != cudaSuccess)
        return VMOE_ERR_CUDA;
    limit[dev].store(bytes, std::memory_order_release);
    return VMOE_OK;
}

// Programmatic dependent launch (see launch_kernel); both are no-ops in a
// kernel launched without the attribute.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_launch_dependents() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// 8 bf16 <-> 8 floats through one 16-byte vector.
__device__ __forceinline__ void bf16x8_to_f32(const uint4 &v, float *out) {
    const __nv_bfloat162 *h = reinterpret_cast<const __nv_bfloat162 *>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        float2 f = __bfloat1622float2(h[i]);
        out[2 * i] = f.x;
        out[2 * i + 1] = f.y;
    }
}

__device__ __forceinline__ uint4 f32_to_bf16x8(const float *in) {
    uint4 v;
    __nv_bfloat162 *h = reinterpret_cast<__nv_bfloat162 *>(&v);
#pragma unroll
    for (int i = 0; i < 4; ++i) h[i] = __floats2bfloat162_rn(in[2 * i], in[2 * i + 1]);
    return v;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
    __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&h);
}

// Warp-level bf16 tensor-core product D += A B, m16n8k16, fp32 accumulate.
__device__ __forceinline__ void mma_bf16_16816(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                               uint32_t a3, uint32_t b0, uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
        "{%8, %9}, {%0, %1, %2, %3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// An fp32 value as three bf16 parts, w ~= hi + mid + lo to about 24 significant
// bits: each product of a bf16 value with a part is exact in fp32.
__device__ __forceinline__ void split3(float w, __nv_bfloat16 &hi, __nv_bfloat16 &mid,
                                       __nv_bfloat16 &lo) {
    hi = __float2bfloat16_rn(w);
    float r = w - __bfloat162float(hi);
    mid = __float2bfloat16_rn(r);
    lo = __float2bfloat16_rn(r - __bfloat162float(mid));
}

__device__ __forceinline__ uint32_t pack2(__nv_bfloat16 lo_k, __nv_bfloat16 hi_k) {
    return (uint32_t)__bfloat16_as_ushort(lo_k) | ((uint32_t)__bfloat16_as_ushort(hi_k) << 16);
}

// GELU and its derivative: exact erf form by default, tanh form with
// VMOE_GELU_TANH.  Both call CUDA's erff / expf / tanhf.
__device__ __forceinline__ float gelu_f(float h, bool tanh_form) {
    if (tanh_form) {
        const float c = 0.7978845608028654f;  // sqrt(2/pi)
        return 0.5f * h * (1.0f + tanhf(c * (h + 0.044715f * h * h * h)));
    }
    return 0.5f * h * (1.0f + erff(h * 0.7071067811865476f));
}

__device__ __forceinline__ float gelu_deriv_f(float h, bool tanh_form) {
    if (tanh_form) {
        const float c = 0.7978845608028654f;
        float th = tanhf(c * (h + 0.044715f * h * h * h));
        return 0.5f * (1.0f + th) +
               0.5f * h * (1.0f - th * th) * c * (1.0f + 3.0f * 0.044715f * h * h);
    }
    const float inv_sqrt_2pi = 0.3989422804014327f;
    return 0.5f * (1.0f + erff(h * 0.7071067811865476f)) + h * inv_sqrt_2pi * expf(-0.5f * h * h);
}

// Fast exact-form GELU for the bf16 epilogues.  erf(x), x >= 0, by the Hastings
// rational approximation (Abramowitz & Stegun, Handbook of Mathematical
// Functions, formula 7.1.26): erf(x) = 1 - t (a1 + t (a2 + t (a3 + t (a4 + t a5))))
// exp(-x^2), t = 1 / (1 + p x), with |error| <= 1.5e-7 -- far below the bf16
// rounding of the stored outputs.  With x = |h| / sqrt 2 the factor exp(-x^2) =
// exp(-h^2 / 2) is also the one in the normal density, so GELU' costs one
// exponential, one reciprocal and a five-term polynomial.
struct PhiParts {
    float Phi;  // standard normal CDF at h
    float E;    // exp(-h^2 / 2)
};
__device__ __forceinline__ PhiParts phi_parts(float h) {
    const float p = 0.3275911f, a1 = 0.254829592f, a2 = -0.284496736f, a3 = 1.421413741f,
                a4 = -1.453152027f, a5 = 1.061405429f;
    const float x = fabsf(h) * 0.7071067811865476f;
    const float t = __fdividef(1.0f, fmaf(p, x, 1.0f));
    const float poly = t * fmaf(t, fmaf(t, fmaf(t, fmaf(t, a5, a4), a3), a2), a1);
    const float E = __expf(-0.5f * h * h);
    const float tail = 0.5f * poly * E;  // = P(Z > |h|)
    PhiParts r;
    r.Phi = h >= 0.0f ? 1.0f - tail : tail;
    r.E = E;
    return r;
}
__device__ __forceinline__ float gelu_fast(float h, bool tanh_form) {
    if (tanh_form) return gelu_f(h, true);
    return h * phi_parts(h).Phi;
}
__device__ __forceinline__ float gelu_deriv_fast(float h, bool tanh_form) {
    if (tanh_form) return gelu_deriv_f(h, true);
    const PhiParts r = phi_parts(h);
    return fmaf(h * 0.3989422804014327f, r.E, r.Phi);
}

}  // namespace vmoe
