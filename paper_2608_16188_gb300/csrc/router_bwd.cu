// router_bwd.cu -- the router backward: the gradient of <dY, y> through the
// gates with the routing (chosen experts, slots) held fixed, which completes
// the adaptation gradient of the gating network (Section 3.1: the visual
// module, router included, is what gets adapted).
//
//   dgate_j  = <dY[t,n], Ye[t, e_j, s_j]>  for a kept choice, 0 if dropped
//   dlogit   = softmax backward over the k selected logits (renormalised gates)
//              or over all E logits (VMOE_NO_RENORM)
//   dW_r[t]  = x[t]^T dlogit[t],  dbias[t] = sum_n dlogit[t,n]
//   dX[t,n] += W_r[t] dlogit[t,n]
//
// Kernel 1 (router_grad): one warp per token, 16-byte vectors along d, a fixed
// butterfly reduction per dot product.  Kernels 2 and 3 (router_dw, router_dx):
// 64 x 64 output tiles, 4 x 4 fp32 accumulators per thread, the reduction
// dimension staged through shared memory in a fixed order.  No atomics.
#include <math.h>

#include "common.cuh"

namespace vmoe {
namespace {

constexpr int RB_THREADS = 256;
constexpr int RB_WARPS = RB_THREADS / 32;

template <typename T>
__device__ __forceinline__ void load8(const T *p, float *o);
template <>
__device__ __forceinline__ void load8<__nv_bfloat16>(const __nv_bfloat16 *p, float *o) {
    bf16x8_to_f32(__ldg(reinterpret_cast<const uint4 *>(p)), o);
}
template <>
__device__ __forceinline__ void load8<float>(const float *p, float *o) {
    const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
    const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
    o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
    o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
}

template <typename T>
__device__ __forceinline__ float to_f(T v);
template <>
__device__ __forceinline__ float to_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ float to_f<__nv_bfloat16>(__nv_bfloat16 v) { return __bfloat162float(v); }

template <typename T>
__device__ __forceinline__ T from_f(float v);
template <>
__device__ __forceinline__ float from_f<float>(float v) { return v; }
template <>
__device__ __forceinline__ __nv_bfloat16 from_f<__nv_bfloat16>(float v) { return __float2bfloat16_rn(v); }

template <typename T>
__global__ void __launch_bounds__(RB_THREADS)
router_grad_kernel(Dims p, const T *__restrict__ dy, const T *__restrict__ ye,
                   const float *__restrict__ logits, const int32_t *__restrict__ idx,
                   const float *__restrict__ gate, const int32_t *__restrict__ slot,
                   float *__restrict__ dgate, float *__restrict__ dlogits) {
    const long long tn = (long long)blockIdx.x * RB_WARPS + (threadIdx.x >> 5);
    if (tn >= (long long)p.T * p.N) return;
    const int lane = threadIdx.x & 31;
    const int t = (int)(tn / p.N);
    const int k = p.k, E = p.E, d = p.d;
    const T *dyr = dy + tn * d;
    float dg[8], gt[8];
    int ei[8];
    float s = 0.0f;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        dg[j] = 0.0f;
        gt[j] = 0.0f;
        ei[j] = -1;
        if (j >= k) continue;
        const long long a = tn * k + j;
        ei[j] = idx[a];
        gt[j] = gate[a];
        const int sl = slot[a];
        if (sl >= 0) {
            const T *row = ye + (((long long)t * E + ei[j]) * p.C + sl) * d;
            float acc = 0.0f;
            for (int v = lane * 8; v < d; v += 256) {
                float fa[8], fb[8];
                load8<T>(dyr + v, fa);
                load8<T>(row + v, fb);
#pragma unroll
                for (int q = 0; q < 8; ++q) acc = fmaf(fa[q], fb[q], acc);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            dg[j] = acc;
        }
        s = fmaf(gt[j], dg[j], s);
    }
    if (lane == 0)
#pragma unroll
        for (int j = 0; j < 8; ++j)
            if (j < k) dgate[tn * k + j] = dg[j];
    float *dl = dlogits + tn * E;
    if (!(p.flags & VMOE_NO_RENORM)) {
        for (int e = lane; e < E; e += 32) {
            float v = 0.0f;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (ei[j] == e) v = gt[j] * (dg[j] - s);
            dl[e] = v;
        }
    } else {
        const float *l = logits + tn * E;
        float mx = -INFINITY;
        for (int e = lane; e < E; e += 32) mx = fmaxf(mx, l[e]);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        float sum = 0.0f;
        for (int e = lane; e < E; e += 32) sum += expf(l[e] - mx);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        for (int e = lane; e < E; e += 32) {
            float g = 0.0f;
#pragma unroll
            for (int j = 0; j < 8; ++j)
                if (ei[j] == e) g = dg[j];
            dl[e] = expf(l[e] - mx) / sum * (g - s);
        }
    }
}

constexpr int RT = 64;   // output tile edge
constexpr int RKC = 32;  // reduction chunk

// dW_r[t][i][e] = sum_n x[t,n,i] dl[t,n,e]; dbias[t][e] = sum_n dl[t,n,e].
template <typename T>
__global__ void __launch_bounds__(RB_THREADS)
router_dw_kernel(Dims p, const T *__restrict__ x, const float *__restrict__ dl,
                 float *__restrict__ dw, float *__restrict__ dbias) {
    __shared__ __align__(16) float xs[RKC][RT];
    __shared__ __align__(16) float ds[RKC][RT];
    const int t = blockIdx.z, i0 = blockIdx.x * RT, e0 = blockIdx.y * RT;
    const int tid = threadIdx.x, ti = tid / 16, tj = tid % 16;
    const int d = p.d, E = p.E, N = p.N;
    const T *xt = x + (long long)t * N * d;
    const float *dlt = dl + (long long)t * N * E;
    float acc[4][4] = {};
    float bacc = 0.0f;
    const bool do_bias = dbias != nullptr && blockIdx.x == 0 && tid < RT && e0 + tid < E;
    for (int n0 = 0; n0 < N; n0 += RKC) {
        for (int i = tid; i < RKC * RT; i += RB_THREADS) {
            const int r = i / RT, c = i % RT;
            const int n = n0 + r;
            xs[r][c] = (n < N && i0 + c < d) ? to_f(xt[(long long)n * d + i0 + c]) : 0.0f;
            ds[r][c] = (n < N && e0 + c < E) ? dlt[(long long)n * E + e0 + c] : 0.0f;
        }
        __syncthreads();
        // two-level sum (per chunk, then across chunks): the rounding error grows
        // with sqrt(RKC) + sqrt(N / RKC) instead of sqrt(N)
        float cacc[4][4] = {};
#pragma unroll 4
        for (int r = 0; r < RKC; ++r) {
            float av[4], bv[4];
#pragma unroll
            for (int a = 0; a < 4; ++a) av[a] = xs[r][ti * 4 + a];
#pragma unroll
            for (int b = 0; b < 4; ++b) bv[b] = ds[r][tj * 4 + b];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) cacc[a][b] = fmaf(av[a], bv[b], cacc[a][b]);
        }
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) acc[a][b] += cacc[a][b];
        if (do_bias) {
            float cb = 0.0f;
            for (int r = 0; r < RKC; ++r) cb += ds[r][tid];
            bacc += cb;
        }
        __syncthreads();
    }
    float *dwt = dw + (long long)t * d * E;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int i = i0 + ti * 4 + a;
        if (i >= d) continue;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int e = e0 + tj * 4 + b;
            if (e < E) dwt[(long long)i * E + e] = acc[a][b];
        }
    }
    if (do_bias) dbias[(long long)t * E + e0 + tid] = bacc;
}

// dx[t,n,i] += sum_e dl[t,n,e] W_r[t][i][e], summed in fp32 and rounded once.
template <typename T>
__global__ void __launch_bounds__(RB_THREADS)
router_dx_kernel(Dims p, const float *__restrict__ dl, const float *__restrict__ wr,
                 T *__restrict__ dx) {
    // [e][token] and [e][i], padded so the transposing stores fall in distinct banks
    __shared__ float ls[RKC][RT + 1];
    __shared__ float ws[RKC][RT + 1];
    const int t = blockIdx.z, n0 = blockIdx.x * RT, i0 = blockIdx.y * RT;
    const int tid = threadIdx.x, tn_ = tid / 16, ti = tid % 16;
    const int d = p.d, E = p.E, N = p.N;
    const float *dlt = dl + (long long)t * N * E;
    const float *wrt = wr + (long long)t * d * E;
    float acc[4][4] = {};
    for (int e0 = 0; e0 < E; e0 += RKC) {
        for (int i = tid; i < RKC * RT; i += RB_THREADS) {
            const int c = i / RKC, r = i % RKC;  // consecutive threads walk e (contiguous)
            const int e = e0 + r;
            ls[r][c] = (n0 + c < N && e < E) ? dlt[(long long)(n0 + c) * E + e] : 0.0f;
            ws[r][c] = (i0 + c < d && e < E) ? wrt[(long long)(i0 + c) * E + e] : 0.0f;
        }
        __syncthreads();
#pragma unroll 4
        for (int r = 0; r < RKC; ++r) {
            float av[4], bv[4];
#pragma unroll
            for (int a = 0; a < 4; ++a) av[a] = ls[r][tn_ * 4 + a];
#pragma unroll
            for (int b = 0; b < 4; ++b) bv[b] = ws[r][ti * 4 + b];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(av[a], bv[b], acc[a][b]);
        }
        __syncthreads();
    }
    T *dxt = dx + (long long)t * N * d;
#pragma unroll
    for (int a = 0; a < 4; ++a) {
        const int n = n0 + tn_ * 4 + a;
        if (n >= N) continue;
#pragma unroll
        for (int b = 0; b < 4; ++b) {
            const int i = i0 + ti * 4 + b;
            if (i < d) {
                T *o = dxt + (long long)n * d + i;
                *o = from_f<T>(to_f(*o) + acc[a][b]);
            }
        }
    }
}

template <typename T>
int run(const Dims &p, const void *x, const float *wr, const float *logits, const int32_t *idx,
        const float *gate, const int32_t *slot, const void *dy, const void *ye, float *dgate,
        float *dlogits, float *dw, float *dbias, void *dx, cudaStream_t s) {
    const long long tokens = (long long)p.T * p.N;
    trace_before(s, "router_grad");
    router_grad_kernel<T><<<(unsigned)((tokens + RB_WARPS - 1) / RB_WARPS), RB_THREADS, 0, s>>>(
        p, (const T *)dy, (const T *)ye, logits, idx, gate, slot, dgate, dlogits);
    trace_after(s);
    int st = launch_result();
    if (st != VMOE_OK) return st;
    dim3 gw((p.d + RT - 1) / RT, (p.E + RT - 1) / RT, p.T);
    trace_before(s, "router_dw");
    router_dw_kernel<T><<<gw, RB_THREADS, 0, s>>>(p, (const T *)x, dlogits, dw, dbias);
    trace_after(s);
    if ((st = launch_result()) != VMOE_OK) return st;
    if (dx == nullptr) return VMOE_OK;
    dim3 gx((p.N + RT - 1) / RT, (p.d + RT - 1) / RT, p.T);
    trace_before(s, "router_dx");
    router_dx_kernel<T><<<gx, RB_THREADS, 0, s>>>(p, dlogits, wr, (T *)dx);
    trace_after(s);
    return launch_result();
}

}  // namespace

int launch_router_bwd(const Dims &p, const void *x, const float *w_router, const float *logits,
                      const int32_t *idx, const float *gate, const int32_t *slot, const void *dy,
                      const void *ye, float *dgate, float *dlogits, float *dw_router, float *dbias,
                      void *dx, cudaStream_t s) {
    if (p.bf16)
        return run<__nv_bfloat16>(p, x, w_router, logits, idx, gate, slot, dy, ye, dgate, dlogits,
                                  dw_router, dbias, dx, s);
    return run<float>(p, x, w_router, logits, idx, gate, slot, dy, ye, dgate, dlogits, dw_router,
                      dbias, dx, s);
}

}  // namespace vmoe
