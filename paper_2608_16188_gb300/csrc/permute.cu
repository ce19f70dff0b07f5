// permute.cu -- K2 dispatch (token rows -> expert-contiguous [T,E,C,d]
// buffers) and K5 combine (expert rows -> token order, gate-weighted).
//
// Both are pure data movement with one warp per row and 16-byte vectors
// (d % 8 == 0 for bf16 and fp32 rows alike).  Dispatch is a scatter: warp w
// < T*N*k copies the kept choice w to its slot; warps past that zero the
// padding rows s >= load of every group, so every element of dst is written
// exactly once and no memset is needed.  Combine is the gather form of the
// scatter-add: a warp per token (persistent warps, the next token's routing
// prefetched) sums its kept choices in the order j = 0..k-1 in fp32 and
// writes the row once, with no atomics.
#include "common.cuh"

namespace vmoe {
namespace {

constexpr int PM_THREADS = 256;
constexpr int PM_WARPS = PM_THREADS / 32;

template <typename T>
struct Vec;
template <>
struct Vec<float> {
    static constexpr int n = 4;
    __device__ static void load(const uint4 &v, float *o) {
        o[0] = __uint_as_float(v.x);
        o[1] = __uint_as_float(v.y);
        o[2] = __uint_as_float(v.z);
        o[3] = __uint_as_float(v.w);
    }
    __device__ static uint4 store(const float *o) {
        return make_uint4(__float_as_uint(o[0]), __float_as_uint(o[1]), __float_as_uint(o[2]),
                          __float_as_uint(o[3]));
    }
};
template <>
struct Vec<__nv_bfloat16> {
    static constexpr int n = 8;
    __device__ static void load(const uint4 &v, float *o) { bf16x8_to_f32(v, o); }
    __device__ static uint4 store(const float *o) { return f32_to_bf16x8(o); }
};

template <typename T>
__global__ void __launch_bounds__(PM_THREADS)
dispatch_kernel(Dims p, const T *__restrict__ src, const float *__restrict__ weight,
                const int32_t *__restrict__ idx, const int32_t *__restrict__ slot,
                const int32_t *__restrict__ load, T *__restrict__ dst) {
    pdl_wait();
    constexpr int V = Vec<T>::n;
    const long long row = (long long)blockIdx.x * PM_WARPS + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    const int nvec = p.d / V;
    const long long n_assign = (long long)p.T * p.N * p.k;
    if (row < n_assign) {
        int s = slot[row];
        if (s < 0) return;
        long long tn = row / p.k;  // t*N + n
        int t = (int)(tn / p.N);
        int e = idx[row];
        const uint4 *in = reinterpret_cast<const uint4 *>(src + tn * p.d);
        uint4 *out = reinterpret_cast<uint4 *>(dst + (((long long)t * p.E + e) * p.C + s) * p.d);
        const float w = weight == nullptr ? 1.0f : weight[row];
        // All of a lane's loads are issued before its stores (up to UNR 16-byte
        // vectors per pass) so a warp keeps several row segments in flight.
        constexpr int UNR = 4;
        for (int v0 = lane; v0 < nvec; v0 += 32 * UNR) {
            uint4 buf[UNR];
#pragma unroll
            for (int u = 0; u < UNR; ++u) {
                int v = v0 + 32 * u;
                if (v < nvec) buf[u] = __ldg(in + v);
            }
#pragma unroll
            for (int u = 0; u < UNR; ++u) {
                int v = v0 + 32 * u;
                if (v >= nvec) continue;
                if (weight == nullptr) {
                    out[v] = buf[u];
                } else {
                    float f[V];
                    Vec<T>::load(buf[u], f);
#pragma unroll
                    for (int q = 0; q < V; ++q) f[q] *= w;
                    out[v] = Vec<T>::store(f);
                }
            }
        }
        return;
    }
    long long r = row - n_assign;  // padding candidate: (g, s)
    if (r >= (long long)p.T * p.E * p.C) return;
    long long g = r / p.C;
    int s = (int)(r - g * p.C);
    if (s < load[g]) return;
    uint4 *out = reinterpret_cast<uint4 *>(dst + r * p.d);
    for (int v = lane; v < nvec; v += 32) out[v] = make_uint4(0u, 0u, 0u, 0u);
}

// KMAX >= p.k is a compile-time bound so the gathered rows stay in registers.
// Persistent warps: warp w takes tokens w, w + W, ... (W warps in the grid)
// and fetches the next token's routing while the current token's rows load.
template <typename T, int KMAX>
__global__ void __launch_bounds__(PM_THREADS)
combine_kernel(Dims p, const T *__restrict__ src, const float *__restrict__ weight,
               const int32_t *__restrict__ idx, const int32_t *__restrict__ slot,
               T *__restrict__ dst) {
    pdl_wait();
    constexpr int V = Vec<T>::n;
    const long long TN = (long long)p.T * p.N;
    const long long nw = (long long)gridDim.x * PM_WARPS;
    long long tn = (long long)blockIdx.x * PM_WARPS + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    const int nvec = p.d / V;
    int e[KMAX], sl[KMAX];
    float wj[KMAX];
    auto routing = [&](long long tok, int (&ee)[KMAX], int (&ss)[KMAX], float (&ww)[KMAX]) {
#pragma unroll
        for (int j = 0; j < KMAX; ++j) {
            ee[j] = 0;
            ss[j] = -1;
            ww[j] = 0.0f;
            if (j < p.k && tok < TN) {
                ee[j] = __ldg(idx + tok * p.k + j);
                ss[j] = __ldg(slot + tok * p.k + j);
                ww[j] = weight ? __ldg(weight + tok * p.k + j) : 1.0f;
            }
        }
    };
    routing(tn, e, sl, wj);
    for (; tn < TN; tn += nw) {
        const int t = (int)(tn / p.N);
        const uint4 *rows[KMAX];
#pragma unroll
        for (int j = 0; j < KMAX; ++j)
            rows[j] = sl[j] >= 0 ? reinterpret_cast<const uint4 *>(
                                       src + (((long long)t * p.E + e[j]) * p.C + sl[j]) * p.d)
                                 : nullptr;
        uint4 *out = reinterpret_cast<uint4 *>(dst + tn * p.d);
        int e2[KMAX], s2[KMAX];
        float w2[KMAX];
        bool next_loaded = false;
        // Up to UNR vectors per lane per pass, all k source rows loaded before the
        // sums, so each warp has k * UNR 16-byte loads in flight.
        constexpr int UNR = 3;
        for (int v0 = lane; v0 < nvec; v0 += 32 * UNR) {
            uint4 buf[KMAX][UNR];
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                if (rows[j] == nullptr) continue;
#pragma unroll
                for (int u = 0; u < UNR; ++u) {
                    int v = v0 + 32 * u;
                    if (v < nvec) buf[j][u] = __ldg(rows[j] + v);
                }
            }
            if (!next_loaded) {  // the next token's routing, behind this token's rows
                routing(tn + nw, e2, s2, w2);
                next_loaded = true;
            }
#pragma unroll
            for (int u = 0; u < UNR; ++u) {
                int v = v0 + 32 * u;
                if (v >= nvec) continue;
                float acc[V];
#pragma unroll
                for (int q = 0; q < V; ++q) acc[q] = 0.0f;
#pragma unroll
                for (int j = 0; j < KMAX; ++j) {  // fixed order j = 0..k-1
                    if (rows[j] == nullptr) continue;
                    float f[V];
                    Vec<T>::load(buf[j][u], f);
#pragma unroll
                    for (int q = 0; q < V; ++q) acc[q] = fmaf(wj[j], f[q], acc[q]);
                }
                out[v] = Vec<T>::store(acc);
            }
        }
        if (!next_loaded) routing(tn + nw, e2, s2, w2);
#pragma unroll
        for (int j = 0; j < KMAX; ++j) {
            e[j] = e2[j];
            sl[j] = s2[j];
            wj[j] = w2[j];
        }
    }
}

}  // namespace

int launch_dispatch(const Dims &p, const void *src, const float *weight, const int32_t *idx,
                    const int32_t *slot, const int32_t *load, void *dst, cudaStream_t s) {
    long long rows = (long long)p.T * p.N * p.k + (long long)p.T * p.E * p.C;
    long long blocks = (rows + PM_WARPS - 1) / PM_WARPS;
    if (blocks > 0x7fffffffLL) return VMOE_ERR_UNSUPPORTED;
    int st;
    trace_before(s, "dispatch");
    if (p.bf16)
        st = launch_kernel(dispatch_kernel<__nv_bfloat16>, dim3((unsigned)blocks), dim3(PM_THREADS), 0, s,
            p, (const __nv_bfloat16 *)src, weight, idx, slot, load, (__nv_bfloat16 *)dst);
    else
        st = launch_kernel(dispatch_kernel<float>, dim3((unsigned)blocks), dim3(PM_THREADS), 0, s,
            p, (const float *)src, weight, idx, slot, load, (float *)dst);
    trace_after(s);
    return st;
}

// Persistent grid: at most as many CTAs as fit on the GPU at once.
template <typename T, int KMAX>
static unsigned combine_grid(long long blocks) {
    static std::atomic<int> per_sm[64];  // per device; the same value from every thread
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return (unsigned)blocks;
    if (per_sm[dev].load(std::memory_order_relaxed) < 1) {
        int v = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, combine_kernel<T, KMAX>, PM_THREADS, 0) !=
                cudaSuccess || v < 1)
            v = 1;
        per_sm[dev] = v;
    }
    const long long cap = (long long)per_sm[dev] * num_sms();
    return (unsigned)(blocks < cap ? blocks : cap);
}

template <typename T>
static int combine_as(const Dims &p, const void *src, const float *weight, const int32_t *idx,
                      const int32_t *slot, void *dst, long long blocks, cudaStream_t s) {
    const T *in = (const T *)src;
    T *out = (T *)dst;
    if (p.k == 1)
        return launch_kernel(combine_kernel<T, 1>, dim3(combine_grid<T, 1>(blocks)), dim3(PM_THREADS), 0, s,
                             p, in, weight, idx, slot, out);
    else if (p.k == 2)
        return launch_kernel(combine_kernel<T, 2>, dim3(combine_grid<T, 2>(blocks)), dim3(PM_THREADS), 0, s,
                             p, in, weight, idx, slot, out);
    else if (p.k <= 4)
        return launch_kernel(combine_kernel<T, 4>, dim3(combine_grid<T, 4>(blocks)), dim3(PM_THREADS), 0, s,
                             p, in, weight, idx, slot, out);
    else
        return launch_kernel(combine_kernel<T, 8>, dim3(combine_grid<T, 8>(blocks)), dim3(PM_THREADS), 0, s,
                             p, in, weight, idx, slot, out);
}

int launch_combine(const Dims &p, const void *src, const float *weight, const int32_t *idx,
                   const int32_t *slot, void *dst, cudaStream_t s) {
    long long rows = (long long)p.T * p.N;
    long long blocks = (rows + PM_WARPS - 1) / PM_WARPS;
    trace_before(s, "combine");
    const int st = p.bf16 ? combine_as<__nv_bfloat16>(p, src, weight, idx, slot, dst, blocks, s)
                          : combine_as<float>(p, src, weight, idx, slot, dst, blocks, s);
    trace_after(s);
    return st;
}

}  // namespace vmoe
