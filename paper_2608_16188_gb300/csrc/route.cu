// route.cu -- K1: router GEMV + softmax + top-k gating, then the per-task
// capacity scan (Section 2.1 routing, Challenge #1 capacity limits,
// Section 3.3.1 sequential assignment).
//
// Kernel 1 (route_topk): one CTA per (task, tile of TOK tokens).  The logits
// tile [TOK x E] = x_tile [TOK x d] * W_r[t] [d x E] is accumulated in fp32
// registers (4 tokens x 4 experts per thread, d swept in chunks of 32 staged
// in shared memory, one FMA chain per output in increasing i), then written to
// shared memory and to `logits`.  One warp per token then takes the max, the
// softmax denominator and k rounds of a warp arg-max (larger logit wins, ties
// to the lower expert index).
//
// Kernel 2 (capacity_scan): one CTA per task.  The choice-major assignment
// sequence p = j*N + n is cut into one contiguous chunk per warp; each warp
// ranks its chunk 32 assignments at a time with __match_any_sync, keeping
// per-warp expert counters in shared memory; a per-expert exclusive scan over
// the warps then gives the global rank, which becomes the slot (or -1 once it
// reaches C).  No atomics, so the result is deterministic.
#include <math.h>

#include "common.cuh"

namespace vmoe {
namespace {

constexpr int RT_THREADS = 256;
constexpr int RT_KC = 32;  // d-chunk staged per iteration

// ECH experts per pass, TOK tokens per CTA, TOK * ECH = 16 * RT_THREADS.
template <typename TX, int ECH>
__global__ void __launch_bounds__(RT_THREADS)
route_topk_kernel(Dims p, const TX *__restrict__ x, const float *__restrict__ wr,
                  const float *__restrict__ bias, float *__restrict__ logits,
                  int32_t *__restrict__ out_idx, float *__restrict__ out_gate, int logits_in) {
    constexpr int TOK = 16 * RT_THREADS / ECH;
    constexpr int TX_THREADS = ECH / 4;  // threads along experts
    extern __shared__ __align__(16) float smem[];
    float *xs = smem;                    // [RT_KC][TOK]  (x chunk, transposed)
    float *ws = xs + RT_KC * TOK;        // [RT_KC][ECH]
    float *lg = ws + RT_KC * ECH;        // [TOK][E + 1]

    const int t = blockIdx.y;
    const int n0 = blockIdx.x * TOK;
    const int E = p.E, d = p.d, N = p.N;
    const int ldl = E + 1;
    const int tid = threadIdx.x;
    const int ntok = min(TOK, N - n0);

    if (logits_in) {
        for (int i = tid; i < ntok * E; i += RT_THREADS) {
            int r = i / E, e = i - r * E;
            lg[r * ldl + e] = logits[((long long)t * N + n0 + r) * E + e];
        }
    } else {
        const int tg = tid / TX_THREADS;  // token group: tokens 4*tg .. 4*tg+3
        const int eg = tid % TX_THREADS;  // expert group: experts 4*eg .. 4*eg+3
        const TX *xt = x + ((long long)t * N + n0) * d;
        const float *wt = wr + (long long)t * d * E;
        for (int e0 = 0; e0 < E; e0 += ECH) {
            float acc[4][4];
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[a][b] = 0.0f;
            for (int k0 = 0; k0 < d; k0 += RT_KC) {
                __syncthreads();
                // 16-byte vector loads along d (d % 8 == 0, so a vector is
                // either wholly inside the row or wholly past its end).
                constexpr int VEC = 16 / sizeof(TX);
                for (int i = tid; i < TOK * (RT_KC / VEC); i += RT_THREADS) {
                    int r = i / (RT_KC / VEC), c = (i - r * (RT_KC / VEC)) * VEC;
                    float v[VEC];
                    if (r < ntok && k0 + c < d) {
                        uint4 raw = *reinterpret_cast<const uint4 *>(xt + (long long)r * d + k0 + c);
                        if constexpr (VEC == 8) {
                            bf16x8_to_f32(raw, v);
                        } else {
                            v[0] = __uint_as_float(raw.x);
                            v[1] = __uint_as_float(raw.y);
                            v[2] = __uint_as_float(raw.z);
                            v[3] = __uint_as_float(raw.w);
                        }
                    } else {
#pragma unroll
                        for (int q = 0; q < VEC; ++q) v[q] = 0.0f;
                    }
#pragma unroll
                    for (int q = 0; q < VEC; ++q) xs[(c + q) * TOK + r] = v[q];
                }
                for (int i = tid; i < RT_KC * ECH; i += RT_THREADS) {
                    int r = i / ECH, c = i - r * ECH;
                    float v = 0.0f;
                    if (k0 + r < d && e0 + c < E) v = wt[(long long)(k0 + r) * E + e0 + c];
                    ws[r * ECH + c] = v;
                }
                __syncthreads();
#pragma unroll 8
                for (int kk = 0; kk < RT_KC; ++kk) {
                    float4 av = *reinterpret_cast<const float4 *>(&xs[kk * TOK + 4 * tg]);
                    float4 bv = *reinterpret_cast<const float4 *>(&ws[kk * ECH + 4 * eg]);
                    float a4[4] = {av.x, av.y, av.z, av.w};
                    float b4[4] = {bv.x, bv.y, bv.z, bv.w};
#pragma unroll
                    for (int a = 0; a < 4; ++a)
#pragma unroll
                        for (int b = 0; b < 4; ++b) acc[a][b] = fmaf(a4[a], b4[b], acc[a][b]);
                }
            }
#pragma unroll
            for (int a = 0; a < 4; ++a) {
                int r = 4 * tg + a;
#pragma unroll
                for (int b = 0; b < 4; ++b) {
                    int e = e0 + 4 * eg + b;
                    if (r < ntok && e < E) {
                        float v = acc[a][b];
                        if (bias) v += bias[(long long)t * E + e];
                        lg[r * ldl + e] = v;
                    }
                }
            }
        }
        __syncthreads();
        for (int i = tid; i < ntok * E; i += RT_THREADS) {
            int r = i / E, e = i - r * E;
            logits[((long long)t * N + n0 + r) * E + e] = lg[r * ldl + e];
        }
    }
    __syncthreads();

    // Softmax + top-k, one warp per token.
    const int warp = tid >> 5, lane = tid & 31;
    const bool renorm = !(p.flags & VMOE_NO_RENORM);
    for (int r = warp; r < ntok; r += RT_THREADS / 32) {
        float v[8];
        bool taken[8];
        float mx = -INFINITY;
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            int e = lane + 32 * i;
            float val = -INFINITY;
            if (e < E) {
                val = lg[r * ldl + e];
                if (isnan(val)) val = -INFINITY;  // NaN never wins a comparison
            }
            v[i] = val;
            taken[i] = false;
            mx = fmaxf(mx, val);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
        float sum = 0.0f;
#pragma unroll
        for (int i = 0; i < 8; ++i)
            if (lane + 32 * i < E) sum += expf(v[i] - mx);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);

        float ev[8];
        int ei[8];
        for (int j = 0; j < p.k; ++j) {
            float bv = -INFINITY;
            int be = 0x7fffffff;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                int e = lane + 32 * i;
                if (e < E && !taken[i] && (v[i] > bv || (v[i] == bv && e < be))) {
                    bv = v[i];
                    be = e;
                }
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) {
                float ov = __shfl_xor_sync(0xffffffffu, bv, o);
                int oe = __shfl_xor_sync(0xffffffffu, be, o);
                if (ov > bv || (ov == bv && oe < be)) {
                    bv = ov;
                    be = oe;
                }
            }
#pragma unroll
            for (int i = 0; i < 8; ++i)
                if (lane + 32 * i == be) taken[i] = true;
            ei[j] = be;
            ev[j] = expf(bv - mx);
        }
        if (lane == 0) {
            float kept = 0.0f;
            for (int j = 0; j < p.k; ++j) kept += ev[j];
            long long base = ((long long)t * N + n0 + r) * p.k;
            for (int j = 0; j < p.k; ++j) {
                out_idx[base + j] = ei[j];
                out_gate[base + j] = renorm ? ev[j] / kept : ev[j] / sum;
            }
        }
    }
}

constexpr int CS_THREADS = 256;
constexpr int CS_WARPS = CS_THREADS / 32;

__global__ void __launch_bounds__(CS_THREADS)
capacity_scan_kernel(Dims p, const int32_t *__restrict__ idx, int32_t *__restrict__ slot,
                     int32_t *__restrict__ load) {
    extern __shared__ int cnt[];  // [CS_WARPS][E]
    const int t = blockIdx.x;
    const int E = p.E, N = p.N, k = p.k, C = p.C;
    const int total = k * N;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int i = threadIdx.x; i < CS_WARPS * E; i += CS_THREADS) cnt[i] = 0;
    __syncthreads();

    const int per = ((total + CS_WARPS - 1) / CS_WARPS + 31) & ~31;
    const int beg = min(total, warp * per), end = min(total, beg + per);
    int *my = cnt + warp * E;
    const unsigned lt = (1u << lane) - 1u;
    const long long tb = (long long)t * N * k;
    // Pass 1: rank within the warp's chunk.
    for (int p0 = beg; p0 < end; p0 += 32) {
        int pos = p0 + lane;
        bool valid = pos < end;
        int n = valid ? pos % N : 0, j = valid ? pos / N : 0;
        int e = valid ? idx[tb + (long long)n * k + j] : -1;
        unsigned peers = __match_any_sync(0xffffffffu, e);
        int before = __popc(peers & lt);
        if (valid) slot[tb + (long long)n * k + j] = my[e] + before;
        __syncwarp();
        if (valid && before == 0) my[e] += __popc(peers);
        __syncwarp();
    }
    __syncthreads();
    // Exclusive scan over warps, per expert.
    for (int e = threadIdx.x; e < E; e += CS_THREADS) {
        int run = 0;
        for (int w = 0; w < CS_WARPS; ++w) {
            int c = cnt[w * E + e];
            cnt[w * E + e] = run;
            run += c;
        }
        load[(long long)t * E + e] = min(run, C);
    }
    __syncthreads();
    // Pass 2: global rank -> slot.
    for (int p0 = beg; p0 < end; p0 += 32) {
        int pos = p0 + lane;
        if (pos < end) {
            int n = pos % N, j = pos / N;
            long long a = tb + (long long)n * k + j;
            int e = idx[a];
            int r = slot[a] + my[e];
            slot[a] = r < C ? r : -1;
        }
    }
}

template <typename TX, int ECH>
int launch_topk(const Dims &p, const TX *x, const float *wr, const float *bias, float *logits,
                int32_t *idx, float *gate, cudaStream_t s) {
    constexpr int TOK = 16 * RT_THREADS / ECH;
    size_t smem = sizeof(float) * ((size_t)RT_KC * TOK + (size_t)RT_KC * ECH + (size_t)TOK * (p.E + 1));
    static bool attr_set = false;  // per instantiation; same value on every device
    if (!attr_set) {
        cudaFuncSetAttribute(route_topk_kernel<TX, ECH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             96 * 1024);
        attr_set = true;
    }
    dim3 grid((p.N + TOK - 1) / TOK, p.T);
    trace_before(s, "route_topk");
    route_topk_kernel<TX, ECH><<<grid, RT_THREADS, smem, s>>>(p, x, wr, bias, logits, idx, gate,
                                                              x == nullptr);
    trace_after(s);
    return launch_result();
}

}  // namespace

int launch_route(const Dims &p, const void *x, const float *w_router, const float *bias,
                 float *logits, int32_t *idx, float *gate, int32_t *slot, int32_t *load,
                 cudaStream_t s) {
    int st;
    if (p.bf16) {
        const __nv_bfloat16 *xb = (const __nv_bfloat16 *)x;
        st = p.E <= 32 ? launch_topk<__nv_bfloat16, 32>(p, xb, w_router, bias, logits, idx, gate, s)
                       : launch_topk<__nv_bfloat16, 64>(p, xb, w_router, bias, logits, idx, gate, s);
    } else {
        const float *xf = (const float *)x;
        st = p.E <= 32 ? launch_topk<float, 32>(p, xf, w_router, bias, logits, idx, gate, s)
                       : launch_topk<float, 64>(p, xf, w_router, bias, logits, idx, gate, s);
    }
    if (st != VMOE_OK) return st;
    size_t smem = sizeof(int) * (size_t)CS_WARPS * p.E;
    trace_before(s, "capacity_scan");
    capacity_scan_kernel<<<p.T, CS_THREADS, smem, s>>>(p, idx, slot, load);
    trace_after(s);
    return launch_result();
}

}  // namespace vmoe
