// route.cu -- K1: router GEMV + softmax + top-k gating, then the per-task
// capacity scan (Section 2.1 routing, Challenge #1 capacity limits,
// Section 3.3.1 sequential assignment).
//
// Kernel 1 (route_topk), bf16 tokens: route_mma_kernel below (or, with
// VMOE_ROUTE_TC=1, route_tc_kernel in route_tc.cu on tcgen05) -- the router
// product on the tensor cores (mma.sync) with the fp32 weights split into
// three bf16 parts.  fp32 tokens or given logits: one CTA per (task, tile of
// TOK tokens) on the CUDA cores.  The logits
// tile [TOK x E] = x_tile [TOK x d] * W_r[t] [d x E] is accumulated in fp32
// registers (4 tokens x 4 experts per thread, d swept in chunks of 32 staged
// in shared memory, one FMA chain per output in increasing i), then written to
// shared memory and to `logits`.  One thread per token then takes the max,
// the softmax denominator and the k largest logits (ties to the lower expert
// index).
//
// Kernel 2 (capacity_scan): one CTA per task.  The choice-major assignment
// sequence p = j*N + n is cut into one contiguous chunk per warp; each warp
// ranks its chunk 32 assignments at a time with __match_any_sync, keeping
// per-warp expert counters in shared memory; a per-expert exclusive scan over
// the warps then gives the global rank, which becomes the slot (or -1 once it
// reaches C).  No atomics, so the result is deterministic.
#include <math.h>

#include "common.cuh"
#include "topk.cuh"

namespace vmoe {
namespace {

constexpr int RT_THREADS = 256;
constexpr int RT_KC = 32;  // d-chunk staged per iteration

// Softmax + top-k of `ntok` logit rows held in shared memory (row pitch ldl,
// odd, so the per-thread rows hit distinct banks), one thread per row.
__device__ __forceinline__ void topk_rows(const Dims &p, const float *lg, int ldl, int ntok, int t,
                                          int n0, int32_t *__restrict__ out_idx,
                                          float *__restrict__ out_gate, int nthreads) {
    for (int r = threadIdx.x; r < ntok; r += nthreads)
        topk_row(p, lg + r * ldl, (long long)t * p.N + n0 + r, out_idx, out_gate);
}

// SIMT router for fp32 tokens (or given logits): ECH experts per pass, TOK
// tokens per CTA, TOK * ECH = 16 * RT_THREADS.
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

    topk_rows(p, lg, E + 1, ntok, t, n0, out_idx, out_gate, RT_THREADS);
}

// Tensor-core router for bf16 tokens.  x is exactly representable in bf16, so
// x * W_r is formed as x * W_hi + x * W_mid + x * W_lo with the fp32 router
// weights split into three bf16 parts (W_hi = bf16(W), W_mid = bf16(W - W_hi),
// W_lo = bf16(W - W_hi - W_mid), together about 24 significant bits): every
// partial product is exact in fp32 and the mma.sync m16n8k16 instructions
// accumulate in fp32, so the logits keep fp32 accuracy at a small fraction of
// the CUDA-core instruction count.  One CTA = 4 warps x 16 tokens of one task;
// d is swept in chunks of RM_KC staged in shared memory.  The weight split is
// done while staging, two values per conversion, into [part][expert][k]
// tiles, so that one ldmatrix.x4 gives the B fragments of two 8-expert blocks
// (and one gives a warp's A fragment).
constexpr int RM_TOK = 64;
constexpr int RM_THREADS = 128;
#ifndef VMOE_ROUTE_KC
#define VMOE_ROUTE_KC 128
#endif
constexpr int RM_KC = VMOE_ROUTE_KC;  // d per staged chunk: 128 halves the chunk chain of 64
constexpr int RM_XP = RM_KC + 8;  // row pitch (bf16) of the x and weight tiles: conflict-free ldmatrix

__device__ __forceinline__ void rm_ldsm_x4(uint32_t (&r)[4], const void *smem) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(a));
}

// NB blocks of 8 experts per pass (NB even).
template <int NB>
__global__ void __launch_bounds__(RM_THREADS, 3)
route_mma_kernel(Dims p, const __nv_bfloat16 *__restrict__ x, const float *__restrict__ wr,
                 const float *__restrict__ bias, float *__restrict__ logits,
                 int32_t *__restrict__ out_idx, float *__restrict__ out_gate) {
    static_assert(NB % 2 == 0, "B fragments are loaded two expert blocks at a time");
    pdl_wait();
    constexpr int NP = NB * 8;
    extern __shared__ __align__(16) uint8_t rm_smem[];
    __nv_bfloat16 *xs = reinterpret_cast<__nv_bfloat16 *>(rm_smem);  // [64][RM_XP]
    __nv_bfloat16 *ws = xs + RM_TOK * RM_XP;                         // [3][NP][RM_XP]
    float *lg = reinterpret_cast<float *>(ws + 3 * NP * RM_XP);      // [64][E+1]
    const int t = blockIdx.y, n0 = blockIdx.x * RM_TOK;
    const int E = p.E, d = p.d, N = p.N;
    const int ldl = E + 1;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int g = lane >> 2, tq = lane & 3;
    const int ntok = min(RM_TOK, N - n0);
    const __nv_bfloat16 *xt = x + ((long long)t * N + n0) * d;
    const float *wt = wr + (long long)t * d * E;
    // Per thread and chunk: XV x vectors (16 B each) and WI weight items, an
    // item being 8 consecutive k of one expert.  The next chunk's values are
    // loaded into registers before the current chunk's MMAs run, so global
    // latency overlaps the tensor-core work.
    constexpr int XV = RM_TOK * (RM_KC / 8) / RM_THREADS;
    constexpr int WI = (RM_KC / 8) * NP / RM_THREADS;
    uint4 xv[XV];
    float wv[WI][8];
    auto load_chunk = [&](int e0, int k0) {
#pragma unroll
        for (int q = 0; q < XV; ++q) {
            const int i = tid + q * RM_THREADS;
            const int r = i / (RM_KC / 8), c = (i % (RM_KC / 8)) * 8;
            xv[q] = make_uint4(0, 0, 0, 0);
            if (r < ntok && k0 + c < d)
                xv[q] = __ldg(reinterpret_cast<const uint4 *>(xt + (long long)r * d + k0 + c));
        }
#pragma unroll
        for (int q = 0; q < WI; ++q) {  // consecutive threads: consecutive experts (coalesced)
            const int i = tid + q * RM_THREADS;
            const int n = i % NP, e = e0 + n, kk = k0 + (i / NP) * 8;
#pragma unroll
            for (int r = 0; r < 8; ++r)
                wv[q][r] = (e < E && kk + r < d) ? __ldg(wt + (long long)(kk + r) * E + e) : 0.0f;
        }
    };
    auto stage_chunk = [&]() {
#pragma unroll
        for (int q = 0; q < XV; ++q) {
            const int i = tid + q * RM_THREADS;
            const int r = i / (RM_KC / 8), c = (i % (RM_KC / 8)) * 8;
            *reinterpret_cast<uint4 *>(xs + r * RM_XP + c) = xv[q];
        }
#pragma unroll
        for (int q = 0; q < WI; ++q) {
            const int i = tid + q * RM_THREADS;
            const int n = i % NP, c = (i / NP) * 8;
            uint32_t hi[4], mid[4], lo[4];
#pragma unroll
            for (int j = 0; j < 4; ++j) {  // split3 of a k pair, both values per conversion
                const __nv_bfloat162 h = __floats2bfloat162_rn(wv[q][2 * j], wv[q][2 * j + 1]);
                const float2 hf = __bfloat1622float2(h);
                const float r0 = wv[q][2 * j] - hf.x, r1 = wv[q][2 * j + 1] - hf.y;
                const __nv_bfloat162 m = __floats2bfloat162_rn(r0, r1);
                const float2 mf = __bfloat1622float2(m);
                const __nv_bfloat162 l = __floats2bfloat162_rn(r0 - mf.x, r1 - mf.y);
                hi[j] = *reinterpret_cast<const uint32_t *>(&h);
                mid[j] = *reinterpret_cast<const uint32_t *>(&m);
                lo[j] = *reinterpret_cast<const uint32_t *>(&l);
            }
            *reinterpret_cast<uint4 *>(ws + (0 * NP + n) * RM_XP + c) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
            *reinterpret_cast<uint4 *>(ws + (1 * NP + n) * RM_XP + c) = make_uint4(mid[0], mid[1], mid[2], mid[3]);
            *reinterpret_cast<uint4 *>(ws + (2 * NP + n) * RM_XP + c) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
    };
    // ldmatrix row addresses: A, rows warp*16 + (lane & 15), k offset 8 (lane >> 4);
    // B, expert (lane & 7) + 8 (lane >> 4) of a block pair, k offset 8 ((lane >> 3) & 1)
    const __nv_bfloat16 *xa = xs + (warp * 16 + (lane & 15)) * RM_XP + (lane >> 4) * 8;
    const __nv_bfloat16 *wb = ws + ((lane & 7) + (lane >> 4) * 8) * RM_XP + ((lane >> 3) & 1) * 8;
    for (int e0 = 0; e0 < E; e0 += NP) {
        float acc[NB][4];
#pragma unroll
        for (int nb = 0; nb < NB; ++nb)
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[nb][i] = 0.0f;
        load_chunk(e0, 0);
        for (int k0 = 0; k0 < d; k0 += RM_KC) {
            __syncthreads();  // the previous chunk's fragments have been read
            stage_chunk();
            __syncthreads();
            if (k0 + RM_KC < d) load_chunk(e0, k0 + RM_KC);
#pragma unroll
            for (int ks = 0; ks < RM_KC; ks += 16) {
                uint32_t a[4];
                rm_ldsm_x4(a, xa + ks);
#pragma unroll
                for (int np = 0; np < NB / 2; ++np) {
                    uint32_t b[3][4];  // [part][b0, b1 of block 2np; b0, b1 of block 2np+1]
#pragma unroll
                    for (int sp = 0; sp < 3; ++sp) rm_ldsm_x4(b[sp], wb + (sp * NP + np * 16) * RM_XP + ks);
#pragma unroll
                    for (int h = 0; h < 2; ++h)
#pragma unroll
                        for (int sp = 2; sp >= 0; --sp)  // smallest part first
                            mma_bf16_16816(acc[2 * np + h], a[0], a[1], a[2], a[3], b[sp][2 * h], b[sp][2 * h + 1]);
                }
            }
        }
#pragma unroll
        for (int nb = 0; nb < NB; ++nb)
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = warp * 16 + g + (i >> 1) * 8;
                const int e = e0 + nb * 8 + 2 * tq + (i & 1);
                if (r < ntok && e < E) lg[r * ldl + e] = acc[nb][i] + (bias ? bias[(long long)t * E + e] : 0.0f);
            }
    }
    __syncthreads();
    for (int i = tid; i < ntok * E; i += RM_THREADS) {
        const int r = i / E, e = i - r * E;
        logits[((long long)t * N + n0 + r) * E + e] = lg[r * ldl + e];
    }
    topk_rows(p, lg, ldl, ntok, t, n0, out_idx, out_gate, RM_THREADS);
}

template <int NB>
int launch_mma_router(const Dims &p, const __nv_bfloat16 *x, const float *wr, const float *bias,
                      float *logits, int32_t *idx, float *gate, cudaStream_t s) {
    constexpr int NP = NB * 8;
    size_t smem = (size_t)RM_TOK * RM_XP * 2 + (size_t)3 * NP * RM_XP * 2 + (size_t)RM_TOK * (p.E + 1) * 4;
    if (smem > 227 * 1024) return VMOE_ERR_UNSUPPORTED;
    static std::atomic<int> smem_limit[64];  // the size depends on E
    if (const int st = raise_smem_limit((const void *)route_mma_kernel<NB>, smem_limit, (int)smem)) return st;
    dim3 grid((p.N + RM_TOK - 1) / RM_TOK, p.T);
    trace_before(s, "route_topk");
    const int st = launch_kernel(route_mma_kernel<NB>, grid, dim3(RM_THREADS), smem, s, p, x, wr, bias,
                                 logits, idx, gate);
    trace_after(s);
    return st;
}

// SMEM_IDX: the task's idx array and the temporary ranks live in shared memory
// (read and written with coalesced accesses); otherwise they stay in global memory.
// CS_THREADS: 1024 (32 warps, 4 rounds of 32 assignments per warp at N k = 3152)
// while the per-warp expert counters stay small (E <= 128), else 256.
template <bool SMEM_IDX, int CS_THREADS>
__global__ void __launch_bounds__(CS_THREADS)
capacity_scan_kernel(Dims p, const int32_t *__restrict__ idx, int32_t *__restrict__ slot,
                     int32_t *__restrict__ load) {
    constexpr int CS_WARPS = CS_THREADS / 32;
    pdl_wait();
    extern __shared__ int cs_smem[];
    int *cnt = cs_smem;  // [CS_WARPS][E]
    const int t = blockIdx.x;
    const int E = p.E, N = p.N, k = p.k, C = p.C;
    const int total = k * N;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long tb = (long long)t * N * k;
    int *sidx = cs_smem + CS_WARPS * E;  // [N*k] in token-major (memory) order
    int *srank = sidx + total;           // [N*k]
    for (int i = threadIdx.x; i < CS_WARPS * E; i += CS_THREADS) cnt[i] = 0;
    if (SMEM_IDX)
        for (int i = threadIdx.x; i < total; i += CS_THREADS) sidx[i] = idx[tb + i];
    __syncthreads();
    const int32_t *src = SMEM_IDX ? sidx : idx + tb;
    int32_t *rank = SMEM_IDX ? srank : slot + tb;

    const int per = ((total + CS_WARPS - 1) / CS_WARPS + 31) & ~31;
    const int beg = min(total, warp * per), end = min(total, beg + per);
    int *my = cnt + warp * E;
    const unsigned lt = (1u << lane) - 1u;
    // Pass 1: rank within the warp's chunk of the choice-major sequence p = j*N + n.
    for (int p0 = beg; p0 < end; p0 += 32) {
        int pos = p0 + lane;
        bool valid = pos < end;
        int n = valid ? pos % N : 0, j = valid ? pos / N : 0;
        int e = valid ? src[n * k + j] : -1;
        unsigned peers = __match_any_sync(0xffffffffu, e);
        int before = __popc(peers & lt);
        if (valid) rank[n * k + j] = my[e] + before;
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
    if (SMEM_IDX) {
        // each memory position i = n*k + j belongs to the warp whose chunk holds p = j*N + n
        for (int i = threadIdx.x; i < total; i += CS_THREADS) {
            const int n = i / k, j = i - n * k;
            const int pos = j * N + n;
            const int w = pos / per;
            const int r = srank[i] + cnt[w * E + sidx[i]];
            slot[tb + i] = r < C ? r : -1;
        }
    } else {
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
}

template <typename TX, int ECH>
int launch_topk(const Dims &p, const TX *x, const float *wr, const float *bias, float *logits,
                int32_t *idx, float *gate, cudaStream_t s) {
    constexpr int TOK = 16 * RT_THREADS / ECH;
    size_t smem = sizeof(float) * ((size_t)RT_KC * TOK + (size_t)RT_KC * ECH + (size_t)TOK * (p.E + 1));
    static std::atomic<int> smem_limit[64];
    if (const int st = raise_smem_limit((const void *)route_topk_kernel<TX, ECH>, smem_limit, (int)smem))
        return st;
    dim3 grid((p.N + TOK - 1) / TOK, p.T);
    trace_before(s, "route_topk");
    route_topk_kernel<TX, ECH><<<grid, RT_THREADS, smem, s>>>(p, x, wr, bias, logits, idx, gate,
                                                              x == nullptr);
    trace_after(s);
    return launch_result();
}

template <int CS_THREADS>
int launch_scan(const Dims &p, const int32_t *idx, int32_t *slot, int32_t *load, cudaStream_t s) {
    const size_t total = (size_t)p.N * p.k;
    const size_t smem_small = sizeof(int) * (size_t)(CS_THREADS / 32) * p.E;
    const size_t smem_big = smem_small + sizeof(int) * 2 * total;
    if (smem_big <= 96 * 1024) {
        static std::atomic<int> smem_limit[64];
        if (const int st = raise_smem_limit((const void *)capacity_scan_kernel<true, CS_THREADS>, smem_limit,
                                            (int)smem_big))
            return st;
        return launch_kernel(capacity_scan_kernel<true, CS_THREADS>, dim3(p.T), dim3(CS_THREADS), smem_big,
                             s, p, idx, slot, load);
    }
    return launch_kernel(capacity_scan_kernel<false, CS_THREADS>, dim3(p.T), dim3(CS_THREADS), smem_small,
                         s, p, idx, slot, load);
}

}  // namespace

int launch_route(const Dims &p, const void *x, const float *w_router, const float *bias,
                 float *logits, int32_t *idx, float *gate, int32_t *slot, int32_t *load,
                 cudaStream_t s) {
    int st;
    if (p.bf16 && x != nullptr) {
        const __nv_bfloat16 *xb = (const __nv_bfloat16 *)x;
        if (route_tc_enabled() && route_tc_width(p) > 0)
            st = launch_route_tc(p, xb, w_router, bias, logits, idx, gate, s);
        else
            st = p.E <= 32 ? launch_mma_router<4>(p, xb, w_router, bias, logits, idx, gate, s)
                           : launch_mma_router<8>(p, xb, w_router, bias, logits, idx, gate, s);
    } else if (p.bf16) {  // given logits: no GEMV
        st = launch_topk<__nv_bfloat16, 64>(p, nullptr, w_router, bias, logits, idx, gate, s);
    } else {
        const float *xf = (const float *)x;
        st = p.E <= 32 ? launch_topk<float, 32>(p, xf, w_router, bias, logits, idx, gate, s)
                       : launch_topk<float, 64>(p, xf, w_router, bias, logits, idx, gate, s);
    }
    if (st != VMOE_OK) return st;
    trace_before(s, "capacity_scan");
    st = p.E <= 128 ? launch_scan<1024>(p, idx, slot, load, s) : launch_scan<256>(p, idx, slot, load, s);
    trace_after(s);
    return st;
}

}  // namespace vmoe
