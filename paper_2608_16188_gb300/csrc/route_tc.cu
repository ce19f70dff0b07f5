// route_tc.cu -- K1 for bf16 tokens on the tcgen05 tensor cores: the router
// product x W_r[t] (Section 2.1 routing), then the softmax and the top-k.
//
// Accuracy.  The fp32 router weights are split into three bf16 parts,
// W = W_hi + W_mid + W_lo with W_hi = bf16(W), W_mid = bf16(W - W_hi),
// W_lo = bf16(W - W_hi - W_mid) (about 24 significant bits together).  A bf16
// token value times a bf16 part is exact in fp32; the three parts sit side by
// side as the 3 EP rows of one B operand, so one MMA per k-step gives the
// three partial products in fp32 TMEM columns, and the epilogue adds them,
// smallest part first: the logits keep fp32 accuracy on the bf16 tensor pipe.
//
// Work split.  Each task gets floor(SMs / T) CTAs (at least one, at most one
// per 32-token unit); CTA c of task t takes a contiguous, balanced range of
// 32-token units.  A CTA therefore splits its task's W_r only once, into
// shared memory, where it stays for all of the CTA's tokens: K-major, 128-byte
// swizzle, laid out [k-block of 64][part][expert][64 k] so that each k-block
// is one B operand of N = 3 EP rows (EP = E rounded up to 16, zero rows past
// E).  The split runs on all warps while the TMA producer has already
// filled the x ring, so its latency overlaps the first loads.
//
// Roles after the split (256 threads):
//   warp 0      TMA producer: 128-token x 64-k slots of x, one 128-row box
//               for a full tile; a range's last tile loads only the 32-row
//               boxes it needs (rows of a slot past them are stale and give
//               accumulator rows that are never read).
//   warp 1      MMA issuer: tcgen05.mma M = 128, N = 3 EP, K = 16, one per
//               k-step, accumulator double-buffered in TMEM (2 x 3 EP columns).
//   warps 4-7   epilogue: one thread per token (its TMEM lane) loads the
//               3 EP accumulator columns, adds the parts and the bias, stores
//               its logits row and
//               takes the softmax and the top-k in registers, with the same
//               operations in the same order as topk_row.
//   warps 2-3   take part in the split only.
//
// Measured on GB300 (us per launch, traced; the mma.sync router of route.cu in
// brackets): alone, 28.7 (31.2) at 17 tasks x 1576 tokens, 23.3 (27.1) at 6 x
// 3152, 14.3 (12.3) at 4 x 1576 with d = 384; inside the 17-task step, 37.6
// (31.5).  Time stamps of a CTA show its x stream at 10-16 GB/s per SM inside
// the step against 16-20 GB/s alone, while the mma.sync router keeps its
// speed, so this kernel is opt-in (VMOE_ROUTE_TC=1).
//
// Every mbarrier wait is bounded (4 s); on expiry the device status word is
// set to VMOE_ERR_DEVICE_TIMEOUT, the roles leave their loops, the producer
// lets its copies in flight land, the MMA thread waits for its MMAs, and TMEM
// is freed before the CTA returns.
#include "gemm_tc.cuh"
#include "topk.cuh"

namespace vmoe {
namespace {

using namespace tc;

constexpr int RC_THREADS = 256;
constexpr int RC_TOK = 128;                      // tokens per tile (TMEM lanes)
constexpr int RC_BOX = 32;                       // rows per x box = token unit
constexpr uint32_t RC_SLOT = RC_TOK * BK * 2;    // 16 KB: one x slot
constexpr uint32_t RC_BOX_BYTES = RC_BOX * BK * 2;
constexpr int RC_MAX_STAGES = 8;
constexpr int RC_SMEM_CAP = 232448;              // 227 KB
constexpr int RC_FIXED = 1024 + 256;             // alignment slack + barriers and words

struct RcArgs {
    int T, N, d, E, k;
    unsigned flags;
    int cpt;      // CTAs per task
    int units;    // 32-token units per task
    int stages;
    const float *wr;    // [T, d, E]
    const float *bias;  // [T, E] or null
    float *logits;      // [T, N, E]
    int32_t *idx;       // [T, N, k]
    float *gate;        // [T, N, k]
    int *status;
};

// Bytes of the resident split weights: d/64 k-blocks x 3 parts x EP rows x 128 B.
__host__ __device__ constexpr size_t rc_w_bytes(int d, int EP) { return (size_t)(d / 64) * 3 * EP * 128; }

// Softmax + top-k of one token whose E logits are in registers (EP >= E).
// The operations and their order are those of topk_row, so equal logits give
// bitwise equal indices and gates.
template <int EP>
__device__ __forceinline__ void topk_regs(const RcArgs &a, float (&w)[EP], long long tok) {
    const int E = a.E;
    const bool renorm = !(a.flags & VMOE_NO_RENORM);
    float mx = -INFINITY;
#pragma unroll
    for (int e = 0; e < EP; ++e) {
        w[e] = isnan(w[e]) ? -INFINITY : w[e];
        if (e < E) mx = fmaxf(mx, w[e]);
    }
    float sum = 0.0f;
#pragma unroll
    for (int e = 0; e < EP; ++e)
        if (e < E) sum += expf(w[e] - mx);
    float pv = INFINITY;
    int pe = -1;
    float kept = 0.0f;
    float ev[8];
    int ei[8];
#pragma unroll
    for (int j = 0; j < 8; ++j) {
        ev[j] = 0.0f;
        ei[j] = 0;
        if (j >= a.k) continue;
        float bv = -INFINITY;
        int be = -1;
#pragma unroll
        for (int e = 0; e < EP; ++e) {
            if (e >= E) continue;
            const float v = w[e];
            const bool after = v < pv || (v == pv && e > pe);
            if (after && (be < 0 || v > bv)) {
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
    const long long base = tok * a.k;
#pragma unroll
    for (int j = 0; j < 8; ++j)
        if (j < a.k) {
            a.idx[base + j] = ei[j];
            a.gate[base + j] = renorm ? ev[j] / kept : ev[j] / sum;
        }
}

template <int EP>
__global__ void __launch_bounds__(RC_THREADS, 1)
route_tc_kernel(const __grid_constant__ CUtensorMap tmX, const __grid_constant__ CUtensorMap tmX128, RcArgs a) {
    constexpr int NW = 3 * EP;  // MMA N: the three parts of EP experts
    constexpr uint32_t IDESC = idesc_bf16(RC_TOK, NW, false, false);
    constexpr uint32_t TMEM_COLS = 2 * NW <= 128 ? 128 : (2 * NW <= 256 ? 256 : 512);
    constexpr int NB16 = EP / 16;  // tcgen05.ld x16 loads per part

    extern __shared__ uint8_t rc_raw[];
    const uint32_t raw_addr = smem_u32(rc_raw);
    uint8_t *smem = rc_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
    const int d = a.d, NKB = d / BK, S = a.stages;
    uint8_t *wsm = smem;                                     // split weights
    uint8_t *xsm = smem + rc_w_bytes(d, EP);                 // x ring
    uint64_t *bars = reinterpret_cast<uint64_t *>(xsm + (size_t)S * RC_SLOT);
    int *misc = reinterpret_cast<int *>(bars + 2 * RC_MAX_STAGES + 5);  // [0] tmem base, [1] abort
    const uint32_t w_addr = smem_u32(wsm), x_addr = smem_u32(xsm);
    auto bar_full = [&](int s) { return smem_u32(bars + s); };
    auto bar_empty = [&](int s) { return smem_u32(bars + RC_MAX_STAGES + s); };
    auto bar_tfull = [&](int b) { return smem_u32(bars + 2 * RC_MAX_STAGES + b); };
    auto bar_tempty = [&](int b) { return smem_u32(bars + 2 * RC_MAX_STAGES + 2 + b); };
    const uint32_t bar_drain = smem_u32(bars + 2 * RC_MAX_STAGES + 4);
    volatile int *abort_flag = misc + 1;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int t = blockIdx.x / a.cpt, c = blockIdx.x % a.cpt;
    const int u0 = (int)((long long)c * a.units / a.cpt), u1 = (int)((long long)(c + 1) * a.units / a.cpt);
    const int n_begin = u0 * RC_BOX, n_end = min(a.N, u1 * RC_BOX);
    const int ntiles = (n_end - n_begin + RC_TOK - 1) / RC_TOK;
    const int total = ntiles * NKB;  // (tile, k-block) steps

    if (tid == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(bar_full(s), 1);
            mbar_init(bar_empty(s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(bar_tfull(b), 1);
            mbar_init(bar_tempty(b), 4);
        }
        mbar_init(bar_drain, 1);
        misc[1] = 0;
        fence_barrier_init();
        prefetch_map(&tmX);
        prefetch_map(&tmX128);
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(misc), TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = (uint32_t)misc[0];
    pdl_wait();

    // x slot loads of step i = (tile i / NKB, k-block i % NKB) into stage i % S.
    auto issue = [&](int i) {
        const int j = i / NKB, kb = i - j * NKB, s = i % S;
        const int n = n_begin + j * RC_TOK;
        const int nbox = (min(RC_TOK, n_end - n) + RC_BOX - 1) / RC_BOX;
        const uint32_t fb = bar_full(s);
        mbar_expect_tx(fb, (uint32_t)nbox * RC_BOX_BYTES);
        if (nbox * RC_BOX == RC_TOK)  // a full tile: one 128-row box
            tma_load_3d(x_addr + s * RC_SLOT, &tmX128, fb, kb * BK, n, t);
        else
            for (int b = 0; b < nbox; ++b)
                tma_load_3d(x_addr + s * RC_SLOT + b * RC_BOX_BYTES, &tmX, fb, kb * BK, n + b * RC_BOX, t);
    };
    const int prefill = min(S, total);
    int last_i[RC_MAX_STAGES];  // producer: the last step issued into each stage

    // ---- split W_r[t] into the three bf16 parts, all threads.  Item = 8
    // consecutive k of one expert (one 16-byte chunk of a K-major row); items
    // run expert-fastest so that the loads of a warp are coalesced.  A thread
    // loads up to IB items at once; the first round is issued before the x
    // prefill so that these loads do not queue behind the x stream.
    {
        const float *wt = a.wr + (long long)t * d * a.E;
        const int items = (d / 8) * EP;
        constexpr int IB = 12;
        float v[IB][8];
        auto load_round = [&](int i0) {
#pragma unroll
            for (int q = 0; q < IB; ++q) {
                const int i = i0 + q * RC_THREADS;
                const int e = i % EP, kc = i / EP;
#pragma unroll
                for (int r = 0; r < 8; ++r)
                    v[q][r] = (i < items && e < a.E) ? __ldg(wt + (long long)(kc * 8 + r) * a.E + e) : 0.0f;
            }
        };
        auto store_round = [&](int i0) {
#pragma unroll
            for (int q = 0; q < IB; ++q) {
                const int i = i0 + q * RC_THREADS;
                if (i >= items) continue;
                const int e = i % EP, kc = i / EP, kb = kc >> 3, ch = kc & 7;
                uint32_t hi[4], mid[4], lo[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const __nv_bfloat162 h = __floats2bfloat162_rn(v[q][2 * j], v[q][2 * j + 1]);
                    const float2 hf = __bfloat1622float2(h);
                    const float r0 = v[q][2 * j] - hf.x, r1 = v[q][2 * j + 1] - hf.y;
                    const __nv_bfloat162 m = __floats2bfloat162_rn(r0, r1);
                    const float2 mf = __bfloat1622float2(m);
                    const __nv_bfloat162 l = __floats2bfloat162_rn(r0 - mf.x, r1 - mf.y);
                    hi[j] = *reinterpret_cast<const uint32_t *>(&h);
                    mid[j] = *reinterpret_cast<const uint32_t *>(&m);
                    lo[j] = *reinterpret_cast<const uint32_t *>(&l);
                }
                const uint32_t off = (uint32_t)e * 128u + (uint32_t)((ch ^ (e & 7)) * 16);
                uint8_t *tile0 = wsm + (size_t)(kb * 3) * EP * 128;
                *reinterpret_cast<uint4 *>(tile0 + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
                *reinterpret_cast<uint4 *>(tile0 + EP * 128 + off) = make_uint4(mid[0], mid[1], mid[2], mid[3]);
                *reinterpret_cast<uint4 *>(tile0 + 2 * EP * 128 + off) = make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
        };
        load_round(tid);
        if (warp == 0 && lane == 0) {
            for (int s = 0; s < RC_MAX_STAGES; ++s) last_i[s] = -1;
            for (int i = 0; i < prefill; ++i) {  // fresh slots: nothing to wait for
                issue(i);
                last_i[i] = i;
            }
        }
        store_round(tid);
        for (int i0 = tid + IB * RC_THREADS; i0 < items; i0 += IB * RC_THREADS) {
            load_round(i0);
            store_round(i0);
        }
        fence_proxy_async();  // the split is read by the tensor cores (async proxy)
    }
    __syncthreads();

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            for (int i = prefill; i < total; ++i) {
                const int s = i % S;
                if (!wait_phase(bar_empty(s), (uint32_t)((i / S) & 1) ^ 1u, abort_flag, a.status)) break;
                issue(i);
                last_i[s] = i;
            }
            if (*abort_flag) {  // let copies in flight land before the CTA exits
                int dummy = 0;
                for (int s = 0; s < S; ++s) {
                    if (last_i[s] < 0) continue;
                    const unsigned long long t0 = global_ns();
                    while (!mbar_try_wait(bar_full(s), (uint32_t)((last_i[s] / S) & 1)) &&
                           global_ns() - t0 < 100000000ull)
                        ++dummy;
                }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        bool ok = true;
        for (int j = 0; j < ntiles && ok; ++j) {
            const int acc = j & 1;
            if (!wait_phase(bar_tempty(acc), (uint32_t)((j >> 1) & 1) ^ 1u, abort_flag, a.status)) break;
            tc_fence_after();
            const uint32_t dtmem = tmem_base + (uint32_t)(acc * NW);
            for (int kb = 0; kb < NKB; ++kb) {
                const int i = j * NKB + kb, s = i % S;
                if (!wait_phase(bar_full(s), (uint32_t)((i / S) & 1), abort_flag, a.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (lane == 0) {
                    const uint32_t sa = x_addr + s * RC_SLOT;
                    const uint32_t sb = w_addr + (uint32_t)(kb * NW) * 128;
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)
                        mma_bf16(dtmem, sdesc_sw128(sa + kk * 32, 16, 1024), sdesc_sw128(sb + kk * 32, 16, 1024),
                                 IDESC, (kb | kk) != 0 ? 1u : 0u);
                    mma_commit(bar_empty(s));
                }
                __syncwarp();
            }
            if (!ok) break;
            if (lane == 0) mma_commit(bar_tfull(acc));
            __syncwarp();
        }
        if (lane == 0) {  // all MMAs of this CTA complete before TMEM is freed
            mma_commit(bar_drain);
            const unsigned long long t0 = global_ns();
            while (!mbar_try_wait(bar_drain, 0) && global_ns() - t0 < 1000000000ull) {
            }
        }
        __syncwarp();
    } else if (warp >= 4) {
        // ------------------------------------------------------------ epilogue
        const int q = warp & 3;  // TMEM lane quarter of this warp
        const int E = a.E;
        float bv[EP];  // the task's bias (0 past E or without one)
#pragma unroll
        for (int e = 0; e < EP; ++e) bv[e] = (a.bias && e < E) ? __ldg(a.bias + (long long)t * E + e) : 0.0f;
        for (int j = 0; j < ntiles; ++j) {
            const int acc = j & 1;
            if (!wait_phase(bar_tfull(acc), (uint32_t)((j >> 1) & 1), abort_flag, a.status)) break;
            tc_fence_after();
            // parts: columns [0, EP) hi, [EP, 2 EP) mid, [2 EP, 3 EP) lo; sum
            // lo + mid, then + hi
            const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * NW);
            float w[EP];
            if constexpr (EP <= 32) {
                uint32_t r[3][NB16][16];
#pragma unroll
                for (int sp = 0; sp < 3; ++sp)
#pragma unroll
                    for (int h = 0; h < NB16; ++h) tmem_ld16(taddr + sp * EP + 16 * h, r[sp][h]);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < EP; ++e)
                    w[e] = (__uint_as_float(r[2][e >> 4][e & 15]) + __uint_as_float(r[1][e >> 4][e & 15])) +
                           __uint_as_float(r[0][e >> 4][e & 15]);
            } else {
                uint32_t r[NB16][16];
#pragma unroll
                for (int h = 0; h < NB16; ++h) tmem_ld16(taddr + 2 * EP + 16 * h, r[h]);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < EP; ++e) w[e] = __uint_as_float(r[e >> 4][e & 15]);
#pragma unroll
                for (int h = 0; h < NB16; ++h) tmem_ld16(taddr + EP + 16 * h, r[h]);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < EP; ++e) w[e] += __uint_as_float(r[e >> 4][e & 15]);
#pragma unroll
                for (int h = 0; h < NB16; ++h) tmem_ld16(taddr + 16 * h, r[h]);
                tmem_ld_wait();
#pragma unroll
                for (int e = 0; e < EP; ++e) w[e] += __uint_as_float(r[e >> 4][e & 15]);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_tempty(acc));
            const int n = n_begin + j * RC_TOK + q * 32 + lane;
            if (n < n_end) {
#pragma unroll
                for (int e = 0; e < EP; ++e) w[e] += bv[e];
                const long long tok = (long long)t * a.N + n;
                float *lrow = a.logits + tok * E;
                if ((E & 3) == 0) {
#pragma unroll
                    for (int e = 0; e < EP; e += 4)
                        if (e < E) *reinterpret_cast<float4 *>(lrow + e) = make_float4(w[e], w[e + 1], w[e + 2], w[e + 3]);
                } else {
#pragma unroll
                    for (int e = 0; e < EP; ++e)
                        if (e < E) lrow[e] = w[e];
                }
                topk_regs<EP>(a, w, tok);
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem_base, TMEM_COLS);
}

template <int EP>
int launch_ep(const Dims &p, const __nv_bfloat16 *x, const float *wr, const float *bias, float *logits,
              int32_t *idx, float *gate, cudaStream_t s) {
    const size_t wbytes = rc_w_bytes(p.d, EP);
    int stages = (int)((RC_SMEM_CAP - RC_FIXED - (long long)wbytes) / RC_SLOT);
    if (stages > RC_MAX_STAGES) stages = RC_MAX_STAGES;
    if (stages < 2) return VMOE_ERR_UNSUPPORTED;
    const size_t smem = RC_FIXED + wbytes + (size_t)stages * RC_SLOT;
    CUtensorMap tmX, tmX128;
    if (!make_map(&tmX, x, (uint64_t)p.d, (uint64_t)p.N, (uint64_t)p.T, RC_BOX) ||
        !make_map(&tmX128, x, (uint64_t)p.d, (uint64_t)p.N, (uint64_t)p.T, RC_TOK))
        return VMOE_ERR_CUDA;
    static std::atomic<int> smem_limit[64];
    if (const int st = raise_smem_limit((const void *)route_tc_kernel<EP>, smem_limit, (int)smem)) return st;
    RcArgs a = {};
    a.T = p.T;
    a.N = p.N;
    a.d = p.d;
    a.E = p.E;
    a.k = p.k;
    a.flags = p.flags;
    a.units = (p.N + RC_BOX - 1) / RC_BOX;
    int cpt = num_sms() / p.T;
    a.cpt = cpt < 1 ? 1 : (cpt > a.units ? a.units : cpt);
    a.stages = stages;
    a.wr = wr;
    a.bias = bias;
    a.logits = logits;
    a.idx = idx;
    a.gate = gate;
    a.status = device_status_word();
    trace_before(s, "route_topk");
    const int st = launch_kernel(route_tc_kernel<EP>, dim3((unsigned)(p.T * a.cpt)), dim3(RC_THREADS), smem, s,
                                 tmX, tmX128, a);
    trace_after(s);
    return st;
}

}  // namespace

// The expert count rounded up to 16 (the MMA's N), or 0 when the tcgen05
// router does not take the problem: d a multiple of 64, E <= 64, the split
// weights and two x slots within shared memory.
int route_tc_width(const Dims &p) {
    if (!p.bf16 || p.d % BK != 0 || p.d <= 0 || p.E < 1 || p.E > 64 || p.k < 1 || p.k > 8) return 0;
    const int ep = (p.E + 15) / 16 * 16;
    const int EP = ep == 48 ? 64 : ep;
    if ((long long)RC_FIXED + (long long)rc_w_bytes(p.d, EP) + 2LL * RC_SLOT > RC_SMEM_CAP) return 0;
    return EP;
}

int launch_route_tc(const Dims &p, const __nv_bfloat16 *x, const float *wr, const float *bias, float *logits,
                    int32_t *idx, float *gate, cudaStream_t s) {
    switch (route_tc_width(p)) {
        case 16: return launch_ep<16>(p, x, wr, bias, logits, idx, gate, s);
        case 32: return launch_ep<32>(p, x, wr, bias, logits, idx, gate, s);
        case 64: return launch_ep<64>(p, x, wr, bias, logits, idx, gate, s);
        default: return VMOE_ERR_UNSUPPORTED;
    }
}

}  // namespace vmoe
