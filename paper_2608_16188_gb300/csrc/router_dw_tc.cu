// router_dw_tc.cu -- dW_r = x^T dlogit and dbias of the router backward on the
// sm_103a tensor cores (tcgen05, TMEM, TMA): the gradient of the router
// weights and bias (Section 3.1 adapts the gating network with the rest of the
// visual module; Section 2.1: logits = x W_r + b, gates a softmax of them).
//
// Per task t and 128-row slice of d:  D [128 x 3E] = x[t][:, slice]^T P[t],
// where P stacks the three bf16 parts of the fp32 dlogit along N:
// hi = bf16(dl), mid = bf16(dl - hi), lo = bf16(dl - hi - mid), together about
// 24 significant bits.  x is exact in bf16, so every product is exact in fp32
// and the MMA accumulates in fp32; dW_r = (D_lo + D_mid) + D_hi.
//   A = x (M = the slice's d rows, K = tokens): MN-major, by TMA, 64 tokens
//       per k-block.
//   B = P (K = tokens, N = 3E): K-major, written by the converter warps
//       straight into the 128-byte-swizzled operand layout as they split
//       dlogit (which they also sum for dbias).  A k-block's dlogit rows are
//       one contiguous span of 64 E floats, brought into the same stage as x
//       by one bulk copy, so the converters read shared memory only.
// The tokens of a task are split over the RW_RS CTAs of a thread-block
// cluster; their partial tiles and dbias partials are summed through
// distributed shared memory in rank order: deterministic, no atomics.
//
// Roles (192 threads): warp 0 TMA producer, warp 1 MMA issuer, warps 2-5
// converters and then the epilogue (one TMEM lane = one d row each).  Every
// wait is bounded in time; a wait that runs out sets the library's status
// word, and every thread still reaches the cluster barriers.
#include <cooperative_groups.h>

#include "gemm_tc.cuh"

namespace cg = cooperative_groups;

namespace vmoe {
namespace {

using namespace tc;

// CTAs per cluster (the token split): 2, so that at 17 ViT-B tasks the 204 CTAs
// (two fit an SM) run as one wave; 3 made 306, two more than fit.
constexpr int RW_RS = 2;
constexpr int RW_STAGES = 3;   // operand ring depth
constexpr int RW_THREADS = 192;
constexpr int RW_KB = 64;      // tokens per k-block

// 1-D bulk copy global -> shared memory, completing on an mbarrier (both
// addresses 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar) {
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
                     dst),
                 "l"(src), "r"(bytes), "r"(bar)
                 : "memory");
}

template <int E>
struct RwShape {
    static constexpr int NP = 3 * E;                      // MMA N: three parts of E experts
    static constexpr uint32_t A_BYTES = 128 * RW_KB * 2;  // x: 2 chunks of 64 d x 64 tokens
    static constexpr uint32_t B_BYTES = NP * RW_KB * 2;   // P: NP rows of 64 tokens
    static constexpr uint32_t DL_BYTES = RW_KB * E * 4;   // the k-block's dlogit rows (fp32)
    static constexpr uint32_t STAGE = A_BYTES + B_BYTES + DL_BYTES;
    static constexpr uint32_t TMEM_COLS = NP <= 128 ? 128 : 256;
    static constexpr int RP = E + 1;                      // partial-tile row pitch (floats)
    static constexpr int NUM_BARS = 3 * RW_STAGES + 2;    // fullA, fullB, empty; tfull, drain
    // the partial tile [128][RP] reuses stage 0 once every MMA is done
    static constexpr size_t SMEM = 1024 + (size_t)RW_STAGES * STAGE + 4 * E * 4 + E * 4 + NUM_BARS * 8 + 16;
    static_assert(STAGE % 1024 == 0, "stages stay 1024-byte aligned");
    static_assert(128 * RP * 4 <= STAGE, "the partial tile fits a stage");
    static_assert(NP % 16 == 0 && NP <= 256, "MMA N");
};

template <int E>
__global__ void __cluster_dims__(RW_RS, 1, 1) __launch_bounds__(RW_THREADS, 1)
router_dw_tc_kernel(const __grid_constant__ CUtensorMap tmX, Dims p, const float *__restrict__ dl,
                    float *__restrict__ dw, float *__restrict__ dbias, int *status) {
    using S = RwShape<E>;
    constexpr int NP = S::NP, RP = S::RP;
    constexpr uint32_t IDESC = idesc_bf16(128, NP, true, false);  // A MN-major, B K-major
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
    float *part = reinterpret_cast<float *>(smem);  // [128][RP], after the main loop
    float *bpart = reinterpret_cast<float *>(smem + RW_STAGES * S::STAGE);  // [4][E]
    float *bsum = bpart + 4 * E;                                            // [E]
    uint64_t *bars = reinterpret_cast<uint64_t *>(bsum + E);
    int *misc = reinterpret_cast<int *>(bars + S::NUM_BARS);  // [0] tmem base, [1] abort
    auto bar_fa = [&](int s) { return smem_u32(bars + s); };
    auto bar_fb = [&](int s) { return smem_u32(bars + RW_STAGES + s); };
    auto bar_em = [&](int s) { return smem_u32(bars + 2 * RW_STAGES + s); };
    const uint32_t bar_tfull = smem_u32(bars + 3 * RW_STAGES);
    const uint32_t bar_drain = smem_u32(bars + 3 * RW_STAGES + 1);
    volatile int *abort_flag = misc + 1;

    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = p.d, N = p.N;
    const int t = blockIdx.z, d0 = blockIdx.y * 128;
    const int n_beg = (int)((long long)N * rank / RW_RS);
    const int n_end = (int)((long long)N * (rank + 1) / RW_RS);
    const int nkb = (n_end - n_beg + RW_KB - 1) / RW_KB;

    if (tid == 0) {
        for (int s = 0; s < RW_STAGES; ++s) {
            mbar_init(bar_fa(s), 1);
            mbar_init(bar_fb(s), 4);
            mbar_init(bar_em(s), 1);
        }
        mbar_init(bar_tfull, 1);
        mbar_init(bar_drain, 1);
        misc[1] = 0;
        fence_barrier_init();
        fence_proxy_async();
        prefetch_map(&tmX);
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(misc), S::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = (uint32_t)misc[0];

    if (warp == 0) {
        // ------------------------------------------------------------ producer: x k-blocks
        if (lane == 0) {
            int issued[RW_STAGES] = {};
            for (int kb = 0; kb < nkb; ++kb) {
                const int s = kb % RW_STAGES;
                if (!wait_phase(bar_em(s), (uint32_t)((kb / RW_STAGES) & 1) ^ 1u, abort_flag, status)) break;
                const int n0 = n_beg + kb * RW_KB, rem = min(RW_KB, n_end - n0);
                const uint32_t sa = smem_u32(smem) + s * S::STAGE;
                const uint32_t dl_bytes = (uint32_t)rem * E * 4;  // this rank's tokens only
                mbar_expect_tx(bar_fa(s), S::A_BYTES + dl_bytes);
                tma_load_4d(sa, &tmX, bar_fa(s), 0, n0, d0 / 64, t);
                bulk_load(sa + S::A_BYTES + S::B_BYTES, dl + ((long long)t * N + n0) * E, dl_bytes, bar_fa(s));
                ++issued[s];
            }
            if (*abort_flag) {  // let copies in flight land
                const unsigned long long t0 = global_ns();
                for (int s = 0; s < RW_STAGES; ++s)
                    if (issued[s] > 0)
                        while (!mbar_try_wait(bar_fa(s), (uint32_t)((issued[s] - 1) & 1)) &&
                               global_ns() - t0 < 100000000ull) {
                        }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        bool ok = true;
        for (int kb = 0; kb < nkb && ok; ++kb) {
            const int s = kb % RW_STAGES;
            const uint32_t ph = (uint32_t)((kb / RW_STAGES) & 1);
            if (!wait_phase(bar_fa(s), ph, abort_flag, status) || !wait_phase(bar_fb(s), ph, abort_flag, status)) {
                ok = false;
                break;
            }
            tc_fence_after();
            uint8_t *st = smem + s * S::STAGE;
            const int rem = min(RW_KB, n_end - (n_beg + kb * RW_KB));  // tokens of this rank here
            const int nk = (rem + 15) >> 4;
            if (rem < nk * 16) {  // rows [rem, 16 nk) of x belong to the next rank: zeroed
                const int rows = nk * 16 - rem, units = 2 * rows * 8;
                for (int i = lane; i < units; i += 32) {
                    const int c = i / (rows * 8), w = i - c * rows * 8;
                    *reinterpret_cast<uint4 *>(st + c * 8192 + (rem + (w >> 3)) * 128 + (w & 7) * 16) =
                        make_uint4(0, 0, 0, 0);
                }
                fence_proxy_async();
            }
            __syncwarp();
            if (lane == 0) {
                const uint32_t sa = smem_u32(st), sb = sa + S::A_BYTES;
                for (int kk = 0; kk < nk; ++kk)
                    mma_bf16(tmem_base, operand_desc(sa, kk, true), operand_desc(sb, kk, false), IDESC,
                             (kb | kk) != 0 ? 1u : 0u);
                mma_commit(bar_em(s));
            }
            __syncwarp();
        }
        if (lane == 0) {
            if (ok && nkb > 0) mma_commit(bar_tfull);
            else mbar_arrive(bar_tfull);  // nothing accumulated: the epilogue writes zeros
            mma_commit(bar_drain);
            const unsigned long long t0 = global_ns();
            while (!mbar_try_wait(bar_drain, 0) && global_ns() - t0 < 1000000000ull) {
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ converters, then epilogue
        const int cw = warp - 2;  // 16 tokens of each k-block
        float bacc[E / 32];
#pragma unroll
        for (int ec = 0; ec < E / 32; ++ec) bacc[ec] = 0.0f;
        for (int kb = 0; kb < nkb; ++kb) {
            const int s = kb % RW_STAGES;
            if (!wait_phase(bar_fa(s), (uint32_t)((kb / RW_STAGES) & 1), abort_flag, status)) break;
            uint8_t *bt = smem + s * S::STAGE + S::A_BYTES;
            const float *dls = reinterpret_cast<const float *>(bt + S::B_BYTES);  // [64][E]
            const int rem = min(RW_KB, n_end - (n_beg + kb * RW_KB));  // rows past rem were not copied
#pragma unroll
            for (int ec = 0; ec < E / 32; ++ec) {
                const int e = ec * 32 + lane;
                float v[16];
#pragma unroll
                for (int r = 0; r < 16; ++r) {
                    const int i = cw * 16 + r;
                    v[r] = i < rem ? dls[i * E + e] : 0.0f;
                    bacc[ec] += v[r];
                }
#pragma unroll
                for (int u8 = 0; u8 < 2; ++u8) {  // 8 tokens = one 16-byte unit of each part row
                    uint32_t w[3][4];
#pragma unroll
                    for (int j = 0; j < 4; ++j) {
                        const float a0 = v[u8 * 8 + 2 * j], a1 = v[u8 * 8 + 2 * j + 1];
                        const __nv_bfloat162 h = __floats2bfloat162_rn(a0, a1);
                        const float2 hf = __bfloat1622float2(h);
                        const float r0 = a0 - hf.x, r1 = a1 - hf.y;
                        const __nv_bfloat162 m = __floats2bfloat162_rn(r0, r1);
                        const float2 mf = __bfloat1622float2(m);
                        const __nv_bfloat162 l = __floats2bfloat162_rn(r0 - mf.x, r1 - mf.y);
                        w[0][j] = *reinterpret_cast<const uint32_t *>(&h);
                        w[1][j] = *reinterpret_cast<const uint32_t *>(&m);
                        w[2][j] = *reinterpret_cast<const uint32_t *>(&l);
                    }
                    const int unit = cw * 2 + u8;
#pragma unroll
                    for (int sp = 0; sp < 3; ++sp) {
                        const int row = sp * E + e;
                        *reinterpret_cast<uint4 *>(bt + row * 128 + ((unit ^ (row & 7)) << 4)) =
                            make_uint4(w[sp][0], w[sp][1], w[sp][2], w[sp][3]);
                    }
                }
            }
            fence_proxy_async();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_fb(s));
        }
#pragma unroll
        for (int ec = 0; ec < E / 32; ++ec) bpart[cw * E + ec * 32 + lane] = bacc[ec];
        // epilogue: this thread's row of the slice, the three parts summed
        const int q = warp & 3, row = q * 32 + lane;
        const bool have = wait_phase(bar_tfull, 0, abort_flag, status) && nkb > 0;
        tc_fence_after();
#pragma unroll
        for (int ec = 0; ec < E / 32; ++ec) {
            uint32_t rh[32], rm[32], rl[32];
            if (have) {
                const uint32_t ta = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(ec * 32);
                tmem_ld32(ta, rh);
                tmem_ld32(ta + E, rm);
                tmem_ld32(ta + 2 * E, rl);
                tmem_ld_wait();
            }
#pragma unroll
            for (int j = 0; j < 32; ++j)
                part[row * RP + ec * 32 + j] =
                    have ? (__uint_as_float(rl[j]) + __uint_as_float(rm[j])) + __uint_as_float(rh[j]) : 0.0f;
        }
        tc_fence_before();
        named_bar(1, 128);  // the four converter warps' dbias partials are in place
        if (tid - 64 < E) {
            const int e = tid - 64;
            bsum[e] = ((bpart[e] + bpart[E + e]) + bpart[2 * E + e]) + bpart[3 * E + e];
        }
    }

    cluster.sync();  // every rank's partial tile and dbias partial is complete
    // rank r sums rows [r ROWS, (r + 1) ROWS) of the slice over the ranks, in rank order
    constexpr int ROWS = (128 + RW_RS - 1) / RW_RS;
    float *dwt = dw + (long long)t * d * E;
    for (int v = tid; v < ROWS * E; v += RW_THREADS) {  // (part is stage 0: every MMA is done)
        const int m = rank * ROWS + v / E, n = v % E;
        if (m >= 128) continue;
        float sum = 0.0f;
#pragma unroll
        for (int r = 0; r < RW_RS; ++r) sum += cluster.map_shared_rank(part, r)[m * RP + n];
        if (d0 + m < d) dwt[(long long)(d0 + m) * E + n] = sum;
    }
    if (dbias != nullptr && blockIdx.y == 0 && rank == 0 && tid < E) {
        float b = 0.0f;
#pragma unroll
        for (int r = 0; r < RW_RS; ++r) b += cluster.map_shared_rank(bsum, r)[tid];
        dbias[(long long)t * E + tid] = b;
    }
    cluster.sync();  // every rank's shared memory stays alive until the remote reads are done
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem_base, S::TMEM_COLS);
}

template <int E>
int launch_rw(const Dims &p, const __nv_bfloat16 *x, const float *dl, float *dw, float *dbias, cudaStream_t s) {
    using S = RwShape<E>;
    static std::atomic<int> smem_limit[64];
    if (const int st = raise_smem_limit((const void *)router_dw_tc_kernel<E>, smem_limit, (int)S::SMEM))
        return st;
    CUtensorMap mx;  // x [T][N][d] as {64, N, d / 64, T}: 64-token boxes of two 64-wide d chunks
    if (!make_map_chunked(&mx, x, p.d, p.N, p.T, RW_KB, 2)) return VMOE_ERR_CUDA;
    dim3 grid(RW_RS, p.d / 128, p.T);
    router_dw_tc_kernel<E><<<grid, RW_THREADS, S::SMEM, s>>>(mx, p, dl, dw, dbias, device_status_word());
    return launch_result();
}

}  // namespace

// The tensor-core router weight gradient, or VMOE_ERR_UNSUPPORTED where it does
// not apply (then the caller runs the mma.sync kernel): bf16 x, E = 32 or 64,
// d a multiple of 128.
int launch_router_dw_tc(const Dims &p, const __nv_bfloat16 *x, const float *dl, float *dw, float *dbias,
                        cudaStream_t s) {
    if (!p.bf16 || p.d % 128 != 0 || p.N < 1) return VMOE_ERR_UNSUPPORTED;
    if (p.E == 32) return launch_rw<32>(p, x, dl, dw, dbias, s);
    if (p.E == 64) return launch_rw<64>(p, x, dl, dw, dbias, s);
    return VMOE_ERR_UNSUPPORTED;
}

}  // namespace vmoe
