// gemm_tc2.cuh -- the weight gradients of the expert FFN (dW1 = Xe^T dH,
// dW2 = A^T dYe) on pairs of SMs: tcgen05.mma with cta_group::2, one
// 256 x 256 output tile per MMA, the B operand resident per work unit.
//
//   D[g][M][N] = A[g][K rows][M]^T B[g][K rows][N],  K = load[g] rows
//
// A thread-block cluster of two CTAs (ranks 0 and 1) works on one 256 x 256
// tile at a time: CTA r holds rows [128 r, 128 r + 128) of the tile's A^T
// (A columns) and columns [128 r, 128 r + 128) of its B, and its TMEM holds
// output rows [128 r, 128 r + 128) x 256 columns.  Against one SM per 128 x 256
// tile this halves the B bytes each SM loads per output byte, which leaves room
// in shared memory for a second resident B buffer: the next unit's B tile
// loads while this unit's MMAs run, instead of stalling the pair at every unit
// boundary.
//
// One work unit = (group, 256-column tile): its B tile -- every K row, and with
// KSPLIT the residual rows after them -- is loaded once and reused by all M/256
// row tiles of the group; their A k-blocks stream through a ring.
//
// Roles, per CTA (320 threads):
//   warp 0      TMA producer: its own A and B halves into its own shared memory.
//               A k-blocks complete on the leader's `afull` (both CTAs' bytes).
//               With two B buffers a B tile completes on this CTA's own `bfull`;
//               with one (K > 128 rows) each k-block piece of a dense B tile
//               completes on the leader's `bfull` of that piece, like A.
//   warp 1      B hand-over: with two B buffers (and for compact B) it waits for
//               this CTA's B copy, zeroes the rows of a compact B's first
//               k-block that belong to a neighbour, then arrives on the leader's
//               `bready` (count 2: both CTAs).  In the leader (rank 0) lane 0
//               also issues the MMAs once both CTAs' operands are in and commits
//               them with a multicast arrive on both CTAs' `aempty`, `bempty`
//               (per piece with one B buffer) and `tfull`.
//   warps 2-9   epilogue: tcgen05.ld of this CTA's 128 accumulator rows, arrive on
//               the leader's `tempty` (count 16: 8 warps x 2 CTAs), bf16 packing
//               and TMA bulk tensor stores from 128-byte-swizzled staging.
//               Units of an empty group (load 0) are written as zeros by the
//               epilogue alone; they take no MMA and no accumulator.
// Every wait is bounded in time as in grouped_gemm_kernel.  A CTA that gives up
// also raises its peer's abort flag, both CTAs leave their loops, meet at the
// closing cluster barrier and free the TMEM pair together.
#pragma once

#include "gemm_tc.cuh"

namespace vmoe {
namespace tc {

__device__ __forceinline__ uint32_t cluster_ctarank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// Address of the same shared-memory variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t mapa_shared(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
// Arrive on an mbarrier that may live in the peer CTA (release at cluster scope).
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr)
                 : "memory");
}
__device__ __forceinline__ bool mbar_try_wait_cluster(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.acquire.cluster.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
// Bounded wait with acquire at cluster scope (barriers the peer CTA arrives on).
static __device__ __noinline__ bool wait_phase_cluster(uint32_t bar, uint32_t parity,
                                                       volatile int *abort_flag, int *status) {
    if (mbar_try_wait_cluster(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait_cluster(bar, parity)) return true;
        if ((i & 63u) == 0) {
            if (*abort_flag) return false;
            if (global_ns() - t0 > TIMEOUT_NS) {
                *abort_flag = 1;
                if (status) atomicExch(status, (int)VMOE_ERR_DEVICE_TIMEOUT);
                return false;
            }
        }
    }
}
__device__ __forceinline__ void st_cluster_u32(uint32_t cluster_addr, uint32_t v) {
    asm volatile("st.relaxed.cluster.shared::cluster.u32 [%0], %1;" ::"r"(cluster_addr), "r"(v) : "memory");
}
__device__ __forceinline__ void cluster_sync_all() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                     : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void mma_pair_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                              uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive on barrier `bar` (same offset) in both CTAs of the pair once every
// MMA issued so far by this thread has completed.
__device__ __forceinline__ void mma_pair_commit_both(uint32_t bar) {
    const uint16_t mask = 3;
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 "
        "[%0], %1;" ::"r"(bar),
        "h"(mask)
        : "memory");
}
__device__ __forceinline__ void mma_pair_commit_local(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

// TMA load into this CTA's shared memory whose completion (bytes) is signalled
// on an mbarrier of either CTA of the pair -- here the leader's.
__device__ __forceinline__ void tma_load_4d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar_cluster,
                                                 int c0, int c1, int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}
// Plain remote arrive (release at CTA scope), for barriers whose waiter orders
// through tcgen05 fences rather than through memory.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t cluster_addr) {
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}

// Shared memory of the pair kernel, per CTA.  KB = one k-block (64 K rows) of
// 128 columns = 16 KB, for A and B alike.  The B region holds one or two
// resident B tiles (NKB k-blocks, twice with KSPLIT); what is left of a 224 KB
// budget goes to the A ring and the epilogue staging.
//   dW1, C <= 128 (KSPLIT, NKB 2): B 2 x 64 KB, A 4 slots, staging 32 KB
//   dW1, C <= 256 (KSPLIT, NKB 4): B 1 x 128 KB, A 4 slots, staging 32 KB
//   dW2, C <= 128 (NKB 2):         B 2 x 32 KB, A 6 slots, staging 2 x 32 KB
//   dW2, C <= 256 (NKB 4):         B 1 x 64 KB, A 6 slots, staging 2 x 32 KB
template <bool KSPLIT, int NKB>
struct PairShape {
    static constexpr int MP = 256;                  // tile rows (MMA M), 128 per CTA
    static constexpr int BN = 256;                  // tile columns (MMA N), 128 per CTA
    static constexpr uint32_t KB = 64 * 128 * 2;    // one k-block of one operand half
    static constexpr uint32_t B_BUF = (KSPLIT ? 2u : 1u) * NKB * KB;
    // two B buffers for tiles of at most 128 K rows; a tile of more rows is
    // held once and refilled piece by piece (its shared memory goes to a
    // double-buffered epilogue staging where it fits)
    static constexpr int B_BUFS = (B_BUF <= 65536u && NKB <= 2) ? 2 : 1;
    static constexpr uint32_t BUDGET = 224u * 1024u;
    static constexpr uint32_t REST = BUDGET - B_BUFS * B_BUF;
    static constexpr int STG_BUFS = REST >= 160u * 1024u ? 2 : 1;
    static constexpr int A_SLOTS = (int)((REST - STG_BUFS * 32768u) / KB);
    static constexpr uint32_t EPI_BYTES = 8u * STG_BUFS * 4096u;
    static constexpr uint32_t TMEM_COLS = 2 * BN;
    static constexpr int NUM_BARS = 2 * A_SLOTS + 3 * B_BUFS * (B_BUFS == 1 ? NKB : 1) + 5;
    static constexpr size_t SMEM_BYTES =
        1024 + (size_t)B_BUFS * B_BUF + (size_t)A_SLOTS * KB + EPI_BYTES + NUM_BARS * 8 + 16;
    static_assert(A_SLOTS >= 2, "A ring too shallow");
    static_assert(SMEM_BYTES <= 232448, "over the 227 KB shared-memory limit");
};

// Which units each SM pair works on.  By default (enabled = 0) pair c takes
// units c, c + P, c + 2P, ... of P pairs -- a static round-robin over units
// of nearly equal cost.  With enabled = 1 pair c takes the contiguous units
// [first[c], first[c] + count[c]): the per-group pair shares of the
// fill-clamp-refill allocation (Section 3.2.2), each group's units split
// evenly over the pairs of its share (vmoe_plan_shares; the memory-budgeted
// backward, whose loads are on the host).
constexpr int MAX_PAIRS = 128;
struct PairSchedule {
    int enabled;
    int32_t first[MAX_PAIRS];
    int32_t count[MAX_PAIRS];
};

// K rows of a group with load L are taken in nkb = ceil(L / 64) k-blocks
// aligned to the END of its rows: k-block j covers rows [L - 64 (nkb - j),
// L - 64 (nkb - j - 1)), so only k-block 0 is partial and its missing rows lie
// BEFORE row 0 of the group, where the tensor map reads zeros (a box may start
// at a negative coordinate).  No padding row [L, C) is ever loaded, so nothing
// needs zeroing and the MMAs skip the k-block's leading all-zero 16-row steps.
// (In the memory-budgeted backward B comes from a compact buffer, where the
// rows before an entry belong to its neighbour: the tail warp zeroes them.)
template <bool KSPLIT, int NKB>
__global__ void __launch_bounds__(THREADS, 1)
wgrad_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                  const __grid_constant__ CUtensorMap tmBlo, const __grid_constant__ CUtensorMap tmD,
                  Args args, const __grid_constant__ PairSchedule sched) {
    using S = PairShape<KSPLIT, NKB>;
    constexpr uint32_t IDESC = idesc_bf16(S::MP, S::BN, true, true);
    constexpr int AS = S::A_SLOTS, BB = S::B_BUFS;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
    uint8_t *b_res = smem;                            // BB x [part][kb] k-blocks
    uint8_t *a_ring = b_res + BB * S::B_BUF;          // AS k-blocks
    uint8_t *epi_base = a_ring + AS * S::KB;
    uint64_t *bars = reinterpret_cast<uint64_t *>(epi_base + S::EPI_BYTES);
    int *misc = reinterpret_cast<int *>(bars + S::NUM_BARS);  // [0] tmem base, [1] abort
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    auto bar = [&](int i) { return smem_u32(bars + i); };
    // afull: the leader's counts both CTAs' bytes of the slot (the peer's is unused)
    auto bar_afull = [&](int i) { return bar(i); };
    auto bar_aempty = [&](int i) { return bar(AS + i); };
    // B barriers.  Two buffers: one piece per buffer (the whole tile), handed
    // to the leader by the tail warp once both CTAs' copies landed.  One
    // buffer: one piece per k-block, each released by the last row tile's
    // MMAs on it, so that the next unit's B streams in piece by piece behind
    // that row tile; dense pieces complete on the leader's barrier, like A,
    // and need no hand-over.
    constexpr bool PIECES = BB == 1;
    constexpr int NPC = PIECES ? NKB : 1;  // B pieces per buffer
    constexpr int BP = BB * NPC;
    auto bar_bfull = [&](int bb, int pc) { return bar(2 * AS + bb * NPC + pc); };
    auto bar_bempty = [&](int bb, int pc) { return bar(2 * AS + BP + bb * NPC + pc); };
    auto bar_bready = [&](int bb, int pc) { return bar(2 * AS + 2 * BP + bb * NPC + pc); };
    auto bar_tfull = [&](int i) { return bar(2 * AS + 3 * BP + i); };
    auto bar_tempty = [&](int i) { return bar(2 * AS + 3 * BP + 2 + i); };
    const uint32_t bar_drain = bar(2 * AS + 3 * BP + 4);
    volatile int *abort_flag = misc + 1;
    // the peer's abort flag, raised when this CTA gives up
    const uint32_t peer_abort = mapa_shared(smem_u32(misc + 1), rank ^ 1u);

    if (tid == 0) {
        for (int i = 0; i < AS; ++i) {
            mbar_init(bar_afull(i), 1);
            mbar_init(bar_aempty(i), 1);
        }
        for (int i = 0; i < BB; ++i)
            for (int pc = 0; pc < NPC; ++pc) {
                mbar_init(bar_bfull(i, pc), 1);
                mbar_init(bar_bempty(i, pc), 1);
                mbar_init(bar_bready(i, pc), 2);
            }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_tfull(i), 1);
            mbar_init(bar_tempty(i), 16);
        }
        mbar_init(bar_drain, 1);
        misc[1] = 0;
        fence_barrier_init();
        fence_proxy_async();
        prefetch_map(&tmA);
        prefetch_map(&tmB);
        if (KSPLIT) prefetch_map(&tmBlo);
        prefetch_map(&tmD);
    }
    if (warp == 0) {
        tmem_alloc_pair(smem_u32(misc), S::TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync_all();  // barriers initialised and TMEM allocated in both CTAs
    tc_fence_after();
    pdl_wait();  // the predecessor's outputs are complete from here on
    const uint32_t tmem_base = (uint32_t)misc[0];
    const int cid = blockIdx.x >> 1, ncl = gridDim.x >> 1;
    const int total = args.G * args.tiles_n;
    const int tiles_m = args.tiles_m;  // M / 256
    const bool cmpb = (args.compact & CMP_B) != 0;  // B rows from crow, residual after L
    // this pair's units: u = u_first, u_first + u_step, ... < u_end
    const int u_first = sched.enabled ? sched.first[cid] : cid;
    const int u_step = sched.enabled ? 1 : ncl;
    const int u_end = sched.enabled ? min(total, sched.first[cid] + sched.count[cid]) : total;
    int crow = 0;
    auto decode = [&](int u, int &g, int &n_blk, int &L) {
        const int i = u / args.tiles_n;
        g = real_group(args, i);
        crow = args.crow ? __ldg(args.crow + i) : 0;
        n_blk = u - i * args.tiles_n;
        L = __ldg(args.load + g);
        L = L < 0 ? 0 : (L > args.C ? args.C : L);
    };
    auto give_up = [&]() {
        if (*abort_flag && lane == 0) st_cluster_u32(peer_abort, 1u);
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int ub = 0, ka = 0;
            bool ok = true;
            // uses of each B piece so far (their parity gives the phase)
            int b_issued[BP] = {}, a_issued[AS] = {};
            for (int u = u_first; u < u_end && ok; u += u_step) {
                int g, n_blk, L;
                decode(u, g, n_blk, L);
                if (u + u_step >= u_end) pdl_launch_dependents();  // this pair's last unit
                const int nkb = (L + BK - 1) / BK;
                if (nkb == 0) continue;
                const int r0 = L - nkb * BK;  // first row of k-block 0 (<= 0)
                const int bb = ub % BB;
                const uint32_t bdst = smem_u32(b_res) + bb * S::B_BUF;
                const int bchunk = n_blk * 4 + (int)rank * 2;
                ++ub;
                // B piece pc = k-blocks [kb0, kb1) (and their residual), once its
                // previous use has been released by the MMAs
                auto load_b = [&](int pc, int kb0, int kb1) -> bool {
                    int &nb = b_issued[bb * NPC + pc];
                    if (!wait_phase(bar_bempty(bb, pc), (uint32_t)(nb & 1) ^ 1u, abort_flag, args.status))
                        return false;
                    ++nb;
                    const uint32_t fb = bar_bfull(bb, pc);
                    const uint32_t bytes = (KSPLIT ? 2u : 1u) * (uint32_t)(kb1 - kb0) * S::KB;
                    const bool on_leader = PIECES && !cmpb;
                    const uint32_t fbl = mapa_shared(fb, 0);
                    if (on_leader) {
                        if (leader) mbar_expect_tx(fb, 2u * bytes);  // both CTAs' halves
                    } else {
                        mbar_expect_tx(fb, bytes);
                    }
                    for (int kb = kb0; kb < kb1; ++kb) {
                        const int r = r0 + kb * BK;
                        const uint32_t d0 = bdst + kb * S::KB, d1 = bdst + (NKB + kb) * S::KB;
                        if (cmpb) {
                            tma_load_4d(d0, &tmB, fb, 0, crow + r, bchunk, 0);
                            if (KSPLIT) tma_load_4d(d1, &tmB, fb, 0, crow + L + r, bchunk, 0);
                        } else if (on_leader) {
                            tma_load_4d_pair(d0, &tmB, fbl, 0, r, bchunk, g);
                            if (KSPLIT) tma_load_4d_pair(d1, &tmBlo, fbl, 0, r, bchunk, g);
                        } else {
                            tma_load_4d(d0, &tmB, fb, 0, r, bchunk, g);
                            if (KSPLIT) tma_load_4d(d1, &tmBlo, fb, 0, r, bchunk, g);
                        }
                    }
                    return true;
                };
                // Two buffers: the whole tile at once (its buffer was freed a
                // unit ago).  One: each piece just before the first row tile's
                // A k-block that needs it.
                if (!PIECES) ok = load_b(0, 0, nkb);
                for (int m = 0; m < tiles_m && ok; ++m)
                    for (int kb = 0; kb < nkb; ++kb, ++ka) {
                        if (PIECES && m == 0 && !load_b(kb, kb, kb + 1)) {
                            ok = false;
                            break;
                        }
                        const int sl = ka % AS;
                        if (!wait_phase(bar_aempty(sl), (uint32_t)((ka / AS) & 1) ^ 1u, abort_flag,
                                        args.status)) {
                            ok = false;
                            break;
                        }
                        if (leader) mbar_expect_tx(bar_afull(sl), 2u * S::KB);  // both CTAs' halves
                        tma_load_4d_pair(smem_u32(a_ring) + sl * S::KB, &tmA, mapa_shared(bar_afull(sl), 0),
                                         0, r0 + kb * BK, m * 4 + (int)rank * 2, g);
                        ++a_issued[sl];
                    }
            }
            if (*abort_flag) {  // let copies in flight land before the CTA exits
                const unsigned long long t0 = global_ns();
                // (dense B pieces, like A, complete on the leader's barriers)
                if (leader || !PIECES || cmpb)
                    for (int i = 0; i < BP; ++i)
                        if (b_issued[i] > 0)
                            while (!mbar_try_wait(bar_bfull(i / NPC, i % NPC), (uint32_t)((b_issued[i] - 1) & 1)) &&
                                   global_ns() - t0 < 100000000ull) {
                            }
                // the leader's afull counts the peer's copies too; the peer waits
                // for the leader at the closing cluster barrier
                if (leader)
                    for (int i = 0; i < AS; ++i)
                        if (a_issued[i] > 0)
                            while (!mbar_try_wait(bar_afull(i), (uint32_t)((a_issued[i] - 1) & 1)) &&
                                   global_ns() - t0 < 200000000ull) {
                            }
            }
        }
        __syncwarp();
        give_up();
    } else if (warp == 1) {
        // ------------------------------------------------------------ B hand-over (+ MMA in the leader)
        int ub = 0, ka = 0, it = 0;
        int b_used[BP] = {};  // uses of each B piece so far (their parity gives the phase)
        bool ok = true;
        for (int u = u_first; u < u_end && ok; u += u_step) {
            int g, n_blk, L;
            decode(u, g, n_blk, L);
            const int nkb = (L + BK - 1) / BK;
            if (nkb == 0) continue;
            const int z = nkb * BK - L;  // leading rows of k-block 0 outside the group
            const int skip = z >> 4;     // all-zero 16-row steps of k-block 0
            const int bb = ub % BB;
            uint8_t *bres = b_res + bb * S::B_BUF;
            ++ub;
            // Piece pc of this unit's B: wait for this CTA's copy, zero the
            // compact-B rows of k-block 0 that belong to a neighbour, hand it
            // to the leader; the leader waits until both CTAs have.
            auto hand_over = [&](int pc) -> bool {
                const uint32_t ph = (uint32_t)(b_used[bb * NPC + pc] & 1);
                ++b_used[bb * NPC + pc];
                if (!wait_phase(bar_bfull(bb, pc), ph, abort_flag, args.status)) return false;
                if (cmpb && pc == 0 && z > 0) {
                    // compact B: rows [0, z) of k-block 0 (both parts) hold the
                    // neighbouring entry's rows; zero them (two 64-wide chunks each)
                    for (int part = 0; part < (KSPLIT ? 2 : 1); ++part) {
                        uint8_t *tile = bres + part * NKB * S::KB;
                        for (int i = lane; i < 2 * z * 8; i += 32) {
                            const int c = i / (z * 8), w = i - c * z * 8;
                            *reinterpret_cast<uint4 *>(tile + c * (BK * 128) + (w >> 3) * 128 + (w & 7) * 16) =
                                make_uint4(0, 0, 0, 0);
                        }
                    }
                    fence_proxy_async();
                }
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(mapa_shared(bar_bready(bb, pc), 0));
                return !leader || wait_phase_cluster(bar_bready(bb, pc), ph, abort_flag, args.status);
            };
            if (!PIECES || cmpb)
                for (int pc = 0; pc < (PIECES ? nkb : 1) && ok; ++pc) ok = hand_over(pc);
            if (!leader || !ok) continue;
            for (int m = 0; m < tiles_m && ok; ++m, ++it) {
                const int acc = it & 1;
                const bool last_m = m == tiles_m - 1;
                if (!wait_phase(bar_tempty(acc), (uint32_t)((it >> 1) & 1) ^ 1u, abort_flag, args.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                for (int kb = 0; kb < nkb; ++kb, ++ka) {
                    if (PIECES && !cmpb && m == 0) {  // dense B piece kb: both halves landed
                        const uint32_t ph = (uint32_t)(b_used[bb * NPC + kb] & 1);
                        ++b_used[bb * NPC + kb];
                        if (!wait_phase(bar_bfull(bb, kb), ph, abort_flag, args.status)) {
                            ok = false;
                            break;
                        }
                    }
                    const int sl = ka % AS;
                    if (!wait_phase(bar_afull(sl), (uint32_t)((ka / AS) & 1), abort_flag, args.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    if (lane == 0) {
                        const int k0 = kb == 0 ? skip : 0;
                        const uint32_t dtmem = tmem_base + (uint32_t)(acc * S::BN);
                        const uint32_t a0 = smem_u32(a_ring) + sl * S::KB;
#pragma unroll 1
                        for (int part = 0; part < (KSPLIT ? 2 : 1); ++part) {
                            const uint32_t b0 = smem_u32(bres) + (part * NKB + kb) * S::KB;
                            for (int kk = k0; kk < BK / 16; ++kk)
                                mma_pair_bf16(dtmem, operand_desc(a0, kk, true), operand_desc(b0, kk, true),
                                              IDESC, (kb | part | (kk - k0)) != 0 ? 1u : 0u);
                        }
                        mma_pair_commit_both(bar_aempty(sl));
                        // the last row tile's MMAs on a piece are its last use
                        if (PIECES && last_m) mma_pair_commit_both(bar_bempty(bb, kb));
                    }
                    __syncwarp();
                }
                if (!ok) break;
                if (lane == 0) mma_pair_commit_both(bar_tfull(acc));
                __syncwarp();
            }
            if (!ok) break;
            if (!PIECES && lane == 0) mma_pair_commit_both(bar_bempty(bb, 0));  // B may be replaced now
            __syncwarp();
        }
        if (leader && lane == 0) {  // all MMAs of the pair complete before TMEM is freed
            mma_pair_commit_local(bar_drain);
            const unsigned long long t0 = global_ns();
            while (!mbar_try_wait(bar_drain, 0) && global_ns() - t0 < 1000000000ull) {
            }
        }
        __syncwarp();
        give_up();
    } else {
        // ------------------------------------------------------------ epilogue
        const int ew = warp - 2;
        const int q = warp & 3;
        const int half = ew >> 2;
        constexpr int COLS = S::BN / 2;  // 128 columns per warp
        uint8_t *stg = epi_base + ew * S::STG_BUFS * 4096;
        int nstore = 0, it = 0;
        bool ok = true;
        for (int u = u_first; u < u_end && ok; u += u_step) {
            int g, n_blk, L;
            decode(u, g, n_blk, L);
            for (int m = 0; m < tiles_m; ++m) {
                const int row0 = m * S::MP + (int)rank * 128 + q * 32;
                const int colw = n_blk * S::BN + half * COLS;
                uint32_t r[COLS / 32][32];
                if (L > 0) {
                    const int acc = it & 1;
                    if (!wait_phase(bar_tfull(acc), (uint32_t)((it >> 1) & 1), abort_flag, args.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t trow = tmem_base + ((uint32_t)(q * 32) << 16) +
                                          (uint32_t)(acc * S::BN + half * COLS);
#pragma unroll
                    for (int i = 0; i < COLS / 32; ++i) tmem_ld32(trow + i * 32, r[i]);
                    tmem_ld_wait();
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive_remote(mapa_shared(bar_tempty(acc), 0));
                    ++it;
                } else {
#pragma unroll
                    for (int i = 0; i < COLS / 32; ++i)
#pragma unroll
                        for (int j = 0; j < 32; ++j) r[i][j] = 0u;
                }
#pragma unroll
                for (int c = 0; c < COLS / 64; ++c) {
                    uint8_t *buf = stg + (S::STG_BUFS == 2 ? (nstore & 1) * 4096 : 0);
                    if (lane == 0 && nstore >= S::STG_BUFS) {
                        if (S::STG_BUFS == 2) bulk_wait_read1();
                        else bulk_wait_read0();
                    }
                    __syncwarp();
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const uint32_t *src = &r[2 * c + (j >> 2)][(j & 3) * 8];
                        uint4 pk;
                        pk.x = pack_bf16x2(__uint_as_float(src[0]), __uint_as_float(src[1]));
                        pk.y = pack_bf16x2(__uint_as_float(src[2]), __uint_as_float(src[3]));
                        pk.z = pack_bf16x2(__uint_as_float(src[4]), __uint_as_float(src[5]));
                        pk.w = pack_bf16x2(__uint_as_float(src[6]), __uint_as_float(src[7]));
                        *reinterpret_cast<uint4 *>(buf + lane * 128 + ((j ^ (lane & 7)) << 4)) = pk;
                    }
                    fence_proxy_async();
                    __syncwarp();
                    if (lane == 0) {
                        tma_store_3d(&tmD, smem_u32(buf), colw + c * 64, row0, g);
                        bulk_commit();
                    }
                    ++nstore;
                }
            }
        }
        if (lane == 0) bulk_wait_all();
        __syncwarp();
        give_up();
    }

    tc_fence_before();
    cluster_sync_all();  // no MMA, copy or remote arrive of either CTA is still in flight
    tc_fence_after();
    if (warp == 0) tmem_dealloc_pair(tmem_base, S::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Row-mode grouped GEMM on SM pairs, for groups of more than 128 rows:
//
//   D[g][rows][N] = act[g][rows][K] * B[g],  B MN-major ([K][N]) or K-major ([N][K])
//
// A pair tile is 256 rows x BN columns (MMA M = 256): CTA r loads rows
// [128 r, 128 r + 128) of the tile's A and columns [BN/2 r, BN/2 (r + 1)) of its
// B, so each SM streams half of the weight tile a 128-row tile would need.  At
// these shapes the one-SM kernel is held back by the bytes in flight per SM,
// not by HBM: the pair both halves the bytes per output and fits a deeper ring
// (6 stages of 32 KB at BN 256, 8 of 24 KB at BN 128).  Both CTAs' copies of a
// stage complete on the leader's `full` barrier; the leader's MMA thread
// commits with a multicast arrive on both CTAs' `empty` and `tfull`; the
// epilogue is the one-SM kernel's (row-masked stores of this CTA's 128 rows,
// GELU / GELU' fused), arriving on the leader's `tempty` (count 16).
// A tile's rows past the group's load are neither loaded (A boxes of 64, 32
// and 16 rows as in the one-SM kernel) nor stored.
template <int BN, bool B_MN, int EPI>
struct RowPairShape {
    static constexpr int PM = 256;                           // rows of a pair tile
    static constexpr int BNC = BN / 2;                       // B columns per CTA
    static constexpr uint32_t A_BYTES = 128 * BK * 2;        // this CTA's 128 rows x 64 K
    static constexpr uint32_t B_BYTES = BNC * BK * 2;
    static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr int EPI_BYTES = 8 * EPI_WARP_BYTES;
    static constexpr size_t FIXED = 1024 + EPI_BYTES + 16 + THREADS * 4 + (MAX_G + 1) * 4 + 8 * 32;
    static constexpr int STAGES_FIT = (int)((232448 - FIXED) / STAGE_BYTES);
    static constexpr int STAGES = STAGES_FIT > 8 ? 8 : STAGES_FIT;
    static constexpr int NUM_BARS = 2 * STAGES + 5;
    static constexpr uint32_t TMEM_COLS = 2 * BN;
    static constexpr size_t SMEM_BYTES = 1024 + (size_t)STAGES * STAGE_BYTES + EPI_BYTES + NUM_BARS * 8 + 16 +
                                         THREADS * 4 + (MAX_G + 1) * 4;
    static_assert(SMEM_BYTES <= 232448, "over the 227 KB shared-memory limit");
};

__device__ __forceinline__ void tma_load_3d_pair(uint32_t dst, const CUtensorMap *map, uint32_t bar_cluster,
                                                 int c0, int c1, int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes.cta_group::2"
        " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar_cluster), "r"(c0), "r"(c1), "r"(c2)
        : "memory");
}

// Rows of a CTA's 128-row half that hold valid rows, rounded up to 16 (0..128).
__device__ __forceinline__ int half_rows(int rem) {
    return rem >= 128 ? 128 : (rem <= 0 ? 0 : ((rem + 15) & ~15));
}

template <int BN, bool B_MN, int EPI>
__global__ void __launch_bounds__(THREADS, 1)
row_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                const __grid_constant__ TailMaps tmAt, Args args) {
    using S = RowPairShape<BN, B_MN, EPI>;
    constexpr int STAGES = S::STAGES;
    constexpr int PM = S::PM, BNC = S::BNC;
    constexpr uint32_t IDESC = idesc_bf16(PM, BN, false, B_MN);

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
    const uint32_t tiles_addr = smem_u32(smem);
    uint8_t *epi_base = smem + STAGES * S::STAGE_BYTES;
    uint64_t *bars = reinterpret_cast<uint64_t *>(epi_base + S::EPI_BYTES);
    int *misc = reinterpret_cast<int *>(bars + S::NUM_BARS);  // [0] tmem base, [1] abort, [2] total
    int *scan_tmp = misc + 4;
    int *prefix = scan_tmp + THREADS;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;
    auto bar_full = [&](int s) { return smem_u32(bars + s); };  // the leader's counts both CTAs
    auto bar_empty = [&](int s) { return smem_u32(bars + STAGES + s); };
    auto bar_tfull = [&](int a) { return smem_u32(bars + 2 * STAGES + a); };
    auto bar_tempty = [&](int a) { return smem_u32(bars + 2 * STAGES + 2 + a); };
    const uint32_t bar_drain = smem_u32(bars + 2 * STAGES + 4);
    volatile int *abort_flag = misc + 1;
    const uint32_t peer_abort = mapa_shared(smem_u32(misc + 1), rank ^ 1u);

    if (tid == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(bar_full(s), 1);
            mbar_init(bar_empty(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(bar_tfull(a), 1);
            mbar_init(bar_tempty(a), 16);
        }
        mbar_init(bar_drain, 1);
        misc[1] = 0;
        fence_barrier_init();
        fence_proxy_async();
        prefetch_map(&tmA);
        prefetch_map(&tmB);
        for (int i = 0; i < 3; ++i) prefetch_map(&tmAt.a[i]);
    }
    if (warp == 0) {
        tmem_alloc_pair(smem_u32(misc), S::TMEM_COLS);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    cluster_sync_all();  // barriers initialised and TMEM allocated in both CTAs
    tc_fence_after();
    pdl_wait();  // the predecessor's outputs (loads, operands) are complete from here on

    // Tile count and per-group tile prefix (ceil(load / 256) x N/BN tiles a
    // group), computed alike by both CTAs.
    {
        const int G = args.G;
        const int per = (G + THREADS - 1) / THREADS;
        const int g0 = min(G, tid * per), g1 = min(G, g0 + per);
        int local = 0;
        for (int g = g0; g < g1; ++g) {
            int L = __ldg(args.load + real_group(args, g));
            L = L < 0 ? 0 : (L > args.C ? args.C : L);
            local += ((L + PM - 1) / PM) * args.tiles_n;
        }
        scan_tmp[tid] = local;
        __syncthreads();
        if (warp == 0) {
            constexpr int PER = THREADS / 32;
            int v[PER], sum = 0;
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                v[i] = scan_tmp[lane * PER + i];
                sum += v[i];
            }
            int incl = sum;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y;
            }
            int run = incl - sum;
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                scan_tmp[lane * PER + i] = run;
                run += v[i];
            }
            if (lane == 31) misc[2] = incl;
        }
        __syncthreads();
        int run = scan_tmp[tid];
        for (int g = g0; g < g1; ++g) {
            prefix[g] = run;
            int L = __ldg(args.load + real_group(args, g));
            L = L < 0 ? 0 : (L > args.C ? args.C : L);
            run += ((L + PM - 1) / PM) * args.tiles_n;
        }
        if (tid == 0) prefix[G] = misc[2];
    }
    __syncthreads();
    const int total = misc[2];
    const uint32_t tmem_base = (uint32_t)misc[0];
    const int cid = blockIdx.x >> 1, ncl = gridDim.x >> 1;
    const int kblocks = args.K_fixed / BK;
    // tile u -> entry g, real group gr, compact row crow, 256-row block m_blk, column tile n_blk, rows
    auto decode = [&](int u, int &g, int &gr, int &crow, int &m_blk, int &n_blk, int &rows_valid) {
        int lo = 0, hi = args.G;  // prefix[lo] <= u < prefix[hi]
        while (hi - lo > 1) {
            const int mid = (lo + hi) >> 1;
            if (prefix[mid] <= u) lo = mid; else hi = mid;
        }
        g = lo;
        gr = real_group(args, lo);
        crow = args.crow ? __ldg(args.crow + lo) : 0;
        const int local = u - prefix[lo];
        m_blk = local / args.tiles_n;
        n_blk = local - m_blk * args.tiles_n;
        int L = __ldg(args.load + gr);
        rows_valid = L < 0 ? 0 : (L > args.C ? args.C : L);
    };
    auto give_up = [&]() {
        if (*abort_flag && lane == 0) st_cluster_u32(peer_abort, 1u);
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int issued[STAGES];
#pragma unroll
            for (int s = 0; s < STAGES; ++s) issued[s] = 0;
            bool ok = true;
            const bool cmpa = (args.compact & CMP_A) != 0;
            for (int u = cid; u < total && ok; u += ncl) {
                int g, gr, crow, m_blk, n_blk, rows_valid;
                decode(u, g, gr, crow, m_blk, n_blk, rows_valid);
                if (u + ncl >= total) pdl_launch_dependents();  // this pair's last tile
                const int base_row = m_blk * PM;
                const int rn = half_rows(rows_valid - base_row - (int)rank * 128);
                const int rn_peer = half_rows(rows_valid - base_row - (int)(rank ^ 1u) * 128);
                const int r0 = (cmpa ? crow : 0) + base_row + (int)rank * 128, gz = cmpa ? 0 : gr;
                for (int kb = 0; kb < kblocks; ++kb) {
                    if (!wait_phase(bar_empty(stage), phase ^ 1u, abort_flag, args.status)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = tiles_addr + stage * S::STAGE_BYTES;
                    const uint32_t sb = sa + S::A_BYTES;
                    const uint32_t fb = mapa_shared(bar_full(stage), 0);
                    if (leader)  // both CTAs' A rows and B halves
                        mbar_expect_tx(bar_full(stage), (uint32_t)(rn + rn_peer) * (BK * 2) + 2 * S::B_BYTES);
                    // A rows [0, rn) of this CTA's half; rows past rn keep stale data,
                    // which only reaches output rows past the load -- never stored
                    if (rn == 128) {
                        tma_load_3d_pair(sa, &tmA, fb, kb * BK, r0, gz);
                    } else {
                        int off = 0;
                        if (rn & 64) {
                            tma_load_3d_pair(sa, &tmAt.a[0], fb, kb * BK, r0, gz);
                            off = 64;
                        }
                        if (rn & 32) {
                            tma_load_3d_pair(sa + off * (BK * 2), &tmAt.a[1], fb, kb * BK, r0 + off, gz);
                            off += 32;
                        }
                        if (rn & 16) tma_load_3d_pair(sa + off * (BK * 2), &tmAt.a[2], fb, kb * BK, r0 + off, gz);
                    }
                    if (B_MN)
                        tma_load_4d_pair(sb, &tmB, fb, 0, kb * BK, n_blk * (BN / 64) + (int)rank * (BNC / 64), gr);
                    else
                        tma_load_3d_pair(sb, &tmB, fb, kb * BK, n_blk * BN + (int)rank * BNC, gr);
                    issued[stage]++;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (*abort_flag && leader) {  // copies in flight (both CTAs') land before the pair exits
                const unsigned long long t0 = global_ns();
                for (int s = 0; s < STAGES; ++s)
                    if (issued[s] > 0)
                        while (!mbar_try_wait(bar_full(s), (uint32_t)((issued[s] - 1) & 1)) &&
                               global_ns() - t0 < 200000000ull) {
                        }
            }
        }
        __syncwarp();
        give_up();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer (leader)
        if (leader) {
            int stage = 0;
            uint32_t phase = 0;
            int it = 0;
            bool ok = true;
            for (int u = cid; u < total && ok; u += ncl, ++it) {
                const int acc = it & 1;
                if (!wait_phase(bar_tempty(acc), (uint32_t)((it >> 1) & 1) ^ 1u, abort_flag, args.status))
                    break;
                tc_fence_after();
                const uint32_t dtmem = tmem_base + (uint32_t)(acc * BN);
                for (int kb = 0; kb < kblocks; ++kb) {
                    if (!wait_phase(bar_full(stage), phase, abort_flag, args.status)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t sa = tiles_addr + stage * S::STAGE_BYTES;
                    const uint32_t sb = sa + S::A_BYTES;
                    if (lane == 0) {
#pragma unroll
                        for (int kk = 0; kk < BK / 16; ++kk)
                            mma_pair_bf16(dtmem, operand_desc(sa, kk, false), operand_desc(sb, kk, B_MN), IDESC,
                                          (kb | kk) != 0 ? 1u : 0u);
                        mma_pair_commit_both(bar_empty(stage));
                    }
                    __syncwarp();
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
                if (!ok) break;
                if (lane == 0) mma_pair_commit_both(bar_tfull(acc));
                __syncwarp();
            }
            if (lane == 0) {  // all MMAs of the pair complete before TMEM is freed
                mma_pair_commit_local(bar_drain);
                const unsigned long long t0 = global_ns();
                while (!mbar_try_wait(bar_drain, 0) && global_ns() - t0 < 1000000000ull) {
                }
            }
            __syncwarp();
        }
        give_up();
    } else {
        // ------------------------------------------------------------ epilogue (row-masked st.global)
        // As in grouped_gemm_kernel's row mode, for this CTA's 128 rows of the
        // pair tile: warps w and w+4 share TMEM lane quarter q = w & 3 and split
        // the BN columns in halves; each thread owns one row.
        const int ew = warp - 2;
        const int q = warp & 3;
        const int half = ew >> 2;
        constexpr int COLS = BN / 2;
        constexpr int NCH = COLS / 32;
        uint8_t *stg = epi_base + ew * EPI_WARP_BYTES;
        const bool tanh_form = args.gelu_tanh != 0;
        const int sub_r = lane >> 2, sub_c = lane & 3;
        struct T {
            int g, gr, crow, m_blk, n_blk, rows_valid;
        };
        auto dec = [&](int u) {
            T t;
            decode(u, t.g, t.gr, t.crow, t.m_blk, t.n_blk, t.rows_valid);
            return t;
        };
        uint4 hcur[4], hnxt[4];
        auto load_h = [&](const T &tl, int c, uint4 (&dst)[4]) {
            const int r0 = tl.m_blk * PM + (int)rank * 128 + q * 32;
            if (r0 + lane < tl.rows_valid) {
                const uint4 *src = reinterpret_cast<const uint4 *>(
                    args.aux + (long long)tl.gr * args.sAux + (long long)(r0 + lane) * args.ldd +
                    tl.n_blk * BN + half * COLS + c * 32);
#pragma unroll
                for (int i = 0; i < 4; ++i) dst[i] = __ldg(src + i);
            } else {
#pragma unroll
                for (int i = 0; i < 4; ++i) dst[i] = make_uint4(0, 0, 0, 0);
            }
        };
        auto store_rows = [&](__nv_bfloat16 *base, int nvalid) {
            __syncwarp();
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const int r = i * 8 + sub_r;
                if (r < nvalid)
                    *reinterpret_cast<uint4 *>(base + (long long)r * args.ldd + sub_c * 8) =
                        *reinterpret_cast<const uint4 *>(stg + r * 80 + sub_c * 16);
            }
            __syncwarp();
        };
        int it = 0;
        bool ok = true;
        T t = dec(cid < total ? cid : 0);
        if (EPI == EPI_DGELU && cid < total) load_h(t, 0, hcur);
        for (int u = cid; u < total && ok; u += ncl, ++it) {
            const bool have_next = u + ncl < total;
            const T tn = dec(have_next ? u + ncl : u);
            const int acc = it & 1;
            if (!wait_phase(bar_tfull(acc), (uint32_t)((it >> 1) & 1), abort_flag, args.status)) break;
            tc_fence_after();
            const int row0 = t.m_blk * PM + (int)rank * 128 + q * 32;  // this warp's first row in the group
            int nvalid = t.rows_valid - row0;
            nvalid = nvalid < 0 ? 0 : (nvalid > 32 ? 32 : nvalid);
            const bool cmpd = (args.compact & CMP_D) != 0;
            const long long gofs = (cmpd ? (long long)t.crow * args.ldd : (long long)t.gr * args.sD) +
                                   (long long)row0 * args.ldd + t.n_blk * BN + half * COLS;
            const long long gofs2 = cmpd ? gofs + (long long)t.rows_valid * args.ldd : gofs;
            const uint32_t trow = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN + half * COLS);
            for (int c = 0; c < NCH; ++c) {
                if (EPI == EPI_DGELU) {
                    if (c + 1 < NCH) load_h(t, c + 1, hnxt);
                    else if (have_next) load_h(tn, 0, hnxt);
                }
                if (nvalid > 0) {
                    float v[32];
                    uint32_t r[32];
                    tmem_ld32(trow + c * 32, r);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
                    if (EPI == EPI_DGELU) {
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            float hv[8];
                            bf16x8_to_f32(hcur[i], hv);
#pragma unroll
                            for (int e = 0; e < 8; ++e) v[i * 8 + e] *= gelu_deriv_fast(hv[e], tanh_form);
                        }
                    }
#pragma unroll
                    for (int i = 0; i < 4; ++i)
                        *reinterpret_cast<uint4 *>(stg + lane * 80 + i * 16) = f32_to_bf16x8(v + i * 8);
                    store_rows(args.D + gofs + c * 32, nvalid);
                    if (EPI == EPI_DGELU) {  // residual v - bf16(v): dH = hi + lo to ~16 bits
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            float lv[8];
#pragma unroll
                            for (int e = 0; e < 8; ++e) {
                                const float x = v[i * 8 + e];
                                lv[e] = x - __bfloat162float(__float2bfloat16_rn(x));
                            }
                            *reinterpret_cast<uint4 *>(stg + lane * 80 + i * 16) = f32_to_bf16x8(lv);
                        }
                        store_rows(args.D2 + gofs2 + c * 32, nvalid);
                    }
                    if (EPI == EPI_GELU) {
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            float gv[8];
#pragma unroll
                            for (int e = 0; e < 8; ++e) gv[e] = gelu_fast(v[i * 8 + e], tanh_form);
                            *reinterpret_cast<uint4 *>(stg + lane * 80 + i * 16) = f32_to_bf16x8(gv);
                        }
                        store_rows(args.D2 + gofs2 + c * 32, nvalid);
                    }
                }
                if (EPI == EPI_DGELU) {
#pragma unroll
                    for (int i = 0; i < 4; ++i) hcur[i] = hnxt[i];
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote(mapa_shared(bar_tempty(acc), 0));
            t = tn;
        }
        give_up();
    }

    tc_fence_before();
    cluster_sync_all();  // no MMA, copy or remote arrive of either CTA is still in flight
    tc_fence_after();
    if (warp == 0) tmem_dealloc_pair(tmem_base, S::TMEM_COLS);
}

// Clusters of two that fit on the device at once (cached per device); 0 if
// the query fails.
int pair_clusters(const void *kern, size_t smem);

template <bool KSPLIT, int NKB>
int launch_pair(const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &mblo, const CUtensorMap &md,
                const Args &a, long long units, cudaStream_t s, const char *name,
                const PairSchedule *sched = nullptr) {
    using S = PairShape<KSPLIT, NKB>;
    auto kern = wgrad_pair_kernel<KSPLIT, NKB>;
    static std::atomic<int> smem_limit[64];
    if (const int st = raise_smem_limit((const void *)kern, smem_limit, (int)S::SMEM_BYTES)) return st;
    if (units <= 0) return VMOE_OK;
    const int ncl = pair_clusters((const void *)kern, S::SMEM_BYTES);
    if (ncl <= 0) return VMOE_ERR_CUDA;
    long long clusters = units < ncl ? units : ncl;
    PairSchedule sc;
    sc.enabled = 0;
    if (sched && sched->enabled) {  // a share schedule names its own pairs
        sc = *sched;
        int used = 0;
        for (int c = 0; c < MAX_PAIRS; ++c)
            if (sc.count[c] > 0) used = c + 1;
        if (used > ncl) return VMOE_ERR_INVALID;
        clusters = used;
    }
    if (clusters <= 0) return VMOE_OK;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * clusters));
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = S::SMEM_BYTES;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 2 : 1;
    trace_before(s, name);
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, ma, mb, mblo, md, a, sc);
    trace_after(s);
    return e == cudaSuccess ? VMOE_OK : VMOE_ERR_CUDA;
}


template <int BN, bool B_MN, int EPI>
int launch_row_pair(const CUtensorMap &ma, const CUtensorMap &mb, const TailMaps &mat, const Args &a,
                    long long max_tiles, cudaStream_t s, const char *name) {
    using S = RowPairShape<BN, B_MN, EPI>;
    auto kern = row_pair_kernel<BN, B_MN, EPI>;
    static std::atomic<int> smem_limit[64];
    if (const int st = raise_smem_limit((const void *)kern, smem_limit, (int)S::SMEM_BYTES)) return st;
    if (max_tiles <= 0) return VMOE_OK;
    const int ncl = pair_clusters((const void *)kern, S::SMEM_BYTES);
    if (ncl <= 0) return VMOE_ERR_CUDA;
    const long long clusters = max_tiles < ncl ? max_tiles : ncl;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)(2 * clusters));
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = S::SMEM_BYTES;
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 2 : 1;
    trace_before(s, name);
    const cudaError_t e = cudaLaunchKernelEx(&cfg, kern, ma, mb, mat, a);
    trace_after(s);
    return e == cudaSuccess ? VMOE_OK : VMOE_ERR_CUDA;
}

// SM pairs the weight-gradient kernel for capacity C runs on at once (its
// dynamic shared-memory limit raised first); 0 if the query fails.
template <bool KSPLIT>
int pair_wgrad_capacity(int C) {
    if (C <= 2 * BK) {
        using S = PairShape<KSPLIT, 2>;
        static std::atomic<int> lim[64];
        if (raise_smem_limit((const void *)wgrad_pair_kernel<KSPLIT, 2>, lim, (int)S::SMEM_BYTES)) return 0;
        return pair_clusters((const void *)wgrad_pair_kernel<KSPLIT, 2>, S::SMEM_BYTES);
    }
    using S = PairShape<KSPLIT, 4>;
    static std::atomic<int> lim[64];
    if (raise_smem_limit((const void *)wgrad_pair_kernel<KSPLIT, 4>, lim, (int)S::SMEM_BYTES)) return 0;
    return pair_clusters((const void *)wgrad_pair_kernel<KSPLIT, 4>, S::SMEM_BYTES);
}

// Row-mode GEMM: D[g][C rows][N] = act[g][C][K] * B, B MN-major ([K][N]) or
// K-major ([N][K]).
// sD / sAux / sAct: group strides (elements) of D and D2, of aux, and of act;
// 0 means the dense [G, C, width] layout.
// Groups of more than 128 rows (C > 128) can run on SM pairs (row_pair_kernel,
// 256-row tiles) with VMOE_ROW_PAIR=1 in the environment.  It is off by default:
// measured on GB300 it is no faster than the one-SM kernel (ViT-B, 6 tasks,
// C 247: FC1 + GELU 0.324 against 0.305 ms, dA 0.381 / 0.377, FC2 0.210 / 0.210;
// ViT-S, 4 tasks, C 493: 0.293 against 0.286 ms a step).  Its lower bytes per SM
// do not pay there, as those GEMMs are held back by their output stores and by
// read latency rather than by the operand bytes each SM loads.
template <int EPI, bool B_MN>
int row_gemm(const Dims &p, const __nv_bfloat16 *act, int K, const __nv_bfloat16 *w, int N,
             const int32_t *load, __nv_bfloat16 *D, __nv_bfloat16 *D2, const __nv_bfloat16 *aux,
             cudaStream_t s, const char *name, long long sD = 0, long long sAux = 0,
             long long sAct = 0, const Slice &sl = Slice()) {
    const int G = p.G(), C = p.C;
    // 256-column tiles, or 128 when N needs it -- and, for a plain-store GEMM,
    // when 256-column tiles would give the SMs fewer than two waves (the slices
    // of the memory-budgeted backward: dX over ~70 groups is 204 wide tiles on
    // 152 SMs); the tile width does not change any output element's sums
    const int entries = sl.n > 0 ? sl.n : G;
    const long long wide_tiles = (long long)entries * ((C + BM - 1) / BM) * (N / 256);
    const bool wide = N % 256 == 0 && !(EPI == EPI_STORE && wide_tiles < 2LL * num_sms());
    const int BN = wide ? 256 : 128;
    const bool pair = row_pair_enabled() && C > BM;
    const int bcols = pair ? BN / 2 : BN;  // B columns one CTA loads
    CUtensorMap ma, mb;
    TailMaps mat;
    const bool cmpa = (sl.compact & CMP_A) != 0;
    auto amap = [&](CUtensorMap *m, uint32_t box) {
        return cmpa ? make_map(m, act, K, (uint64_t)sl.rows, 1, box)
                    : make_map(m, act, K, C, G, box, (uint64_t)sAct);
    };
    if (!amap(&ma, 128) || !amap(&mat.a[0], 64) || !amap(&mat.a[1], 32) || !amap(&mat.a[2], 16))
        return VMOE_ERR_CUDA;
    bool okb = B_MN ? make_map_chunked(&mb, w, N, K, G, 64, bcols / 64) : make_map(&mb, w, K, N, G, bcols);
    if (!okb) return VMOE_ERR_CUDA;
    Args a = base_args(p, load);
    a.N = N;
    a.K_fixed = K;
    a.tiles_n = N / BN;
    a.tiles_m = pair ? (C + 255) / 256 : (C + BM - 1) / BM;
    a.D = D;
    a.D2 = D2;
    a.aux = aux;
    a.sD = sD ? sD : (long long)C * N;
    a.sAux = sAux ? sAux : (long long)C * N;
    a.ldd = N;
    if (sl.n > 0) {
        a.G = sl.n;
        a.glist = sl.glist;
        a.crow = sl.crow;
        a.compact = sl.compact;
    }
    long long max_tiles = (long long)a.G * a.tiles_m * a.tiles_n;
    if (pair)
        return wide ? launch_row_pair<256, B_MN, EPI>(ma, mb, mat, a, max_tiles, s, name)
                    : launch_row_pair<128, B_MN, EPI>(ma, mb, mat, a, max_tiles, s, name);
    const CUtensorMap md = {}, md2 = {};  // row mode stores with st.global: no output maps
    return wide ? launch<256, MODE_ROW, false, B_MN, EPI>(ma, mb, md, md2, mat, a, max_tiles, s, name)
                : launch<128, MODE_ROW, false, B_MN, EPI>(ma, mb, md, md2, mat, a, max_tiles, s, name);
}

// Weight-gradient GEMM: D[g][M][N] = act1[g][C][M]^T * act2[g][C][N], summed
// over each group's load[g] rows; both operands MN-major.
// ksplit: act2 is [G, 2C, N] -- a bf16 part in rows [0, C) and its residual in
// rows [C, 2C) -- and D = act1^T (hi + lo), summed over both halves.
// Kernel choice (measured on GB300, ms per launch, one-SM kernel -> pair):
//   M, N multiples of 256 and C <= 256: the SM-pair kernel above (resident B,
//     double buffered where two B tiles fit) -- dW1 at the 17-task ViT-B step
//     (C 124) 0.568 -> 0.539, at the 6-task one (C 247) 0.479 -> 0.387, at the
//     Zipf-skewed one (C 25) 0.787 -> 0.724; dW2 0.298 -> 0.262 (C 247) and
//     0.732 -> 0.722 (C 25) -- except dW2 with 32 < C <= 128, where the
//     streaming kernel stays faster (0.477 against 0.512 at C 124);
//   otherwise, 32 < C <= 128 with ksplit: the one-SM resident-B kernel;
//   otherwise the streaming grouped GEMM (both halves in its K loop).
// VMOE_PAIR=0 in the environment turns the pair kernel off.
inline int wgrad_gemm(const Dims &p, const __nv_bfloat16 *act1, int M, const __nv_bfloat16 *act2,
                      int N, const int32_t *load, __nv_bfloat16 *D, cudaStream_t s,
                      const char *name, bool ksplit = false, const Slice &sl = Slice(),
                      const PairSchedule *sched = nullptr) {
    const int G = p.G(), C = p.C;
    const bool wide = N % 256 == 0;
    const int BN = wide ? 256 : 128;
    const bool cmpb = (sl.compact & CMP_B) != 0;
    // B: per-group slabs of C (with ksplit 2C) rows, or the compact buffer
    const uint64_t b_rows = cmpb ? (uint64_t)sl.rows : (uint64_t)(ksplit ? 2 * C : C);
    const uint64_t b_outer = cmpb ? 1 : (uint64_t)G;
    CUtensorMap ma, mb, md;
    TailMaps mt;  // the last k-block's boxes of 16, 32 and 48 K rows
    // a_chunks / b_chunks: the 64-column chunks of one A / B box
    auto tail_maps = [&](int a_chunks, int b_chunks) {
        for (int i = 0; i < 3; ++i)
            if (!make_map_chunked(&mt.a[i], act1, M, C, G, 16 * (i + 1), a_chunks) ||
                !make_map_chunked(&mt.b[i], act2, N, b_rows, b_outer, 16 * (i + 1), b_chunks))
                return false;
        return true;
    };
    if (!make_map(&md, D, N, M, G, 32)) return VMOE_ERR_CUDA;  // 64 x 32 store boxes
    Args a = base_args(p, load);
    a.N = N;
    a.M_fixed = M;
    a.D = D;
    a.sD = (long long)M * N;
    a.ldd = N;
    a.ksplit = ksplit ? 1 : 0;
    if (sl.n > 0) {
        a.G = sl.n;
        a.glist = sl.glist;
        a.crow = sl.crow;
        a.compact = sl.compact;
    }
    const bool pair_pays = ksplit || C <= 32 || C > 2 * BK;
    if (pair_enabled() && pair_pays && M % 256 == 0 && N % 256 == 0 && C <= 4 * BK) {
        // Each CTA of a pair loads 128 columns (two chunks) of A and of B.  The
        // group-indexed maps have exactly C rows per group, and with ksplit the
        // residual gets a map of its own (base C rows in, group stride 2C rows),
        // so a k-block starting before row 0 reads zeros in both parts.
        CUtensorMap mblo = {};
        if (!make_map_chunked(&ma, act1, M, C, G, 64, 2)) return VMOE_ERR_CUDA;
        if (cmpb) {
            if (!make_map_chunked(&mb, act2, N, (uint64_t)sl.rows, 1, 64, 2)) return VMOE_ERR_CUDA;
        } else if (!make_map_chunked(&mb, act2, N, C, G, 64, 2, ksplit ? 2 * (uint64_t)C * N : 0) ||
                   (ksplit && !make_map_chunked(&mblo, act2 + (size_t)C * N, N, C, G, 64, 2,
                                                2 * (uint64_t)C * N))) {
            return VMOE_ERR_CUDA;
        }
        a.tiles_m = M / 256;
        a.tiles_n = N / 256;
        const long long units = (long long)a.G * a.tiles_n;
        if (C <= 2 * BK)
            return ksplit ? launch_pair<true, 2>(ma, mb, mblo, md, a, units, s, name, sched)
                          : launch_pair<false, 2>(ma, mb, mblo, md, a, units, s, name, sched);
        return ksplit ? launch_pair<true, 4>(ma, mb, mblo, md, a, units, s, name, sched)
                      : launch_pair<false, 4>(ma, mb, mblo, md, a, units, s, name, sched);
    }
    if (!make_map_chunked(&ma, act1, M, C, G, 64, BM / 64)) return VMOE_ERR_CUDA;
    if (!make_map_chunked(&mb, act2, N, b_rows, b_outer, 64, BN / 64)) return VMOE_ERR_CUDA;
    a.tiles_n = N / BN;
    a.tiles_m = M / BM;
    // Resident B when every group fits one B tile (C <= 128) but is not tiny: with
    // C <= 32 a unit has almost no MMA work to hide its B reload behind, and the
    // streaming kernel, which pipelines across tiles, is faster (measured at the
    // Zipf-skewed workload, C = 25: 0.770 against 0.904 ms; at C = 124 the
    // resident-B kernel wins, 0.566 against 0.749 ms).
    constexpr int BSTAT_MIN_C = 32;
    if (ksplit && N % BSTAT_BN == 0 && C <= 2 * BK && C > BSTAT_MIN_C) {
        using SB = BStatShape<BSTAT_BN, true, BSTAT_BUFS>;
        CUtensorMap mbs;
        if (!make_map_chunked(&mbs, act2, N, b_rows, b_outer, 64, BSTAT_BN / 64)) return VMOE_ERR_CUDA;
        if (!tail_maps(BM / 64, BSTAT_BN / 64)) return VMOE_ERR_CUDA;
        a.tiles_n = N / BSTAT_BN;
        const int nch = (a.tiles_m + SB::MCH - 1) / SB::MCH;
        const long long units = (long long)a.G * a.tiles_n * nch;
        return launch_bstat<BSTAT_BN, true, BSTAT_BUFS>(ma, mbs, md, mt, a, units, s, name);
    }
    long long max_tiles = (long long)a.G * a.tiles_m * a.tiles_n;
    const TailMaps unused{};  // the streaming kernel loads full k-blocks
    return wide ? launch<256, MODE_WGRAD, true, true, EPI_STORE>(ma, mb, md, md, unused, a, max_tiles, s, name)
                : launch<128, MODE_WGRAD, true, true, EPI_STORE>(ma, mb, md, md, unused, a, max_tiles, s, name);
}

}  // namespace tc
}  // namespace vmoe
