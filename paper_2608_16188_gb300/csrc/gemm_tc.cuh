// gemm_tc.cuh -- K3/K4/K6-K9: the bf16 grouped GEMM of the expert FFN on the
// sm_103a tensor cores (tcgen05 + TMEM + TMA), one persistent launch over all
// T*E (task, expert) groups of the merged expert pool.
//
// Structure (one CTA per SM, 320 threads):
//   warp 0      TMA producer: one thread streams 128x64 A tiles and 64xBN B
//               tiles into a STAGES-deep ring of shared-memory slots
//               (128-byte swizzle), signalling `full[s]` with the byte count.
//   warp 1      MMA issuer: one thread issues tcgen05.mma (M=128, N=BN,
//               K=16, bf16 in, fp32 accumulate in TMEM), commits each slot
//               back to `empty[s]` and each finished tile to `tmem_full[a]`.
//               The whole warp zeroes the K-tail rows of weight-gradient tiles.
//   warps 2-9   epilogue: tcgen05.ld of the accumulator (one TMEM lane per
//               thread = one output row; two warps per lane quarter split the
//               columns), the fused elementwise step (GELU, or GELU' of an H
//               prefetched into registers one chunk ahead), bf16 packing, a
//               per-warp staging tile in shared memory and coalesced 16-byte
//               row stores (weight gradients, whose tiles are always full:
//               TMA bulk tensor stores from 128-byte-swizzled staging).
//               The accumulator is double buffered in TMEM
//               (2 x BN columns), so tile i's epilogue overlaps tile i+1's
//               main loop.
// Tiles are distributed statically: CTA b takes tiles b, b + grid, ...  In
// row mode (H = Xe W1 etc.) a group contributes ceil(load/128) x N/BN tiles,
// counted from the device-resident loads by every CTA with a block scan, so
// empty groups cost nothing and no host round trip is needed.  In weight-
// gradient mode (dW1 = Xe^T dH etc.) every group contributes (M/128) x (N/BN)
// tiles whose K = load[g] rows; an empty group's tile is written as zeros.
//
// Every wait on an mbarrier is bounded in time; a wait that runs out sets the
// library's device status word to VMOE_ERR_DEVICE_TIMEOUT and an abort flag
// that the other roles see, and the CTA drains its copies and MMAs in flight
// and frees its TMEM before it returns.
#pragma once

#include <cuda.h>  // CUtensorMap and its enums (types only; the encoder is fetched at run time)

#include "common.cuh"

namespace vmoe {
namespace tc {

constexpr int BM = 128;  // rows of one MMA tile (TMEM lanes)
constexpr int BK = 64;   // K per pipeline slot = one 128-byte swizzle row of bf16
constexpr int THREADS = 320;  // warp 0 TMA, warp 1 MMA, warps 2-9 epilogue
constexpr int EPI_WARP_BYTES = 32 * 80;  // 32 rows x (64 data + 16 pad) bytes

// Row-mode epilogue of the one-SM grouped GEMM: the two-output epilogues
// (FC1 + GELU, dA + GELU') run 16 epilogue warps (4 per TMEM lane quarter),
// the plain store 8, all in 32-column chunks.  The two-output epilogues are
// issue-bound at 8 warps (about 31 instructions per output element); 16 warps
// leave room for 3 pipeline stages instead of 4, which the plain-store GEMMs,
// bound by their operand stream, cannot spare.  Measured on GB300 (ms; 8 -> 16
// warps): dA 0.536 -> 0.518 and FC1 0.485 -> 0.477 at the 17-task ViT-B step,
// 0.370 -> 0.321 and 0.301 -> 0.285 at the 6-task one; FC2 / dX 0.425 ->
// 0.433 / 0.434 -> 0.445 at 17 tasks, hence 8 there.  16-column chunks (4
// stages with 16 warps) gained nothing.
constexpr int EPI_WARP_BYTES_TMA = 2 * 4096;  // two 32 x 64 bf16 tiles, 128-byte swizzle
constexpr int MAX_G = 1024;
constexpr unsigned long long TIMEOUT_NS = 4000000000ull;

enum { MODE_ROW = 0, MODE_WGRAD = 1 };
enum { EPI_STORE = 0, EPI_GELU = 1, EPI_DGELU = 2 };

constexpr int ROW_CH = 32;
template <int MODE, int EPI>
struct Roles {
    static constexpr int EW = (MODE == 0 && EPI != EPI_STORE) ? 16 : 8;  // epilogue warps
    static constexpr int NT = 64 + 32 * EW;  // threads: producer, MMA, epilogue
    static constexpr int PITCH = 80;         // staging row pitch (bytes): 64 data + 16 pad
};

// Epilogue store path per mode.  TMA bulk tensor stores from 128-byte-
// swizzled staging need 64 KB of shared memory, which leaves room for 3
// pipeline slots at BN 256 instead of 4.  Measured on GB300 at the 17-task
// ViT-B step, they pay for the weight gradients (always-full tiles, write-
// bound) only; every row-mode GEMM -- FC1 + GELU and dA + GELU' with their two
// outputs included -- is faster with 4 slots and row-masked st.global (FC1:
// 0.485 ms against 0.492 ms with TMA stores).
template <int MODE, int EPI>
struct UseTmaStore {
    static constexpr bool value = MODE == 1;
};

template <int BN, int MODE, int EPI>
struct Shape {
    // Weight-gradient tiles have K = load <= 2 slots, so 3 slots suffice and
    // leave room for the double-buffered 128-byte-swizzled TMA-store staging.
    static constexpr bool TMA_EPI = UseTmaStore<MODE, EPI>::value;
    static constexpr int NT = Roles<MODE, EPI>::NT;
    static constexpr int EPI_BYTES =
        TMA_EPI ? 8 * EPI_WARP_BYTES_TMA : Roles<MODE, EPI>::EW * 32 * Roles<MODE, EPI>::PITCH;
    static constexpr uint32_t A_BYTES = BM * BK * 2;
    static constexpr uint32_t B_BYTES = BN * BK * 2;
    static constexpr uint32_t STAGE_BYTES = A_BYTES + B_BYTES;
    static constexpr size_t FIXED = 1024 + EPI_BYTES + 16 + NT * 4 + (MAX_G + 1) * 4 + 8 * 21;
    static constexpr int STAGES_FIT = (int)((232448 - FIXED) / STAGE_BYTES);
    static constexpr int STAGES_MAX = TMA_EPI ? (BN == 256 ? 3 : 4) : (BN == 256 ? 4 : 6);
    static constexpr int STAGES = STAGES_FIT < STAGES_MAX ? STAGES_FIT : STAGES_MAX;
    static constexpr uint32_t TMEM_COLS = 2 * BN;
    static constexpr int NUM_BARS = 2 * STAGES + 5;
    static constexpr size_t SMEM_BYTES = 1024 + (size_t)STAGES * STAGE_BYTES + EPI_BYTES +
                                         NUM_BARS * 8 + 16 + NT * 4 + (MAX_G + 1) * 4;
    static_assert(SMEM_BYTES <= 232448, "over the 227 KB shared-memory limit");
};

struct Args {
    int G, C;
    int N;        // output columns
    int K_fixed;  // row mode: reduction length
    int M_fixed;  // weight-gradient mode: output rows
    int tiles_n;  // N / BN
    int tiles_m;  // weight-gradient mode: M_fixed / BM; row mode: ceil(C / BM)
    const int32_t *load;
    __nv_bfloat16 *D;          // output (EPI_DGELU: the bf16 part of dH)
    __nv_bfloat16 *D2;         // EPI_GELU: A = GELU(H); EPI_DGELU: the bf16 residual of dH
    const __nv_bfloat16 *aux;  // EPI_DGELU: H
    long long sD;              // group stride of D / D2 (elements)
    long long sAux;            // group stride of aux (elements)
    int ldd;                   // row stride of D / D2 / aux (elements)
    int ksplit;                // weight-gradient mode: B holds [hi rows; lo rows] (K doubled)
    int gelu_tanh;
    int *status;
    // Slices (the memory-budgeted backward): the launch covers G entries, entry i
    // being group glist[i] of the real tensors (glist NULL: entry i = group i).
    // Operands flagged in `compact` live in a compact buffer instead, entry i's
    // rows starting at row crow[i] (with ksplit / a second output, the residual
    // rows follow the entry's load rows).
    const int32_t *glist;
    const int32_t *crow;
    int compact;               // CMP_* bits
};
enum { CMP_A = 1, CMP_B = 2, CMP_D = 4 };

// Partial-box tensor maps: a group's padding rows [load, C) are not read.
// Row mode: a[0..2] = the A operand with 64-, 32- and 16-row boxes; a tile
// whose valid rows end inside it loads rows [0, 16 ceil(rows / 16)) as at most
// three boxes instead of one 128-row box.
// Weight gradients, resident-B kernel: a[i], b[i] = the A and B operands with
// boxes of 16 (i + 1) K rows, for a group's last k-block when its valid rows
// end inside it.  Such a box lands chunk-major with a chunk stride of
// (rows x 128) bytes, which the k-block's MMA descriptors take as their
// leading byte offset.
struct TailMaps {
    CUtensorMap a[3], b[3];
};
// Rows loaded for a k-block with `rem` valid K rows (>= 1): all BK, or rem
// rounded up to 16.
__host__ __device__ __forceinline__ int tail_rows(int rem) { return rem >= 64 ? 64 : ((rem + 15) & ~15); }
__device__ __forceinline__ int real_group(const Args &a, int i) { return a.glist ? __ldg(a.glist + i) : i; }

// ---------------------------------------------------------------------------
// PTX wrappers.

__device__ __forceinline__ uint32_t smem_u32(const void *p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
                 : "memory");
}
__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}\n"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}
__device__ __forceinline__ unsigned long long global_ns() {
    unsigned long long t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}
// Bounded wait for the phase of parity `parity` of barrier `bar`.
static __device__ __noinline__ bool wait_phase(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                               int *status,
                                               unsigned long long limit_ns = TIMEOUT_NS) {
    if (mbar_try_wait(bar, parity)) return true;
    const unsigned long long t0 = global_ns();
    for (uint32_t i = 1;; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 63u) == 0) {
            if (*abort_flag) return false;
            if (global_ns() - t0 > limit_ns) {
                *abort_flag = 1;
                if (status) atomicExch(status, (int)VMOE_ERR_DEVICE_TIMEOUT);
                return false;
            }
        }
    }
}
__device__ __forceinline__ void fence_barrier_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void fence_proxy_async() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}
__device__ __forceinline__ void tma_load_3d(uint32_t dst, const CUtensorMap *map, uint32_t bar,
                                            int c0, int c1, int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2)
        : "memory");
}
__device__ __forceinline__ void tma_store_3d(const CUtensorMap *map, uint32_t src, int c0, int c1,
                                             int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.global.shared::cta.bulk_group [%0, {%2, %3, %4}], [%1];" ::"l"(
            reinterpret_cast<uint64_t>(map)),
        "r"(src), "r"(c0), "r"(c1), "r"(c2)
        : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read1() {
    asm volatile("cp.async.bulk.wait_group.read 1;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_read0() {
    asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory");
}
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }
__device__ __forceinline__ void tma_load_4d(uint32_t dst, const CUtensorMap *map, uint32_t bar,
                                            int c0, int c1, int c2, int c3) {
    asm volatile(
        "cp.async.bulk.tensor.4d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%3, %4, %5, %6}], [%2];" ::"r"(dst),
        "l"(reinterpret_cast<uint64_t>(map)), "r"(bar), "r"(c0), "r"(c1), "r"(c2), "r"(c3)
        : "memory");
}
// Named barrier over `count` threads (ids 1..15; 0 is __syncthreads).
__device__ __forceinline__ void named_bar(int id, int count) {
    asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(count) : "memory");
}
__device__ __forceinline__ void prefetch_map(const CUtensorMap *map) {
    asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(map)) : "memory");
}
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tc_fence_before() {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void tc_fence_after() {
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void mma_bf16(uint32_t tmem_d, uint64_t adesc, uint64_t bdesc,
                                         uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(tmem_d),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
__device__ __forceinline__ void mma_commit(uint32_t bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                     bar)
                 : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
        "%12, %13, %14, %15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, "
        "%30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]),
          "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]),
          "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, "
        "%12, %13, %14, %15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]),
          "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
}
__device__ __forceinline__ void tmem_ld_wait() {
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// Shared-memory matrix descriptor, 128-byte swizzle (tcgen05 format: start
// address, leading and stride byte offsets in 16-byte units, version 1 at bit
// 46, layout SWIZZLE_128B = 2 at bits 61-63).
__device__ __forceinline__ uint64_t sdesc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo) {
    uint64_t d = (uint64_t)((saddr & 0x3FFFFu) >> 4);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}
// Operand tiles in shared memory:
//  K-major (K contiguous):  rows of 64 K-elements = 128 bytes, 8-row swizzle
//    atoms of 1024 bytes stacked along M/N (SBO = 1024).  Step k16 -> +32 bytes.
//  MN-major (M/N contiguous): chunks of 64 MN-elements x 64 K-rows (8 KiB),
//    one TMA box each, stacked along M/N (LBO = 8192, the MN chunk stride);
//    8-row K groups are 1024 bytes apart (SBO).  Step k16 -> +2048 bytes.
__device__ __forceinline__ uint64_t operand_desc(uint32_t tile, int kk, bool mn_major) {
    return mn_major ? sdesc_sw128(tile + kk * 2048, 8192, 1024)
                    : sdesc_sw128(tile + kk * 32, 16, 1024);
}
// MN-major k-block of `rows` K rows: its MN chunks are rows x 128 bytes apart.
__device__ __forceinline__ uint64_t operand_desc_mn(uint32_t tile, int kk, int rows) {
    return sdesc_sw128(tile + kk * 2048, (uint32_t)rows * 128u, 1024);
}

// Instruction descriptor of tcgen05.mma kind::f16: D fp32 (bits 4-5 = 1),
// A and B bf16 (bits 7-9, 10-12 = 1), A / B MN-major (bits 15 / 16),
// N >> 3 at bits 17-22, M >> 4 at bits 24-28.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool a_mn, bool b_mn) {
    return (1u << 4) | (1u << 7) | (1u << 10) | ((a_mn ? 1u : 0u) << 15) |
           ((b_mn ? 1u : 0u) << 16) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

struct Tile {
    int g, m_blk, n_blk, kblocks, kvalid, rows_valid;
    int khalf;  // weight-gradient mode: k-blocks per half (kblocks = 2 * khalf with ksplit)
    int gr;     // the real group of entry g
    int crow;   // entry g's first row in the compact buffer
};

template <int MODE>
__device__ __forceinline__ Tile decode_tile(const Args &a, const int *prefix, int u) {
    Tile t;
    if (MODE == MODE_ROW) {
        int lo = 0, hi = a.G;  // prefix[lo] <= u < prefix[hi]
        while (hi - lo > 1) {
            int mid = (lo + hi) >> 1;
            if (prefix[mid] <= u) lo = mid; else hi = mid;
        }
        t.g = lo;
        t.gr = real_group(a, lo);
        t.crow = a.crow ? __ldg(a.crow + lo) : 0;
        int local = u - prefix[lo];
        t.m_blk = local / a.tiles_n;
        t.n_blk = local - t.m_blk * a.tiles_n;
        t.kblocks = a.K_fixed / BK;
        t.kvalid = a.K_fixed;
        int L = __ldg(a.load + t.gr);
        t.rows_valid = L < 0 ? 0 : (L > a.C ? a.C : L);
    } else {
        int tpg = a.tiles_m * a.tiles_n;
        t.g = u / tpg;
        t.gr = real_group(a, t.g);
        t.crow = a.crow ? __ldg(a.crow + t.g) : 0;
        int local = u - t.g * tpg;
        t.m_blk = local / a.tiles_n;
        t.n_blk = local - t.m_blk * a.tiles_n;
        int L = __ldg(a.load + t.gr);
        L = L < 0 ? 0 : (L > a.C ? a.C : L);
        t.kvalid = L;
        t.khalf = (L + BK - 1) / BK;
        t.kblocks = a.ksplit ? 2 * t.khalf : t.khalf;
        t.rows_valid = a.M_fixed;
    }
    return t;
}

template <int BN, int MODE, bool A_MN, bool B_MN, int EPI>
__global__ void __launch_bounds__(Roles<MODE, EPI>::NT, 1)
grouped_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmD, const __grid_constant__ CUtensorMap tmD2,
                    const __grid_constant__ TailMaps tmAt, Args args) {
    using S = Shape<BN, MODE, EPI>;
    constexpr int STAGES = S::STAGES;
    constexpr int NT = S::NT;
    constexpr uint32_t IDESC = idesc_bf16(BM, BN, A_MN, B_MN);

    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
    const uint32_t tiles_addr = smem_u32(smem);
    uint8_t *epi_base = smem + STAGES * S::STAGE_BYTES;
    uint64_t *bars = reinterpret_cast<uint64_t *>(epi_base + S::EPI_BYTES);
    int *misc = reinterpret_cast<int *>(bars + S::NUM_BARS);  // [0] tmem base, [1] abort, [2] total
    int *scan_tmp = misc + 4;
    int *prefix = scan_tmp + NT;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar_full = [&](int s) { return smem_u32(bars + s); };
    auto bar_empty = [&](int s) { return smem_u32(bars + STAGES + s); };
    auto bar_tfull = [&](int a) { return smem_u32(bars + 2 * STAGES + a); };
    auto bar_tempty = [&](int a) { return smem_u32(bars + 2 * STAGES + 2 + a); };
    const uint32_t bar_drain = smem_u32(bars + 2 * STAGES + 4);
    volatile int *abort_flag = misc + 1;

    if (tid == 0) {
        for (int s = 0; s < STAGES; ++s) {
            mbar_init(bar_full(s), 1);
            mbar_init(bar_empty(s), 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(bar_tfull(a), 1);
            mbar_init(bar_tempty(a), Roles<MODE, EPI>::EW);
        }
        mbar_init(bar_drain, 1);
        misc[1] = 0;
        fence_barrier_init();
        fence_proxy_async();
        prefetch_map(&tmA);
        prefetch_map(&tmB);
        if (MODE == MODE_ROW)
            for (int i = 0; i < 3; ++i) prefetch_map(&tmAt.a[i]);
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(misc), S::TMEM_COLS);
        tmem_relinquish();
    }
    pdl_wait();  // the predecessor's outputs (loads, operands) are complete from here on

    // Tile count (and, in row mode, the per-group tile prefix).
    int total;
    if (MODE == MODE_ROW) {
        const int G = args.G;
        const int per = (G + NT - 1) / NT;
        const int g0 = min(G, tid * per), g1 = min(G, g0 + per);
        int local = 0;
        for (int g = g0; g < g1; ++g) {
            int L = __ldg(args.load + real_group(args, g));
            L = L < 0 ? 0 : (L > args.C ? args.C : L);
            local += ((L + BM - 1) / BM) * args.tiles_n;
        }
        scan_tmp[tid] = local;
        __syncthreads();
        if (warp == 0) {  // exclusive scan of NT partials, NT/32 per lane
            constexpr int PER = NT / 32;
            int v[PER], s = 0;
#pragma unroll
            for (int i = 0; i < PER; ++i) {
                v[i] = scan_tmp[lane * PER + i];
                s += v[i];
            }
            int incl = s;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                int y = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += y;
            }
            int run = incl - s;
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
            run += ((L + BM - 1) / BM) * args.tiles_n;
        }
        if (tid == 0) prefix[G] = misc[2];
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    total = (MODE == MODE_ROW) ? misc[2] : args.G * args.tiles_m * args.tiles_n;
    const uint32_t tmem_base = (uint32_t)misc[0];

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            int issued[STAGES];
#pragma unroll
            for (int s = 0; s < STAGES; ++s) issued[s] = 0;
            bool ok = true;
            for (int u = blockIdx.x; u < total && ok; u += gridDim.x) {
                const Tile t = decode_tile<MODE>(args, prefix, u);
                if (u + (int)gridDim.x >= total) pdl_launch_dependents();  // this CTA's last tile
                for (int kb = 0; kb < t.kblocks; ++kb) {
                    if (!wait_phase(bar_empty(stage), phase ^ 1u, abort_flag, args.status)) {
                        ok = false;
                        break;
                    }
                    const uint32_t sa = tiles_addr + stage * S::STAGE_BYTES;
                    const uint32_t sb = sa + S::A_BYTES;
                    const uint32_t fb = bar_full(stage);
                    if (MODE == MODE_ROW) {
                        // A rows [0, rn): the tile's valid rows rounded up to 16.  The
                        // slot's rows past rn keep stale data, which only reaches
                        // output rows past rows_valid -- never stored.
                        const int rem_rows = t.rows_valid - t.m_blk * BM;
                        const int rn = rem_rows >= BM ? BM : ((rem_rows + 15) & ~15);
                        const bool cmpa = (args.compact & CMP_A) != 0;
                        const int r0 = (cmpa ? t.crow : 0) + t.m_blk * BM, gz = cmpa ? 0 : t.gr;
                        mbar_expect_tx(fb, (uint32_t)rn * (BK * 2) + S::B_BYTES);
                        if (rn == BM) {
                            tma_load_3d(sa, &tmA, fb, kb * BK, r0, gz);
                        } else {
                            int off = 0;
                            if (rn & 64) {
                                tma_load_3d(sa, &tmAt.a[0], fb, kb * BK, r0, gz);
                                off = 64;
                            }
                            if (rn & 32) {
                                tma_load_3d(sa + off * (BK * 2), &tmAt.a[1], fb, kb * BK, r0 + off, gz);
                                off += 32;
                            }
                            if (rn & 16) tma_load_3d(sa + off * (BK * 2), &tmAt.a[2], fb, kb * BK, r0 + off, gz);
                        }
                        if (B_MN) {  // one 4-D box: BN/64 column chunks of 64 rows
                            tma_load_4d(sb, &tmB, fb, 0, kb * BK, t.n_blk * (BN / 64), t.gr);
                        } else {
                            tma_load_3d(sb, &tmB, fb, kb * BK, t.n_blk * BN, t.gr);
                        }
                    } else {
                        // Weight gradients: K = the group's rows.  With ksplit the second
                        // half of the k-blocks pairs the same A rows with B's residual
                        // rows, which start at row C of the group.
                        // (Tail-sized boxes for the last k-block, as in the resident-B
                        // kernel, made this streaming kernel slower: full boxes here.)
                        mbar_expect_tx(fb, S::STAGE_BYTES);
                        const int hi = (kb >= t.khalf) ? 1 : 0;
                        const int ka = (kb - hi * t.khalf) * BK;
                        const int kbr = hi * args.C + ka;
                        tma_load_4d(sa, &tmA, fb, 0, ka, t.m_blk * (BM / 64), t.gr);
                        if (args.compact & CMP_B)  // residual rows follow the entry's load rows
                            tma_load_4d(sb, &tmB, fb, 0, t.crow + hi * t.kvalid + ka,
                                        t.n_blk * (BN / 64), 0);
                        else
                            tma_load_4d(sb, &tmB, fb, 0, kbr, t.n_blk * (BN / 64), t.gr);
                    }
                    issued[stage]++;
                    if (++stage == STAGES) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (*abort_flag) {  // let copies in flight land before the CTA exits
                int dummy = 0;
                for (int s = 0; s < STAGES; ++s)
                    if (issued[s] > 0) {
                        const unsigned long long t0 = global_ns();
                        while (!mbar_try_wait(bar_full(s), (uint32_t)((issued[s] - 1) & 1)) &&
                               global_ns() - t0 < 100000000ull)
                            ++dummy;
                    }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        int stage = 0;
        uint32_t phase = 0;
        int it = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < total && ok; u += gridDim.x, ++it) {
            const Tile t = decode_tile<MODE>(args, prefix, u);
            const int acc = it & 1;
            const uint32_t aph = (uint32_t)((it >> 1) & 1);
            if (!wait_phase(bar_tempty(acc), aph ^ 1u, abort_flag, args.status)) break;
            tc_fence_after();
            const uint32_t dtmem = tmem_base + (uint32_t)(acc * BN);
            if (t.kblocks == 0) {
                if (lane == 0) mbar_arrive(bar_tfull(acc));
                __syncwarp();
                continue;
            }
            for (int kb = 0; kb < t.kblocks; ++kb) {
                if (!wait_phase(bar_full(stage), phase, abort_flag, args.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t sa = tiles_addr + stage * S::STAGE_BYTES;
                const uint32_t sb = sa + S::A_BYTES;
                int nk = BK / 16;
                if (MODE == MODE_WGRAD && (kb == t.kblocks - 1 || kb == t.khalf - 1)) {
                    // K tail: the MMA reads rows [0, 16*nk) of the slot; rows
                    // [rem, 16*nk) lie past this group's load and are zeroed in
                    // both operands (one 128-byte line per K row per 64-wide chunk).
                    const int rem = t.kvalid - (kb - (kb >= t.khalf ? t.khalf : 0)) * BK;
                    nk = (rem + 15) >> 4;
                    const int z0 = rem, z1 = nk * 16;
                    if (z0 < z1) {
                        const int rows = z1 - z0;
                        constexpr int CH = BM / 64 + BN / 64;
                        const int units = CH * rows * 8;
                        uint8_t *slot_ptr = smem + stage * S::STAGE_BYTES;
                        for (int i = lane; i < units; i += 32) {
                            int c = i / (rows * 8);
                            int w = i - c * rows * 8;
                            int r = z0 + (w >> 3);
                            int q = w & 7;
                            uint8_t *base = (c < BM / 64) ? slot_ptr + c * 8192
                                                          : slot_ptr + S::A_BYTES + (c - BM / 64) * 8192;
                            *reinterpret_cast<uint4 *>(base + r * 128 + q * 16) = make_uint4(0, 0, 0, 0);
                        }
                        fence_proxy_async();
                    }
                    __syncwarp();
                }
                if (lane == 0) {
                    for (int kk = 0; kk < nk; ++kk)
                        mma_bf16(dtmem, operand_desc(sa, kk, A_MN), operand_desc(sb, kk, B_MN), IDESC,
                                 (kb | kk) != 0 ? 1u : 0u);
                    mma_commit(bar_empty(stage));
                }
                __syncwarp();
                if (++stage == STAGES) {
                    stage = 0;
                    phase ^= 1u;
                }
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
    } else if (MODE == MODE_WGRAD) {
        // ------------------------------------------------------------ epilogue (weight gradients)
        // Every tile is full.  Each warp reads all BN/2 accumulator columns of its
        // 32 rows with back-to-back tcgen05.ld before one wait, then writes 64-
        // column chunks into a 128-byte-swizzled 32 x 64 staging tile that one
        // lane stores with a TMA bulk tensor store (two tiles alternate).
        const int ew = warp - 2;
        const int q = warp & 3;
        const int half = ew >> 2;
        constexpr int COLS = BN / 2;
        uint8_t *stg = epi_base + ew * EPI_WARP_BYTES_TMA;
        int nstore = 0;
        int it = 0;
        for (int u = blockIdx.x; u < total; u += gridDim.x, ++it) {
            const Tile t = decode_tile<MODE>(args, prefix, u);
            const int acc = it & 1;
            const uint32_t aph = (uint32_t)((it >> 1) & 1);
            if (!wait_phase(bar_tfull(acc), aph, abort_flag, args.status)) break;
            tc_fence_after();
            const int row0 = t.m_blk * BM + q * 32;
            const int colw = t.n_blk * BN + half * COLS;
            const uint32_t trow = tmem_base + ((uint32_t)(q * 32) << 16) +
                                  (uint32_t)(acc * BN + half * COLS);
            uint32_t r[COLS / 32][32];
            if (t.kblocks > 0) {
#pragma unroll
                for (int i = 0; i < COLS / 32; ++i) tmem_ld32(trow + i * 32, r[i]);
                tmem_ld_wait();
            } else {
#pragma unroll
                for (int i = 0; i < COLS / 32; ++i)
#pragma unroll
                    for (int j = 0; j < 32; ++j) r[i][j] = 0u;
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_tempty(acc));  // the accumulator is in registers now
#pragma unroll
            for (int c = 0; c < COLS / 64; ++c) {
                uint8_t *buf = stg + (nstore & 1) * 4096;
                if (lane == 0 && nstore >= 2) bulk_wait_read1();  // the store that used buf has read it
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
                    tma_store_3d(&tmD, smem_u32(buf), colw + c * 64, row0, t.gr);
                    bulk_commit();
                }
                ++nstore;
            }
        }
        if (lane == 0) bulk_wait_all();
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue (row mode, st.global)
        // Warps 2 .. EW+1.  Warp w works on TMEM lane quarter q = w & 3 (rows
        // 32q .. 32q+31 of the tile), each thread owning one row; the EW / 4
        // warps of a quarter take the tile's CH-column chunks in turn (warp j:
        // chunks j, j + EW/4, ...).  Per chunk: tcgen05.ld, the fused
        // elementwise step, bf16 packing into a per-warp staging tile, and
        // coalesced, row-masked 16-byte stores.
        constexpr int EW = Roles<MODE, EPI>::EW;
        constexpr int WPQ = EW / 4;                 // warps per lane quarter
        constexpr int CH = ROW_CH;                  // columns per chunk
        constexpr int NCH = BN / CH;                // chunks per tile row
        constexpr int PITCH = Roles<MODE, EPI>::PITCH;   // staging row pitch (bytes)
        constexpr int PIECES = CH * 2 / 16;         // 16-byte pieces of a staged row
        constexpr int RPI = 32 / PIECES;            // rows per store instruction
        const int ew = warp - 2;
        const int q = warp & 3;
        const int jw = ew >> 2;
        uint8_t *stg = epi_base + ew * 32 * PITCH;
        const bool tanh_form = args.gelu_tanh != 0;
        const int sub_r = lane / PIECES, sub_c = lane % PIECES;  // row-store mapping
        // EPI_DGELU: the H values of this thread's row for the current chunk,
        // loaded one chunk ahead (and across tiles) so the epilogue never waits
        // on a fresh global load.
        uint4 hcur[CH / 8], hnxt[CH / 8];
        auto load_h = [&](const Tile &tl, int c, uint4 (&dst)[CH / 8]) {
            const int r0 = tl.m_blk * BM + q * 32;
            if (r0 + lane < tl.rows_valid) {
                const uint4 *src = reinterpret_cast<const uint4 *>(
                    args.aux + (long long)tl.gr * args.sAux + (long long)(r0 + lane) * args.ldd +
                    tl.n_blk * BN + c * CH);
#pragma unroll
                for (int i = 0; i < CH / 8; ++i) dst[i] = __ldg(src + i);
            } else {
#pragma unroll
                for (int i = 0; i < CH / 8; ++i) dst[i] = make_uint4(0, 0, 0, 0);
            }
        };
        // Stage 32 packed rows of this warp and store them coalesced, masked to
        // the valid rows.
        auto store_rows = [&](__nv_bfloat16 *base, int nvalid) {
            __syncwarp();
#pragma unroll
            for (int i = 0; i < PIECES; ++i) {
                const int r = i * RPI + sub_r;
                if (r < nvalid)
                    *reinterpret_cast<uint4 *>(base + (long long)r * args.ldd + sub_c * 8) =
                        *reinterpret_cast<const uint4 *>(stg + r * PITCH + sub_c * 16);
            }
            __syncwarp();
        };
        auto stage = [&](const float *v) {
#pragma unroll
            for (int i = 0; i < CH / 8; ++i)
                *reinterpret_cast<uint4 *>(stg + lane * PITCH + i * 16) = f32_to_bf16x8(v + i * 8);
        };
        int it = 0;
        Tile t = decode_tile<MODE>(args, prefix, blockIdx.x < total ? blockIdx.x : 0);
        if (EPI == EPI_DGELU && blockIdx.x < total) load_h(t, jw, hcur);
        for (int u = blockIdx.x; u < total; u += gridDim.x, ++it) {
            const bool have_next = u + (int)gridDim.x < total;
            const Tile tn = decode_tile<MODE>(args, prefix, have_next ? u + gridDim.x : u);
            const int acc = it & 1;
            const uint32_t aph = (uint32_t)((it >> 1) & 1);
            if (!wait_phase(bar_tfull(acc), aph, abort_flag, args.status)) break;
            tc_fence_after();
            const int row0 = t.m_blk * BM + q * 32;  // this warp's first row in the group
            int nvalid = t.rows_valid - row0;
            nvalid = nvalid < 0 ? 0 : (nvalid > 32 ? 32 : nvalid);
            // compact output: the entry's rows from crow, its second output (the
            // residual) after its load rows; else the group's slab
            const bool cmpd = (args.compact & CMP_D) != 0;
            const long long gofs = (cmpd ? (long long)t.crow * args.ldd : (long long)t.gr * args.sD) +
                                   (long long)row0 * args.ldd + t.n_blk * BN;
            const long long gofs2 = cmpd ? gofs + (long long)t.rows_valid * args.ldd : gofs;
            const uint32_t trow = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * BN);
#pragma unroll 1
            for (int c = jw; c < NCH; c += WPQ) {
                if (EPI == EPI_DGELU) {
                    if (c + WPQ < NCH) load_h(t, c + WPQ, hnxt);
                    else if (have_next) load_h(tn, jw, hnxt);
                }
                if (nvalid > 0) {
                    float v[CH];
                    if (t.kblocks > 0) {
                        uint32_t r[CH];
                        if (CH == 32) tmem_ld32(trow + c * CH, *reinterpret_cast<uint32_t(*)[32]>(r));
                        else tmem_ld16(trow + c * CH, *reinterpret_cast<uint32_t(*)[16]>(r));
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < CH; ++i) v[i] = __uint_as_float(r[i]);
                    } else {
#pragma unroll
                        for (int i = 0; i < CH; ++i) v[i] = 0.0f;
                    }
                    if (EPI == EPI_DGELU) {
#pragma unroll
                        for (int i = 0; i < CH / 8; ++i) {
                            float hv[8];
                            bf16x8_to_f32(hcur[i], hv);
#pragma unroll
                            for (int e = 0; e < 8; ++e) v[i * 8 + e] *= gelu_deriv_fast(hv[e], tanh_form);
                        }
                    }
                    stage(v);
                    store_rows(args.D + gofs + c * CH, nvalid);
                    if (EPI == EPI_DGELU) {  // residual v - bf16(v): dH = hi + lo to ~16 bits
                        float lv[CH];
#pragma unroll
                        for (int i = 0; i < CH; ++i) lv[i] = v[i] - __bfloat162float(__float2bfloat16_rn(v[i]));
                        stage(lv);
                        store_rows(args.D2 + gofs2 + c * CH, nvalid);
                    }
                    if (EPI == EPI_GELU) {
                        float gv[CH];
#pragma unroll
                        for (int i = 0; i < CH; ++i) gv[i] = gelu_fast(v[i], tanh_form);
                        stage(gv);
                        store_rows(args.D2 + gofs2 + c * CH, nvalid);
                    }
                }
                if (EPI == EPI_DGELU) {
#pragma unroll
                    for (int i = 0; i < CH / 8; ++i) hcur[i] = hnxt[i];
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(bar_tempty(acc));
            t = tn;
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem_base, S::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Weight gradients with the B operand resident ("B-stationary"), for groups of
// at most 128 rows (C <= 128).
//
//   D[g][m-tile][n-tile] = A[g][K rows][m-tile]^T  B[g][K rows][n-tile]
//
// One work unit = (group g, column tile n, a run of up to MCH row tiles m).
// The unit's B tile -- all K rows, and with KSPLIT the residual rows after
// them -- is loaded once into a resident region and reused by every row tile
// of the run, whose A tiles stream through a two-deep ring.  Against the
// streaming kernel this cuts the L2 -> SM traffic of a 128 x 256 output tile
// from (A + B) per tile to A per tile plus B / MCH.  With B_BUFS = 2 the next
// unit's B tile loads while this unit's row tiles run (BN = 128 keeps two
// resident tiles within shared memory).  Roles, TMEM double buffering, bounded
// waits and the TMA-store epilogue are as in grouped_gemm_kernel.
// Column tile and B buffering of the resident-B weight-gradient kernel: 256
// columns with one resident B tile (default), or 128 columns with two.
// Measured at the 17-task step: 0.580 ms against 0.800 ms -- twice the A
// (L2 -> SM) traffic per output byte costs more than the hidden B loads save.
#ifndef VMOE_BSTAT_BN
#define VMOE_BSTAT_BN 256
#endif
constexpr int BSTAT_BN = VMOE_BSTAT_BN;
constexpr int BSTAT_BUFS = BSTAT_BN == 128 ? 2 : 1;

template <int BN, bool KSPLIT, int B_BUFS>
struct BStatShape {
    static constexpr int MCH = 6;                              // row tiles per unit
    static constexpr uint32_t A_KB = BM * BK * 2;              // one A k-block (16 KB)
    static constexpr uint32_t B_KB = BN * BK * 2;              // one B k-block
    static constexpr uint32_t A_BUF = 2 * A_KB;                // up to 128 K rows
    static constexpr uint32_t B_BYTES = (KSPLIT ? 4 : 2) * B_KB;
    // A ring depth 2 (measured: a single A buffer, which would leave room for
    // double-buffered staging with the split, made dW1 26% slower).
    static constexpr int A_BUFS = 2;
    static constexpr int STG_BUFS = KSPLIT ? 1 : 2;            // 32 x 64 staging tiles per warp
    static constexpr uint32_t EPI_BYTES = 8 * STG_BUFS * 4096;
    static constexpr uint32_t TMEM_COLS = 2 * BN;
    static constexpr int NUM_BARS = 9 + 2 * B_BUFS;
    static constexpr size_t SMEM_BYTES =
        1024 + B_BUFS * B_BYTES + A_BUFS * A_BUF + EPI_BYTES + NUM_BARS * 8 + 16;
};

template <int BN, bool KSPLIT, int B_BUFS>
__global__ void __launch_bounds__(THREADS, 1)
wgrad_bstat_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmD, const __grid_constant__ TailMaps tmT,
                   Args args) {
    using S = BStatShape<BN, KSPLIT, B_BUFS>;
    constexpr uint32_t IDESC = idesc_bf16(BM, BN, true, true);
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw_addr = smem_u32(smem_raw);
    uint8_t *smem = smem_raw + ((1024u - (raw_addr & 1023u)) & 1023u);
    uint8_t *b_res = smem;  // B_BUFS x [hi kb0, hi kb1, lo kb0, lo kb1]
    uint8_t *a_ring = b_res + B_BUFS * S::B_BYTES;          // 2 x [kb0, kb1]
    uint8_t *epi_base = a_ring + S::A_BUFS * S::A_BUF;
    uint64_t *bars = reinterpret_cast<uint64_t *>(epi_base + S::EPI_BYTES);
    int *misc = reinterpret_cast<int *>(bars + S::NUM_BARS);  // [0] tmem base, [1] abort
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    auto bar_afull = [&](int i) { return smem_u32(bars + 0 + i); };
    auto bar_aempty = [&](int i) { return smem_u32(bars + 2 + i); };
    auto bar_tfull = [&](int i) { return smem_u32(bars + 4 + i); };
    auto bar_tempty = [&](int i) { return smem_u32(bars + 6 + i); };
    const uint32_t bar_drain = smem_u32(bars + 8);
    auto bar_bfull = [&](int i) { return smem_u32(bars + 9 + i); };
    auto bar_bempty = [&](int i) { return smem_u32(bars + 9 + B_BUFS + i); };
    volatile int *abort_flag = misc + 1;

    if (tid == 0) {
        for (int i = 0; i < B_BUFS; ++i) {
            mbar_init(bar_bfull(i), 1);
            mbar_init(bar_bempty(i), 1);
        }
        for (int i = 0; i < 2; ++i) {
            mbar_init(bar_afull(i), 1);
            mbar_init(bar_aempty(i), 1);
            mbar_init(bar_tfull(i), 1);
            mbar_init(bar_tempty(i), 8);
        }
        mbar_init(bar_drain, 1);
        misc[1] = 0;
        fence_barrier_init();
        fence_proxy_async();
        prefetch_map(&tmA);
        prefetch_map(&tmB);
        prefetch_map(&tmD);
        for (int i = 0; i < 3; ++i) {
            prefetch_map(&tmT.a[i]);
            prefetch_map(&tmT.b[i]);
        }
    }
    if (warp == 0) {
        tmem_alloc(smem_u32(misc), S::TMEM_COLS);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    pdl_wait();  // the predecessor's outputs are complete from here on
    const uint32_t tmem_base = (uint32_t)misc[0];
    const int nch = (args.tiles_m + S::MCH - 1) / S::MCH;
    const int total = args.G * args.tiles_n * nch;
    // unit u -> entry (its real group g and compact row crow), column tile,
    // first row tile and row-tile count
    int crow = 0;
    auto decode = [&](int u, int &g, int &n_blk, int &m0, int &mcnt, int &L) {
        const int i = u / (args.tiles_n * nch);
        const int r = u - i * args.tiles_n * nch;
        g = real_group(args, i);
        crow = args.crow ? __ldg(args.crow + i) : 0;
        n_blk = r / nch;
        m0 = (r - n_blk * nch) * S::MCH;
        mcnt = min(S::MCH, args.tiles_m - m0);
        L = __ldg(args.load + g);
        L = L < 0 ? 0 : (L > args.C ? args.C : L);
    };

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            int ub = 0;  // units with rows, in order: B buffer ub % B_BUFS
            int ia = 0;
            bool ok = true;
            int b_issued[B_BUFS] = {}, a_issued[2] = {0, 0};
            for (int u = blockIdx.x; u < total && ok; u += gridDim.x) {
                int g, n_blk, m0, mcnt, L;
                decode(u, g, n_blk, m0, mcnt, L);
                if (u + (int)gridDim.x >= total) pdl_launch_dependents();  // this CTA's last unit
                const int nkb = (L + BK - 1) / BK;
                if (nkb == 0) continue;
                const int bb = ub % B_BUFS;
                if (!wait_phase(bar_bempty(bb), (uint32_t)((ub / B_BUFS) & 1) ^ 1u, abort_flag,
                                args.status))
                    break;
                const uint32_t bdst = smem_u32(b_res) + bb * S::B_BYTES;
                // the last k-block loads R = tail_rows(rem) rows (chunk stride R x 128)
                const int Rl = tail_rows(L - (nkb - 1) * BK);
                const uint32_t bbytes = (uint32_t)((nkb - 1) * BK + Rl) * (BN / 64) * 128u;
                mbar_expect_tx(bar_bfull(bb), (KSPLIT ? 2u : 1u) * bbytes);
                const bool cmpb = (args.compact & CMP_B) != 0;  // B rows from crow, residual after L
                for (int kb = 0; kb < nkb; ++kb) {
                    const CUtensorMap *mB = kb == nkb - 1 && Rl < BK ? &tmT.b[Rl / 16 - 1] : &tmB;
                    tma_load_4d(bdst + kb * S::B_KB, mB, bar_bfull(bb), 0,
                                (cmpb ? crow : 0) + kb * BK, n_blk * (BN / 64), cmpb ? 0 : g);
                    if (KSPLIT)
                        tma_load_4d(bdst + (2 + kb) * S::B_KB, mB, bar_bfull(bb), 0,
                                    (cmpb ? crow + L : args.C) + kb * BK, n_blk * (BN / 64),
                                    cmpb ? 0 : g);
                }
                ++b_issued[bb];
                ++ub;
                for (int m = m0; m < m0 + mcnt; ++m, ++ia) {
                    const int ab = ia % S::A_BUFS;
                    if (!wait_phase(bar_aempty(ab), (uint32_t)((ia / S::A_BUFS) & 1) ^ 1u, abort_flag,
                                    args.status)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(bar_afull(ab), (uint32_t)((nkb - 1) * BK + Rl) * (BM / 64) * 128u);
                    for (int kb = 0; kb < nkb; ++kb)
                        tma_load_4d(smem_u32(a_ring) + ab * S::A_BUF + kb * S::A_KB,
                                    kb == nkb - 1 && Rl < BK ? &tmT.a[Rl / 16 - 1] : &tmA,
                                    bar_afull(ab), 0, kb * BK, m * (BM / 64), g);
                    ++a_issued[ab];
                }
            }
            if (*abort_flag) {  // let copies in flight land before the CTA exits
                const unsigned long long t0 = global_ns();
                for (int i = 0; i < B_BUFS; ++i)
                    if (b_issued[i] > 0)
                        while (!mbar_try_wait(bar_bfull(i), (uint32_t)((b_issued[i] - 1) & 1)) &&
                               global_ns() - t0 < 100000000ull) {
                        }
                for (int i = 0; i < 2; ++i)
                    if (a_issued[i] > 0)
                        while (!mbar_try_wait(bar_afull(i), (uint32_t)((a_issued[i] - 1) & 1)) &&
                               global_ns() - t0 < 200000000ull) {
                        }
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        int ub = 0;
        int ia = 0, it = 0;
        bool ok = true;
        // rows [z0, z1) of every 64-wide chunk of the last k-block tile, whose
        // chunks are z1 x 128 bytes apart (it holds z1 = tail_rows rows), are zeroed
        auto zero_rows = [&](uint8_t *tile, int chunks, int z0, int z1) {
            const int rows = z1 - z0;
            const int units = chunks * rows * 8;
            for (int i = lane; i < units; i += 32) {
                const int c = i / (rows * 8);
                const int w = i - c * rows * 8;
                *reinterpret_cast<uint4 *>(tile + c * (z1 * 128) + (z0 + (w >> 3)) * 128 + (w & 7) * 16) =
                    make_uint4(0, 0, 0, 0);
            }
        };
        for (int u = blockIdx.x; u < total && ok; u += gridDim.x) {
            int g, n_blk, m0, mcnt, L;
            decode(u, g, n_blk, m0, mcnt, L);
            const int nkb = (L + BK - 1) / BK;
            const int rem = L - (nkb - 1) * BK;       // valid rows of the last k-block
            const int nk_last = (rem + 15) >> 4;      // MMAs (K = 16) in the last k-block
            const int bb = ub % B_BUFS;
            uint8_t *bres = b_res + bb * S::B_BYTES;
            if (nkb > 0) {
                if (!wait_phase(bar_bfull(bb), (uint32_t)((ub / B_BUFS) & 1), abort_flag, args.status))
                    break;
                tc_fence_after();
                if (rem < nk_last * 16) {  // K tail of the resident B: zero once per unit
                    zero_rows(bres + (nkb - 1) * S::B_KB, BN / 64, rem, nk_last * 16);
                    if (KSPLIT) zero_rows(bres + (1 + nkb) * S::B_KB, BN / 64, rem, nk_last * 16);
                    fence_proxy_async();
                }
                __syncwarp();
            }
            for (int m = m0; m < m0 + mcnt; ++m, ++it) {
                const int acc = it & 1;
                if (!wait_phase(bar_tempty(acc), (uint32_t)((it >> 1) & 1) ^ 1u, abort_flag,
                                args.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                if (nkb == 0) {
                    if (lane == 0) mbar_arrive(bar_tfull(acc));
                    __syncwarp();
                    continue;
                }
                const int ab = ia % S::A_BUFS;
                if (!wait_phase(bar_afull(ab), (uint32_t)((ia / S::A_BUFS) & 1), abort_flag, args.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                uint8_t *abuf = a_ring + ab * S::A_BUF;
                if (rem < nk_last * 16) {
                    zero_rows(abuf + (nkb - 1) * S::A_KB, BM / 64, rem, nk_last * 16);
                    fence_proxy_async();
                }
                __syncwarp();
                if (lane == 0) {
                    const uint32_t dtmem = tmem_base + (uint32_t)(acc * BN);
                    const uint32_t a0 = smem_u32(abuf), b0 = smem_u32(bres);
                    for (int part = 0; part < (KSPLIT ? 2 : 1); ++part)
                        for (int kb = 0; kb < nkb; ++kb) {
                            const int nk = kb == nkb - 1 ? nk_last : BK / 16;
                            const uint32_t at = a0 + kb * S::A_KB;
                            const uint32_t bt = b0 + (part * 2 + kb) * S::B_KB;
                            for (int kk = 0; kk < nk; ++kk)  // k-block of 16 nk rows (the last one: tail_rows)
                                mma_bf16(dtmem, operand_desc_mn(at, kk, nk * 16), operand_desc_mn(bt, kk, nk * 16),
                                         IDESC, (part | kb | kk) != 0 ? 1u : 0u);
                        }
                    mma_commit(bar_aempty(ab));
                    mma_commit(bar_tfull(acc));
                }
                __syncwarp();
                ++ia;
            }
            if (!ok) break;
            if (nkb > 0) {
                if (lane == 0) mma_commit(bar_bempty(bb));  // B may be replaced once these MMAs finish
                __syncwarp();
                ++ub;
            }
        }
        if (lane == 0) {
            mma_commit(bar_drain);
            const unsigned long long t0 = global_ns();
            while (!mbar_try_wait(bar_drain, 0) && global_ns() - t0 < 1000000000ull) {
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int ew = warp - 2;
        const int q = warp & 3;
        const int half = ew >> 2;
        constexpr int COLS = BN / 2;
        uint8_t *stg = epi_base + ew * S::STG_BUFS * 4096;
        int nstore = 0, it = 0;
        bool ok = true;
        for (int u = blockIdx.x; u < total && ok; u += gridDim.x) {
            int g, n_blk, m0, mcnt, L;
            decode(u, g, n_blk, m0, mcnt, L);
            for (int m = m0; m < m0 + mcnt; ++m, ++it) {
                const int acc = it & 1;
                if (!wait_phase(bar_tfull(acc), (uint32_t)((it >> 1) & 1), abort_flag, args.status)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const int row0 = m * BM + q * 32;
                const int colw = n_blk * BN + half * COLS;
                const uint32_t trow = tmem_base + ((uint32_t)(q * 32) << 16) +
                                      (uint32_t)(acc * BN + half * COLS);
                // all of this warp's accumulator columns with one wait, then
                // 32 x 64 chunks through the staging tile(s) and TMA stores
                uint32_t r[COLS / 32][32];
                if (L > 0) {
#pragma unroll
                    for (int i = 0; i < COLS / 32; ++i) tmem_ld32(trow + i * 32, r[i]);
                    tmem_ld_wait();
                } else {
#pragma unroll
                    for (int i = 0; i < COLS / 32; ++i)
#pragma unroll
                        for (int j = 0; j < 32; ++j) r[i][j] = 0u;
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(bar_tempty(acc));
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
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 0) tmem_dealloc(tmem_base, S::TMEM_COLS);
}

// ---------------------------------------------------------------------------
// Host side.

// Encodes a rank-3 bf16 tensor map {inner, mid, outer} (inner contiguous) with
// a {64, box_mid, 1} box and 128-byte swizzle; out-of-range elements read 0.
bool make_map(CUtensorMap *map, const void *base, uint64_t inner, uint64_t mid, uint64_t outer,
              uint32_t box_mid, uint64_t outer_stride_elems = 0);

// Encodes a rank-4 view of a [outer][rows][mn] bf16 tensor whose mn axis is cut
// into 64-element chunks: dims {64, rows, mn/64, outer}.  A {64, box_rows,
// box_chunks, 1} box then lands in shared memory chunk-major -- box_chunks
// tiles of box_rows x 128 bytes (128-byte swizzle) -- which is the MN-major
// operand layout, in one copy instead of one per chunk.
// outer_stride_elems: elements from one outer index to the next (0: rows x mn).
bool make_map_chunked(CUtensorMap *map, const void *base, uint64_t mn, uint64_t rows,
                      uint64_t outer, uint32_t box_rows, uint32_t box_chunks,
                      uint64_t outer_stride_elems = 0);

template <int BN, int MODE, bool A_MN, bool B_MN, int EPI>
int launch(const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &md,
           const CUtensorMap &md2, const TailMaps &mat, const Args &a, long long max_tiles,
           cudaStream_t s, const char *name) {
    using S = Shape<BN, MODE, EPI>;
    auto kern = grouped_gemm_kernel<BN, MODE, A_MN, B_MN, EPI>;
    static std::atomic<int> smem_limit[64];
    if (const int st = raise_smem_limit((const void *)kern, smem_limit, (int)S::SMEM_BYTES)) return st;
    if (max_tiles <= 0) return VMOE_OK;
    long long grid = max_tiles < num_sms() ? max_tiles : num_sms();
    trace_before(s, name);
    const int st = launch_kernel(kern, dim3((unsigned)grid), dim3(S::NT), S::SMEM_BYTES, s, ma, mb,
                                 md, md2, mat, a);
    trace_after(s);
    return st;
}

template <int BN, bool KSPLIT, int B_BUFS>
int launch_bstat(const CUtensorMap &ma, const CUtensorMap &mb, const CUtensorMap &md, const TailMaps &mt,
                 const Args &a, long long units, cudaStream_t s, const char *name) {
    using S = BStatShape<BN, KSPLIT, B_BUFS>;
    auto kern = wgrad_bstat_kernel<BN, KSPLIT, B_BUFS>;
    static std::atomic<int> smem_limit[64];
    if (const int st = raise_smem_limit((const void *)kern, smem_limit, (int)S::SMEM_BYTES)) return st;
    if (units <= 0) return VMOE_OK;
    long long grid = units < num_sms() ? units : num_sms();
    trace_before(s, name);
    const int st = launch_kernel(kern, dim3((unsigned)grid), dim3(THREADS), S::SMEM_BYTES, s, ma, mb,
                                 md, mt, a);
    trace_after(s);
    return st;
}

// A slice of the groups for one launch (the memory-budgeted backward): n
// entries, entry i = group glist[i]; the operands flagged in `compact` live in
// a compact buffer of `rows` rows, entry i's rows from crow[i].  n == 0: all
// groups, nothing compact.
struct Slice {
    const int32_t *glist = nullptr;  // device
    const int32_t *crow = nullptr;   // device
    int n = 0;
    int compact = 0;
    long long rows = 0;
};

inline Args base_args(const Dims &p, const int32_t *load) {
    Args a = {};
    a.G = p.G();
    a.C = p.C;
    a.load = load;
    a.gelu_tanh = (p.flags & VMOE_GELU_TANH) != 0;
    a.status = device_status_word();
    return a;
}

}  // namespace tc
}  // namespace vmoe
