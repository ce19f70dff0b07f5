// attention.cu -- attention experts: H-head softmax attention among the tokens
// routed to each (task, expert) group (Section 2.1 expertizes the ViT's
// attention as well as its MLP; Section 3.2.1's estimator gives such an expert
// buffers of order T d_k for Q / K / V and T^2 for the scores).
//
// One expert's forward, for its L = load[g] routed tokens Xe[g] rows [0, L):
//   QKV = Xe W_qkv           [L, 3 H dk]  (columns: Q heads | K heads | V heads)
//   per head h:  S = Q_h K_h^T / sqrt(dk),  P = softmax over the L keys,  O_h = P V_h
//   Ye = O W_o               [L, d]
// and its backward (routing and gates fixed):
//   dO = dYe W_o^T,  dW_o = O^T dYe,  D = rowsum(dO * O) per head,
//   dS = P * (dO_h V_h^T - D),  dQ_h = dS K_h / sqrt(dk),  dK_h = dS^T Q_h / sqrt(dk),
//   dV_h = P^T dO_h,  dXe = dQKV W_qkv^T,  dW_qkv = Xe^T dQKV.
// The projections and their gradients are the grouped tcgen05 GEMMs of the FFN
// experts (row mode and weight-gradient mode).  The attention core is here:
// flash-attention style kernels on mma.sync (m16n8k16, bf16 in, fp32
// accumulate), one CTA per (group, head, block of 64 rows), 4 warps of 16
// rows.  Each CTA keeps the whole group's keys (or queries) of its head in
// shared memory -- a group holds at most C <= 512 tokens -- so the softmax of a
// row runs online over key blocks of 64 with the row maximum subtracted, and
// the forward saves each row's log-sum-exp for the backward to rebuild P.
// The tiles arrive by cp.async, one commit group per block of 64 keys (or
// queries), so the work on block j overlaps the copies of the blocks after it.
// Keys (or queries) past the load are masked; rows past it are never stored.
// There are no atomics: dQ is one kernel over query blocks, dK and dV another
// over key blocks, so every sum runs in a fixed order.
#include <math.h>

#include "common.cuh"

namespace vmoe {
namespace {

constexpr int AT_DK = 64;       // head dimension
constexpr int AT_BLK = 64;      // rows per CTA block (4 warps x 16)
constexpr int AT_THREADS = 128;
constexpr int AT_PITCH = 72;    // bf16 per shared row: 64 + 8 pad (144 B, conflict-free ldmatrix)
constexpr int AT_MAX_C = 512;
// The backward kernels are built for at least 3 CTAs per SM (at most 170
// registers a thread): dK/dV otherwise takes 222 registers and runs 2 CTAs per
// SM (measured at the 17-task shape: 467 -> 385 us for dK/dV, 314 -> 305 us
// for dQ).  The forward keeps the compiler's choice (104 registers), which
// measured faster than with the bound.
constexpr int AT_MIN_CTAS_BWD = 3;

struct AtArgs {
    int G, C, H;
    const int32_t *load;
    const __nv_bfloat16 *qkv;   // [G, C, 3 H dk]
    const __nv_bfloat16 *o;     // [G, C, H dk]
    const __nv_bfloat16 *dout;  // [G, C, H dk] (backward)
    __nv_bfloat16 *o_out;       // forward output O
    float *lse;                 // [G, H, C]
    float *dsum;                // [G, H, C]: D = rowsum(dO * O)
    __nv_bfloat16 *dqkv;        // [G, C, 3 H dk] (backward output)
    float scale;                // 1 / sqrt(dk)
};

__device__ __forceinline__ void at_ldsm_x4(uint32_t (&r)[4], const __nv_bfloat16 *p) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(a));
}
__device__ __forceinline__ void at_ldsm_x4_t(uint32_t (&r)[4], const __nv_bfloat16 *p) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(a));
}

__device__ __forceinline__ int clamp_load(const int32_t *load, int g, int C) {
    int L = __ldg(load + g);
    return L < 0 ? 0 : (L > C ? C : L);
}

// Rows [r0, r0 + n) of the 64 columns at `col` of a [C][ld] bf16 matrix of group
// g into a shared tile [n][AT_PITCH], rows at or past `valid` zero, by cp.async
// (16-byte copies straight to shared memory, zero-filled past `valid`; an
// invalid row's source address is clamped to row 0, which is not read), in the
// commit group the caller closes.
template <int NTHREADS>
__device__ __forceinline__ void at_cp_rows_n(__nv_bfloat16 *dst, const __nv_bfloat16 *src, int ld, int r0, int n,
                                             int valid, int col) {
    for (int i = threadIdx.x; i < n * 8; i += NTHREADS) {
        const int r = i >> 3, c8 = (i & 7) * 8;
        const bool ok = r0 + r < valid;
        const __nv_bfloat16 *g = src + (long long)(ok ? r0 + r : 0) * ld + col + c8;
        const uint32_t d = (uint32_t)__cvta_generic_to_shared(dst + r * AT_PITCH + c8);
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(d), "l"(g), "r"(ok ? 16 : 0)
                     : "memory");
    }
}
__device__ __forceinline__ void at_cp_rows(__nv_bfloat16 *dst, const __nv_bfloat16 *src, int ld, int r0, int n,
                                           int valid, int col) {
    at_cp_rows_n<AT_THREADS>(dst, src, ld, r0, n, valid, col);
}
__device__ __forceinline__ void at_cp_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
// Waits until at most `pending` of this thread's newest commit groups are still
// in flight (0..7: a group holds at most 8 key or query blocks), then makes
// every thread's landed copies visible to the CTA.
__device__ __forceinline__ void at_cp_wait(int pending) {
    switch (pending) {
        case 0: asm volatile("cp.async.wait_group 0;\n" ::: "memory"); break;
        case 1: asm volatile("cp.async.wait_group 1;\n" ::: "memory"); break;
        case 2: asm volatile("cp.async.wait_group 2;\n" ::: "memory"); break;
        case 3: asm volatile("cp.async.wait_group 3;\n" ::: "memory"); break;
        case 4: asm volatile("cp.async.wait_group 4;\n" ::: "memory"); break;
        case 5: asm volatile("cp.async.wait_group 5;\n" ::: "memory"); break;
        case 6: asm volatile("cp.async.wait_group 6;\n" ::: "memory"); break;
        default: asm volatile("cp.async.wait_group 7;\n" ::: "memory"); break;
    }
    __syncthreads();
}

// A fragments (16 rows x 64 columns, four k16 steps) of a warp's 16 rows of a
// shared tile.
__device__ __forceinline__ void at_afrag(uint32_t (&a)[4][4], const __nv_bfloat16 *tile, int row0) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) at_ldsm_x4(a[ks], tile + (row0 + (lane & 15)) * AT_PITCH + ks * 16 + (lane >> 4) * 8);
}

// acc[8][4] (16 x 64) += A (16 x 64 via four k16 fragments) * B^T, B = 64 rows of
// a shared tile starting at brow: out[i][j] = sum_k A[i][k] B[j][k].
__device__ __forceinline__ void at_mma_abt(float (&acc)[8][4], const uint32_t (&a)[4][4], const __nv_bfloat16 *tile,
                                           int brow) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks)
#pragma unroll
        for (int np = 0; np < 4; ++np) {
            uint32_t b[4];
            at_ldsm_x4(b, tile + (brow + np * 16 + (lane & 7) + (lane >> 4) * 8) * AT_PITCH + ks * 16 +
                              ((lane >> 3) & 1) * 8);
            mma_bf16_16816(acc[2 * np], a[ks][0], a[ks][1], a[ks][2], a[ks][3], b[0], b[1]);
            mma_bf16_16816(acc[2 * np + 1], a[ks][0], a[ks][1], a[ks][2], a[ks][3], b[2], b[3]);
        }
}

// acc[8][4] (16 x 64) += P (16 x 64, fp32 accumulator layout, rounded to bf16)
// * B, B = 64 rows of a shared tile starting at brow (rows = the k index).
__device__ __forceinline__ void at_mma_pb(float (&acc)[8][4], const float (&p)[8][4], const __nv_bfloat16 *tile,
                                          int brow) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int kk = 0; kk < 4; ++kk) {
        const uint32_t a0 = pack_bf16x2(p[2 * kk][0], p[2 * kk][1]);
        const uint32_t a1 = pack_bf16x2(p[2 * kk][2], p[2 * kk][3]);
        const uint32_t a2 = pack_bf16x2(p[2 * kk + 1][0], p[2 * kk + 1][1]);
        const uint32_t a3 = pack_bf16x2(p[2 * kk + 1][2], p[2 * kk + 1][3]);
#pragma unroll
        for (int dp = 0; dp < 4; ++dp) {
            uint32_t b[4];
            const int m = lane >> 3;
            at_ldsm_x4_t(b, tile + (brow + kk * 16 + (m & 1) * 8 + (lane & 7)) * AT_PITCH + dp * 16 + (m >> 1) * 8);
            mma_bf16_16816(acc[2 * dp], a0, a1, a2, a3, b[0], b[1]);
            mma_bf16_16816(acc[2 * dp + 1], a0, a1, a2, a3, b[2], b[3]);
        }
    }
}

__device__ __forceinline__ void at_zero(float (&acc)[8][4]) {
#pragma unroll
    for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.0f;
}

// Writes a warp's 16 x 64 accumulator (times `mul`) as bf16 to rows row0.. of
// dst (row stride ld, column col), rows at or past `valid` skipped.
__device__ __forceinline__ void at_store(const float (&acc)[8][4], float mul, __nv_bfloat16 *dst, int ld, int row0,
                                         int valid, int col) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const int r = row0 + g + 8 * h;
        if (r >= valid) continue;
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
            *reinterpret_cast<uint32_t *>(dst + (long long)r * ld + col + nt * 8 + 2 * t) =
                pack_bf16x2(acc[nt][2 * h] * mul, acc[nt][2 * h + 1] * mul);
    }
}

__device__ __forceinline__ float quad_max(float v) {
    v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 1));
    return fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 2));
}
__device__ __forceinline__ float quad_sum(float v) {
    v += __shfl_xor_sync(0xffffffffu, v, 1);
    return v + __shfl_xor_sync(0xffffffffu, v, 2);
}

// ------------------------------------------------------------------ forward
// CTA (query block, head, group): O and the row log-sum-exp of 64 queries.
__global__ void __launch_bounds__(AT_THREADS) attn_fwd_kernel(AtArgs a) {
    pdl_wait();
    const int qb = blockIdx.x, h = blockIdx.y, g = blockIdx.z;
    const int L = clamp_load(a.load, g, a.C);
    const int q0 = qb * AT_BLK;
    if (q0 >= L) return;
    const int Lp = (L + AT_BLK - 1) / AT_BLK * AT_BLK;
    const int H = a.H, ld = 3 * H * AT_DK;
    extern __shared__ __align__(16) __nv_bfloat16 at_smem[];
    __nv_bfloat16 *qs = at_smem, *ks = qs + AT_BLK * AT_PITCH, *vs = ks + Lp * AT_PITCH;
    const __nv_bfloat16 *src = a.qkv + (long long)g * a.C * ld;
    // commit group 0: the queries and key block 0; group j: key block j
    const int nkb = Lp / AT_BLK;
    at_cp_rows(qs, src, ld, q0, AT_BLK, L, h * AT_DK);
    for (int j = 0; j < nkb; ++j) {
        at_cp_rows(ks + j * AT_BLK * AT_PITCH, src, ld, j * AT_BLK, AT_BLK, L, (H + h) * AT_DK);
        at_cp_rows(vs + j * AT_BLK * AT_PITCH, src, ld, j * AT_BLK, AT_BLK, L, (2 * H + h) * AT_DK);
        at_cp_commit();
    }
    at_cp_wait(nkb - 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, t = lane & 3;
    uint32_t qa[4][4];
    at_afrag(qa, qs, warp * 16);
    float o[8][4], mrow[2] = {-INFINITY, -INFINITY}, lrow[2] = {0.0f, 0.0f};
    at_zero(o);
    for (int kb = 0; kb < Lp; kb += AT_BLK) {
        if (kb > 0) at_cp_wait(nkb - 1 - kb / AT_BLK);
        float s[8][4];
        at_zero(s);
        at_mma_abt(s, qa, ks, kb);
        float mx[2] = {-INFINITY, -INFINITY};
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int key = kb + nt * 8 + 2 * t + (j & 1);
                s[nt][j] = key < L ? s[nt][j] * a.scale : -INFINITY;
                mx[j >> 1] = fmaxf(mx[j >> 1], s[nt][j]);
            }
        float corr[2], rs[2] = {0.0f, 0.0f};
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) {
            const float mn = fmaxf(mrow[h2], quad_max(mx[h2]));
            corr[h2] = __expf(mrow[h2] - mn);
            mrow[h2] = mn;
        }
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                s[nt][j] = __expf(s[nt][j] - mrow[j >> 1]);
                rs[j >> 1] += s[nt][j];
                o[nt][j] *= corr[j >> 1];
            }
#pragma unroll
        for (int h2 = 0; h2 < 2; ++h2) lrow[h2] = lrow[h2] * corr[h2] + quad_sum(rs[h2]);
        at_mma_pb(o, s, vs, kb);
    }
    // O = (P V) / l; lse = m + log l
    const int row0 = q0 + warp * 16, g8 = lane >> 2;
    const long long ob = (long long)g * a.C * (H * AT_DK);
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
        const float inv = 1.0f / lrow[h2];
#pragma unroll
        for (int nt = 0; nt < 8; ++nt) {
            o[nt][2 * h2] *= inv;
            o[nt][2 * h2 + 1] *= inv;
        }
        const int r = row0 + g8 + 8 * h2;
        if (t == 0 && r < L) a.lse[((long long)g * H + h) * a.C + r] = mrow[h2] + logf(lrow[h2]);
    }
    at_store(o, 1.0f, a.o_out + ob, H * AT_DK, row0, L, h * AT_DK);
}

// ------------------------------------------------------------------ backward: dQ (and D)
// CTA (query block, head, group): D = rowsum(dO * O) of its 64 queries, then
// dQ = sum over key blocks of dS K, dS = P * (dO V^T - D), P = exp(S - lse).
__global__ void __launch_bounds__(AT_THREADS, AT_MIN_CTAS_BWD) attn_bwd_dq_kernel(AtArgs a) {
    pdl_wait();
    const int qb = blockIdx.x, h = blockIdx.y, g = blockIdx.z;
    const int L = clamp_load(a.load, g, a.C);
    const int q0 = qb * AT_BLK;
    if (q0 >= L) return;
    const int Lp = (L + AT_BLK - 1) / AT_BLK * AT_BLK;
    const int H = a.H, ld = 3 * H * AT_DK, ldo = H * AT_DK;
    extern __shared__ __align__(16) __nv_bfloat16 at_smem[];
    __nv_bfloat16 *qs = at_smem, *dos = qs + AT_BLK * AT_PITCH, *os = dos + AT_BLK * AT_PITCH;
    __nv_bfloat16 *ks = os + AT_BLK * AT_PITCH, *vs = ks + Lp * AT_PITCH;
    float *dsh = reinterpret_cast<float *>(vs + Lp * AT_PITCH);  // [64] D of the block
    const __nv_bfloat16 *src = a.qkv + (long long)g * a.C * ld;
    const long long ob = (long long)g * a.C * ldo;
    // commit group 0: this block's Q, dO, O and key block 0; group j: key block j
    const int nkb = Lp / AT_BLK;
    at_cp_rows(qs, src, ld, q0, AT_BLK, L, h * AT_DK);
    at_cp_rows(dos, a.dout + ob, ldo, q0, AT_BLK, L, h * AT_DK);
    at_cp_rows(os, a.o + ob, ldo, q0, AT_BLK, L, h * AT_DK);
    for (int j = 0; j < nkb; ++j) {
        at_cp_rows(ks + j * AT_BLK * AT_PITCH, src, ld, j * AT_BLK, AT_BLK, L, (H + h) * AT_DK);
        at_cp_rows(vs + j * AT_BLK * AT_PITCH, src, ld, j * AT_BLK, AT_BLK, L, (2 * H + h) * AT_DK);
        at_cp_commit();
    }
    at_cp_wait(nkb - 1);
    // D: two threads per row, 32 columns each, in a fixed order
    {
        const int r = threadIdx.x >> 1, c0 = (threadIdx.x & 1) * 32;
        float acc = 0.0f;
#pragma unroll 8
        for (int c = 0; c < 32; ++c)
            acc += __bfloat162float(dos[r * AT_PITCH + c0 + c]) * __bfloat162float(os[r * AT_PITCH + c0 + c]);
        acc += __shfl_xor_sync(0xffffffffu, acc, 1);
        if ((threadIdx.x & 1) == 0) {
            dsh[r] = acc;
            if (q0 + r < L) a.dsum[((long long)g * H + h) * a.C + q0 + r] = acc;
        }
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, t = lane & 3, g8 = lane >> 2;
    uint32_t qa[4][4], da[4][4];
    at_afrag(qa, qs, warp * 16);
    at_afrag(da, dos, warp * 16);
    float lse[2], dd[2];
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
        const int rl = warp * 16 + g8 + 8 * h2, r = q0 + rl;
        lse[h2] = r < L ? __ldg(a.lse + ((long long)g * H + h) * a.C + r) : 0.0f;
        dd[h2] = dsh[rl];
    }
    float dq[8][4];
    at_zero(dq);
    for (int kb = 0; kb < Lp; kb += AT_BLK) {
        if (kb > 0) at_cp_wait(nkb - 1 - kb / AT_BLK);
        float s[8][4], dp[8][4];
        at_zero(s);
        at_zero(dp);
        at_mma_abt(s, qa, ks, kb);
        at_mma_abt(dp, da, vs, kb);
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int key = kb + nt * 8 + 2 * t + (j & 1);
                const float p = key < L ? __expf(s[nt][j] * a.scale - lse[j >> 1]) : 0.0f;
                s[nt][j] = p * (dp[nt][j] - dd[j >> 1]);  // dS
            }
        at_mma_pb(dq, s, ks, kb);
    }
    at_store(dq, a.scale, a.dqkv + (long long)g * a.C * ld, ld, q0 + warp * 16, L, h * AT_DK);
}

// ------------------------------------------------------------------ backward: dK, dV
// CTA (key block, head, group): for its 64 keys, over query blocks,
//   P^T = exp(K Q^T / sqrt(dk) - lse),  dV += P^T dO,
//   dS^T = P^T * (V dO^T - D),  dK += dS^T Q / sqrt(dk).
__global__ void __launch_bounds__(AT_THREADS, AT_MIN_CTAS_BWD) attn_bwd_dkv_kernel(AtArgs a) {
    pdl_wait();
    const int kbk = blockIdx.x, h = blockIdx.y, g = blockIdx.z;
    const int L = clamp_load(a.load, g, a.C);
    const int k0 = kbk * AT_BLK;
    if (k0 >= L) return;
    const int Lp = (L + AT_BLK - 1) / AT_BLK * AT_BLK;
    const int H = a.H, ld = 3 * H * AT_DK, ldo = H * AT_DK;
    extern __shared__ __align__(16) __nv_bfloat16 at_smem[];
    __nv_bfloat16 *ks = at_smem, *vs = ks + AT_BLK * AT_PITCH, *qs = vs + AT_BLK * AT_PITCH;
    __nv_bfloat16 *dos = qs + Lp * AT_PITCH;
    float *lse_s = reinterpret_cast<float *>(dos + Lp * AT_PITCH), *d_s = lse_s + Lp;
    const __nv_bfloat16 *src = a.qkv + (long long)g * a.C * ld;
    const long long ob = (long long)g * a.C * ldo;
    // commit group 0: this block's K, V and query block 0; group j: query block j
    const int nqb = Lp / AT_BLK;
    at_cp_rows(ks, src, ld, k0, AT_BLK, L, (H + h) * AT_DK);
    at_cp_rows(vs, src, ld, k0, AT_BLK, L, (2 * H + h) * AT_DK);
    for (int j = 0; j < nqb; ++j) {
        at_cp_rows(qs + j * AT_BLK * AT_PITCH, src, ld, j * AT_BLK, AT_BLK, L, h * AT_DK);
        at_cp_rows(dos + j * AT_BLK * AT_PITCH, a.dout + ob, ldo, j * AT_BLK, AT_BLK, L, h * AT_DK);
        at_cp_commit();
    }
    for (int i = threadIdx.x; i < Lp; i += AT_THREADS) {
        const bool v = i < L;
        lse_s[i] = v ? __ldg(a.lse + ((long long)g * H + h) * a.C + i) : 0.0f;
        d_s[i] = v ? __ldg(a.dsum + ((long long)g * H + h) * a.C + i) : 0.0f;
    }
    at_cp_wait(nqb - 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, t = lane & 3;
    uint32_t ka[4][4], va[4][4];
    at_afrag(ka, ks, warp * 16);
    at_afrag(va, vs, warp * 16);
    float dk[8][4], dv[8][4];
    at_zero(dk);
    at_zero(dv);
    for (int qb = 0; qb < Lp; qb += AT_BLK) {
        if (qb > 0) at_cp_wait(nqb - 1 - qb / AT_BLK);
        float st[8][4], dpt[8][4];
        at_zero(st);
        at_zero(dpt);
        at_mma_abt(st, ka, qs, qb);   // K Q^T: [16 keys x 64 queries]
        at_mma_abt(dpt, va, dos, qb); // V dO^T
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int q = qb + nt * 8 + 2 * t + (j & 1);
                st[nt][j] = q < L ? __expf(st[nt][j] * a.scale - lse_s[q]) : 0.0f;  // P^T
                dpt[nt][j] = st[nt][j] * (dpt[nt][j] - d_s[q]);                     // dS^T
            }
        at_mma_pb(dv, st, dos, qb);
        at_mma_pb(dk, dpt, qs, qb);
    }
    __nv_bfloat16 *dst = a.dqkv + (long long)g * a.C * ld;
    at_store(dk, a.scale, dst, ld, k0 + warp * 16, L, (H + h) * AT_DK);
    at_store(dv, 1.0f, dst, ld, k0 + warp * 16, L, (2 * H + h) * AT_DK);
}

// ------------------------------------------------------------------ backward, groups of <= 128 tokens
// One CTA of 8 warps per (head, group) with L <= 128: S, P, dP and dS are formed
// once for all queries and keys instead of in both kernels above.  Warp w owns
// queries [16 w, 16 w + 16).  Per block of 64 keys: S = Q K^T, dP = dO V^T,
// P = exp(S / sqrt(dk) - lse), dS = P (dP - D) (zero for queries or keys past
// L), dQ += dS K in registers; P and dS (bf16, as the MMAs round them) go to
// shared memory, and warps 0-3 form dV = P^T dO and warps 4-7 dK = dS^T Q for
// the block's 64 keys (16 a warp), summed over the queries in increasing order.
constexpr int AF_THREADS = 256;
constexpr int AF_ROWS = 128;

// acc[8][4] (16 keys x 64) += A^T B: A = 16 key columns (from acol) of a shared
// [query][key] tile, B = a shared [query][64] tile, over queries [0, nq) in
// steps of 16 (A fragments by ldmatrix.trans: A's rows are the tile's columns).
__device__ __forceinline__ void at_mma_tb(float (&acc)[8][4], const __nv_bfloat16 *atile, int acol,
                                          const __nv_bfloat16 *btile, int nq) {
    const int lane = threadIdx.x & 31, m = lane >> 3;
    for (int q0 = 0; q0 < nq; q0 += 16) {
        uint32_t a[4];
        at_ldsm_x4_t(a, atile + (q0 + (lane & 7) + (lane >> 4) * 8) * AT_PITCH + acol + (m & 1) * 8);
#pragma unroll
        for (int dp = 0; dp < 4; ++dp) {
            uint32_t b[4];
            at_ldsm_x4_t(b, btile + (q0 + (m & 1) * 8 + (lane & 7)) * AT_PITCH + dp * 16 + (m >> 1) * 8);
            mma_bf16_16816(acc[2 * dp], a[0], a[1], a[2], a[3], b[0], b[1]);
            mma_bf16_16816(acc[2 * dp + 1], a[0], a[1], a[2], a[3], b[2], b[3]);
        }
    }
}

// A warp's 16 x 64 fp32 tile as bf16 into rows row0.. of a shared [rows][AT_PITCH] tile.
__device__ __forceinline__ void at_put(__nv_bfloat16 *tile, int row0, const float (&v)[8][4]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
            *reinterpret_cast<uint32_t *>(tile + (row0 + g + 8 * h) * AT_PITCH + nt * 8 + 2 * t) =
                pack_bf16x2(v[nt][2 * h], v[nt][2 * h + 1]);
}

__global__ void __launch_bounds__(AF_THREADS, 2) attn_bwd_fused_kernel(AtArgs a) {
    pdl_wait();
    const int h = blockIdx.y, g = blockIdx.z;
    const int L = clamp_load(a.load, g, a.C);
    if (L == 0) return;
    const int Lp = (L + AT_BLK - 1) / AT_BLK * AT_BLK;  // 64 or 128
    const int H = a.H, ld = 3 * H * AT_DK, ldo = H * AT_DK;
    extern __shared__ __align__(16) __nv_bfloat16 at_smem[];
    __nv_bfloat16 *qs = at_smem, *ks = qs + AF_ROWS * AT_PITCH, *vs = ks + AF_ROWS * AT_PITCH;
    __nv_bfloat16 *dos = vs + AF_ROWS * AT_PITCH;
    __nv_bfloat16 *ps = dos + AF_ROWS * AT_PITCH, *dss = ps + AF_ROWS * AT_PITCH;  // one 64-key block
    float *dsh = reinterpret_cast<float *>(dss + AF_ROWS * AT_PITCH), *lse_s = dsh + AF_ROWS;
    const __nv_bfloat16 *src = a.qkv + (long long)g * a.C * ld;
    const long long ob = (long long)g * a.C * ldo;
    // all 128 rows of each tile: rows past L are zero-filled (no global read)
    at_cp_rows_n<AF_THREADS>(qs, src, ld, 0, AF_ROWS, L, h * AT_DK);
    at_cp_rows_n<AF_THREADS>(dos, a.dout + ob, ldo, 0, AF_ROWS, L, h * AT_DK);
    at_cp_rows_n<AF_THREADS>(ks, src, ld, 0, AF_ROWS, L, (H + h) * AT_DK);
    at_cp_rows_n<AF_THREADS>(vs, src, ld, 0, AF_ROWS, L, (2 * H + h) * AT_DK);
    at_cp_commit();
    for (int i = threadIdx.x; i < AF_ROWS; i += AF_THREADS)
        lse_s[i] = i < L ? __ldg(a.lse + ((long long)g * H + h) * a.C + i) : 0.0f;
    // D = rowsum(dO * O): two threads per row, 32 columns each, in a fixed order
    // (O straight from global memory; dO from shared memory once it has landed)
    float oc[32];
    {
        const int r = threadIdx.x >> 1, c0 = (threadIdx.x & 1) * 32;
#pragma unroll
        for (int c = 0; c < 32; c += 8) {
            uint4 v = make_uint4(0, 0, 0, 0);
            if (r < L) v = __ldg(reinterpret_cast<const uint4 *>(a.o + ob + (long long)r * ldo + h * AT_DK + c0 + c));
            bf16x8_to_f32(v, oc + c);
        }
    }
    at_cp_wait(0);
    {
        const int r = threadIdx.x >> 1, c0 = (threadIdx.x & 1) * 32;
        float acc = 0.0f;
#pragma unroll 8
        for (int c = 0; c < 32; ++c) acc += __bfloat162float(dos[r * AT_PITCH + c0 + c]) * oc[c];
        acc += __shfl_xor_sync(0xffffffffu, acc, 1);
        if ((threadIdx.x & 1) == 0) dsh[r] = acc;
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, t = lane & 3, g8 = lane >> 2;
    const int row0 = warp * 16;
    float lse[2], dd[2];
    bool rv[2];
#pragma unroll
    for (int h2 = 0; h2 < 2; ++h2) {
        const int r = row0 + g8 + 8 * h2;
        rv[h2] = r < L;
        lse[h2] = lse_s[r];
        dd[h2] = dsh[r];
    }
    float dq[8][4];
    at_zero(dq);
    for (int kb = 0; kb < Lp; kb += AT_BLK) {
        {
            uint32_t fa[4][4];
            float s[8][4], dp[8][4];
            at_zero(s);
            at_zero(dp);
            at_afrag(fa, qs, row0);
            at_mma_abt(s, fa, ks, kb);
            at_afrag(fa, dos, row0);
            at_mma_abt(dp, fa, vs, kb);
#pragma unroll
            for (int nt = 0; nt < 8; ++nt)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int key = kb + nt * 8 + 2 * t + (j & 1);
                    const bool in = key < L && rv[j >> 1];
                    const float p = in ? __expf(s[nt][j] * a.scale - lse[j >> 1]) : 0.0f;
                    s[nt][j] = p;                                      // P
                    dp[nt][j] = in ? p * (dp[nt][j] - dd[j >> 1]) : 0.0f;  // dS
                }
            at_mma_pb(dq, dp, ks, kb);
            at_put(ps, row0, s);
            at_put(dss, row0, dp);
        }
        __syncthreads();
        {
            float acc[8][4];
            at_zero(acc);
            const int key0 = (warp & 3) * 16;  // the warp's 16 keys of the block
            if (warp < 4) {
                at_mma_tb(acc, ps, key0, dos, Lp);   // dV = P^T dO
                at_store(acc, 1.0f, a.dqkv + (long long)g * a.C * ld, ld, kb + key0, L, (2 * H + h) * AT_DK);
            } else {
                at_mma_tb(acc, dss, key0, qs, Lp);   // dK = dS^T Q / sqrt(dk)
                at_store(acc, a.scale, a.dqkv + (long long)g * a.C * ld, ld, kb + key0, L, (H + h) * AT_DK);
            }
        }
        __syncthreads();  // P and dS of this block are read; the next block rewrites them
    }
    at_store(dq, a.scale, a.dqkv + (long long)g * a.C * ld, ld, row0, L, h * AT_DK);
}

size_t at_smem_fwd(int C) {
    const int Cp = (C + AT_BLK - 1) / AT_BLK * AT_BLK;
    return (size_t)(AT_BLK + 2 * Cp) * AT_PITCH * 2;
}
size_t at_smem_dq(int C) {
    const int Cp = (C + AT_BLK - 1) / AT_BLK * AT_BLK;
    return (size_t)(3 * AT_BLK + 2 * Cp) * AT_PITCH * 2 + AT_BLK * 4;
}
size_t at_smem_fused() { return (size_t)6 * AF_ROWS * AT_PITCH * 2 + 2 * (size_t)AF_ROWS * 4; }
size_t at_smem_dkv(int C) {
    const int Cp = (C + AT_BLK - 1) / AT_BLK * AT_BLK;
    return (size_t)(2 * AT_BLK + 2 * Cp) * AT_PITCH * 2 + 2 * (size_t)Cp * 4;
}

template <typename K>
int at_launch(K kern, const AtArgs &a, size_t smem, std::atomic<int> (&limit)[64], std::atomic<int> (&carveout)[64],
              cudaStream_t s, const char *name) {
    if (const int st = raise_smem_limit((const void *)kern, limit, (int)smem)) return st;
    // all of the SM's shared memory for these kernels (set once per device), so
    // that shared memory does not cap the CTAs per SM below the register bound
    int dev = 0;
    if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64 && !carveout[dev].exchange(1))
        cudaFuncSetAttribute((const void *)kern, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
    dim3 grid((a.C + AT_BLK - 1) / AT_BLK, a.H, a.G);
    trace_before(s, name);
    const int st = launch_kernel(kern, grid, dim3(AT_THREADS), smem, s, a);
    trace_after(s);
    return st;
}

}  // namespace

bool attn_core_supported(int C, int head_dim) { return head_dim == AT_DK && C >= 1 && C <= AT_MAX_C; }

int launch_attn_core_fwd(int G, int C, int H, const int32_t *load, const __nv_bfloat16 *qkv,
                         __nv_bfloat16 *o, float *lse, cudaStream_t s) {
    AtArgs a = {};
    a.G = G;
    a.C = C;
    a.H = H;
    a.load = load;
    a.qkv = qkv;
    a.o_out = o;
    a.lse = lse;
    a.scale = 1.0f / sqrtf((float)AT_DK);
    static std::atomic<int> lim[64], carve[64];
    return at_launch(attn_fwd_kernel, a, at_smem_fwd(C), lim, carve, s, "attn_fwd");
}

int launch_attn_core_bwd(int G, int C, int H, const int32_t *load, const __nv_bfloat16 *qkv,
                         const __nv_bfloat16 *o, const float *lse, const __nv_bfloat16 *dout, float *dsum,
                         __nv_bfloat16 *dqkv, cudaStream_t s) {
    AtArgs a = {};
    a.G = G;
    a.C = C;
    a.H = H;
    a.load = load;
    a.qkv = qkv;
    a.o = o;
    a.lse = const_cast<float *>(lse);
    a.dout = dout;
    a.dsum = dsum;
    a.dqkv = dqkv;
    a.scale = 1.0f / sqrtf((float)AT_DK);
    if (C <= AF_ROWS) {  // every group fits one CTA: S, P, dP and dS formed once
        static std::atomic<int> lim_f[64], carve_f[64];
        const size_t smem = at_smem_fused();
        if (const int st = raise_smem_limit((const void *)attn_bwd_fused_kernel, lim_f, (int)smem)) return st;
        int dev = 0;
        if (cudaGetDevice(&dev) == cudaSuccess && dev >= 0 && dev < 64 && !carve_f[dev].exchange(1))
            cudaFuncSetAttribute((const void *)attn_bwd_fused_kernel,
                                 cudaFuncAttributePreferredSharedMemoryCarveout, 100);
        trace_before(s, "attn_bwd");
        const int st = launch_kernel(attn_bwd_fused_kernel, dim3(1, H, G), dim3(AF_THREADS), smem, s, a);
        trace_after(s);
        return st;
    }
    static std::atomic<int> lim_dq[64], lim_dkv[64], carve_dq[64], carve_dkv[64];
    int st = at_launch(attn_bwd_dq_kernel, a, at_smem_dq(C), lim_dq, carve_dq, s, "attn_bwd_dq");
    if (st != VMOE_OK) return st;
    return at_launch(attn_bwd_dkv_kernel, a, at_smem_dkv(C), lim_dkv, carve_dkv, s, "attn_bwd_dkv");
}

}  // namespace vmoe
