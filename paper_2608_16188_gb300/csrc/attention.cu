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
// flash-attention style kernels on mma.sync (m16n8k16, fp32 accumulate; bf16
// operands in the forward, power-of-two-scaled fp16 in most of the backward),
// one CTA per (group, head, block of 64 rows), 4 warps of 16 rows.  Each CTA
// keeps the whole group's keys (or queries) of its head in
// shared memory -- a group holds at most C <= 512 tokens -- so the softmax of a
// row runs online over key blocks of 64 with the row maximum subtracted, and
// the forward saves each row's log-sum-exp for the backward to rebuild P.
// The tiles arrive by cp.async; in the forward and the dQ kernel, one commit
// group per block of 64 keys, so the work on block j overlaps the copies of the
// blocks after it (dK/dV and the fused backward wait for all of theirs: their
// operand scales span every row).  The dQ kernel of groups above 128 tokens
// keeps bf16 operands and takes dS as a bf16 value plus its bf16 residual, two
// products.  In fp16, every query block's CTA would scale the whole of K and V
// (measured at 8 tasks and C 248: 245 us with the residual, against 297 us
// with K and V scaled once all keys have landed, 326 us with each key block
// scaled as it lands, and 206 us for bf16 with a single product).
// Keys (or queries) past the load are masked; rows past it are never stored.
// There are no atomics: dQ is one kernel over query blocks, dK and dV another
// over key blocks, so every sum runs in a fixed order.
#include <cuda_fp16.h>
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

// The backward runs its products on fp16 operands (see the backward's notes
// below); the forward on bf16.  F16 selects the operand type of a product.
template <bool F16>
__device__ __forceinline__ void at_mma(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                       uint32_t b0, uint32_t b1) {
    if constexpr (F16)
        asm volatile(
            "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0, %1, %2, %3}, {%4, %5, %6, %7}, "
            "{%8, %9}, {%0, %1, %2, %3};"
            : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
            : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
    else
        mma_bf16_16816(c, a0, a1, a2, a3, b0, b1);
}
template <bool F16>
__device__ __forceinline__ uint32_t at_pack(float lo, float hi) {
    if constexpr (F16) {
        __half2 h = __floats2half2_rn(lo, hi);
        return *reinterpret_cast<uint32_t *>(&h);
    } else {
        return pack_bf16x2(lo, hi);
    }
}

// A fragments (16 rows x 64 columns, four k16 steps) of a warp's 16 rows of a
// shared tile.
__device__ __forceinline__ void at_afrag(uint32_t (&a)[4][4], const __nv_bfloat16 *tile, int row0) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) at_ldsm_x4(a[ks], tile + (row0 + (lane & 15)) * AT_PITCH + ks * 16 + (lane >> 4) * 8);
}

// acc[NT][4] (16 x 8 NT) += A (16 x 64 via four k16 fragments) * B^T, B = 8 NT
// rows of a shared tile starting at brow: out[i][j] = sum_k A[i][k] B[j][k].
template <bool F16, int NT = 8>
__device__ __forceinline__ void at_mma_abt(float (&acc)[NT][4], const uint32_t (&a)[4][4], const __nv_bfloat16 *tile,
                                           int brow) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int ks = 0; ks < 4; ++ks)
#pragma unroll
        for (int np = 0; np < NT / 2; ++np) {
            uint32_t b[4];
            at_ldsm_x4(b, tile + (brow + np * 16 + (lane & 7) + (lane >> 4) * 8) * AT_PITCH + ks * 16 +
                              ((lane >> 3) & 1) * 8);
            at_mma<F16>(acc[2 * np], a[ks][0], a[ks][1], a[ks][2], a[ks][3], b[0], b[1]);
            at_mma<F16>(acc[2 * np + 1], a[ks][0], a[ks][1], a[ks][2], a[ks][3], b[2], b[3]);
        }
}

// acc[8][4] (16 x 64) += P (16 x 8 NT, fp32 accumulator layout, rounded to the
// operand type) * B, B = 8 NT rows of a shared tile starting at brow (rows = the
// k index).
template <bool F16, int NT = 8>
__device__ __forceinline__ void at_mma_pb(float (&acc)[8][4], const float (&p)[NT][4], const __nv_bfloat16 *tile,
                                          int brow) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int kk = 0; kk < NT / 2; ++kk) {
        const uint32_t a0 = at_pack<F16>(p[2 * kk][0], p[2 * kk][1]);
        const uint32_t a1 = at_pack<F16>(p[2 * kk][2], p[2 * kk][3]);
        const uint32_t a2 = at_pack<F16>(p[2 * kk + 1][0], p[2 * kk + 1][1]);
        const uint32_t a3 = at_pack<F16>(p[2 * kk + 1][2], p[2 * kk + 1][3]);
#pragma unroll
        for (int dp = 0; dp < 4; ++dp) {
            uint32_t b[4];
            const int m = lane >> 3;
            at_ldsm_x4_t(b, tile + (brow + kk * 16 + (m & 1) * 8 + (lane & 7)) * AT_PITCH + dp * 16 + (m >> 1) * 8);
            at_mma<F16>(acc[2 * dp], a0, a1, a2, a3, b[0], b[1]);
            at_mma<F16>(acc[2 * dp + 1], a0, a1, a2, a3, b[2], b[3]);
        }
    }
}

template <int NT>
__device__ __forceinline__ void at_zero(float (&acc)[NT][4]) {
#pragma unroll
    for (int i = 0; i < NT; ++i)
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
        at_mma_abt<false>(s, qa, ks, kb);
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
        at_mma_pb<false>(o, s, vs, kb);
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

// ------------------------------------------------------------------ backward operands
// The fused backward and the dK/dV kernel take fp16 operands, each staged tile
// scaled by its own power of two (the dQ kernel keeps bf16, see the header).  The inputs are bf16 (8 significant bits), so a bf16 value
// times 2^e converts to fp16 (11 bits) exactly while it stays an fp16 normal;
// the products, exact in either type, are then those of the bf16 path.  What
// changes is the two values the kernels round for the second products, P (for
// dV = P^T dO) and dS (for dQ = dS K and dK = dS^T Q): 11 bits instead of 8.
// Rounded to bf16, the two took 12 heads of 64 at C 124 to 0.021 of a group's
// RMS in dK, over the 2e-2 tolerance; in fp16 the backward is at 0.0045, the
// bf16 rounding of its own outputs.
//
// Scale of a tile whose largest magnitude is M = m 2^x (m in [0.5, 1)):
// 2^e, e = 15 - x, so the tile's largest value lands in [2^14, 2^15) and every
// value down to 2^-29 M is an fp16 normal.  e is clamped to [-120, 60]: a tile
// of values all below 2^-45 is scaled by 2^60 only, exact for values down to
// 2^-74.  dS is scaled from a bound, |dS| <= |dP| + |D| <= 64 max|dO| max|V| +
// max|D| (P <= 1, dP a sum of 64 products), fixed per CTA before any dS is
// formed, so that its sums (dQ over key blocks, dK over queries) stay in one
// scale.  Each CTA picks its own scales.  The unscaling folds into the factors
// the bf16 path already applies: S = acc * 2^-(eQ+eK) / sqrt(dk), the scaled
// dS' = P (acc_dP 2^(eS-eO-eV) - D 2^eS), and each result's store; a folded
// factor's exponent is clamped to [-120, 120] (reached only when both of a
// product's tiles exceed 2^75, where the product overflows fp32 anyway).

// Largest |value| of eight bf16 (a 16-byte piece), folded into m (bf16 bits of
// a non-negative value, which order like the values).
__device__ __forceinline__ uint32_t at_absmax8(const uint4 &v, uint32_t m) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) m = max(m, max(w[j] & 0x7fffu, (w[j] >> 16) & 0x7fffu));
    return m;
}
// Eight bf16 times f as eight fp16.
__device__ __forceinline__ uint4 at_to_f16x8(const uint4 &v, float f) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
    uint32_t o[4];
#pragma unroll
    for (int j = 0; j < 4; ++j)
        o[j] = at_pack<true>(__uint_as_float(w[j] << 16) * f, __uint_as_float(w[j] & 0xffff0000u) * f);
    return make_uint4(o[0], o[1], o[2], o[3]);
}

// Largest |value| of rows [0, nrows) x 64 columns of a shared bf16 tile, as
// the bits of a non-negative float.
template <int NT>
__device__ __forceinline__ uint32_t at_tile_absmax(const __nv_bfloat16 *tile, int nrows) {
    uint32_t m = 0;
    for (int i = threadIdx.x; i < nrows * 8; i += NT)
        m = at_absmax8(*reinterpret_cast<const uint4 *>(tile + (i >> 3) * AT_PITCH + (i & 7) * 8), m);
    return m << 16;
}

// Rows [0, nrows) x 64 columns of a shared bf16 tile, times f, as fp16 in place.
template <int NT>
__device__ __forceinline__ void at_tile_to_f16(__nv_bfloat16 *tile, int nrows, float f) {
    for (int i = threadIdx.x; i < nrows * 8; i += NT) {
        uint4 *ptr = reinterpret_cast<uint4 *>(tile + (i >> 3) * AT_PITCH + (i & 7) * 8);
        *ptr = at_to_f16x8(*ptr, f);
    }
}

// The exponent e of a tile's scale from its largest magnitude (float bits).
__device__ __forceinline__ int at_scale_exp(uint32_t mbits) {
    if (mbits == 0) return 0;
    const int biased = (int)(mbits >> 23);           // 0 for a subnormal M, 255 for inf / nan
    const int x = (biased == 0 ? 1 : biased) - 126;  // M < 2^x
    return min(60, max(-120, 15 - x));
}
// 2^e, e clamped to [-120, 120].
__device__ __forceinline__ float at_exp2c(int e) { return __int_as_float((127 + min(120, max(-120, e))) << 23); }

// Block-wide maxima of NQ non-negative float bit patterns (NW warps; red holds
// NQ * NW words).  Ends with a barrier, after which every thread has them.
template <int NQ, int NW>
__device__ __forceinline__ void at_block_max(uint32_t (&v)[NQ], uint32_t *red) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#pragma unroll
    for (int q = 0; q < NQ; ++q) {
        v[q] = __reduce_max_sync(0xffffffffu, v[q]);
        if (lane == 0) red[q * NW + warp] = v[q];
    }
    __syncthreads();
#pragma unroll
    for (int q = 0; q < NQ; ++q) {
        uint32_t m = 0;
#pragma unroll
        for (int w = 0; w < NW; ++w) m = max(m, red[q * NW + w]);
        v[q] = m;
    }
}

// A CTA's scales, from the block maxima {Q, K, V, dO, D} (float bits): the tile
// factors and the folded ones.
struct AtScales {
    float q, k, v, dO;  // the tiles' factors 2^e
    float s;            // S = acc_S * s
    float dp, d;        // dS' = P (acc_dP * dp - D * d)
    float dv, dk, dq;   // the results' store factors (dK and dQ with 1 / sqrt(dk))
};
__device__ __forceinline__ AtScales at_scales(const uint32_t (&m)[5], float scale) {
    const int eq = at_scale_exp(m[0]), ek = at_scale_exp(m[1]), ev = at_scale_exp(m[2]),
              eo = at_scale_exp(m[3]);
    const float bound = 64.0f * __uint_as_float(m[3]) * __uint_as_float(m[2]) + __uint_as_float(m[4]);
    const int es = at_scale_exp(__float_as_uint(bound));
    AtScales sc;
    sc.q = at_exp2c(eq);
    sc.k = at_exp2c(ek);
    sc.v = at_exp2c(ev);
    sc.dO = at_exp2c(eo);
    sc.s = at_exp2c(-(eq + ek)) * scale;
    sc.dp = at_exp2c(es - eo - ev);
    sc.d = at_exp2c(es);
    sc.dv = at_exp2c(-eo);
    sc.dk = at_exp2c(-(es + eq)) * scale;
    sc.dq = at_exp2c(-(es + ek)) * scale;
    return sc;
}

// v - bf16(v), in place: the part of a value its bf16 rounding drops (dS as
// value + residual carries about 16 significant bits into dQ = dS K).
template <int NT>
__device__ __forceinline__ void at_residual(float (&v)[NT][4]) {
#pragma unroll
    for (int i = 0; i < NT; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) v[i][j] -= __bfloat162float(__float2bfloat16_rn(v[i][j]));
}

// ------------------------------------------------------------------ backward: dQ (and D)
// CTA (query block, head, group): D = rowsum(dO * O) of its 64 queries, then
// dQ = sum over key blocks of dS K, dS = P * (dO V^T - D), P = exp(S - lse);
// bf16 operands, dS entering dQ as a bf16 value and its residual.
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
        at_mma_abt<false>(s, qa, ks, kb);
        at_mma_abt<false>(dp, da, vs, kb);
#pragma unroll
        for (int nt = 0; nt < 8; ++nt)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int key = kb + nt * 8 + 2 * t + (j & 1);
                const float p = key < L ? __expf(s[nt][j] * a.scale - lse[j >> 1]) : 0.0f;
                s[nt][j] = p * (dp[nt][j] - dd[j >> 1]);  // dS
            }
        at_mma_pb<false>(dq, s, ks, kb);  // dS as bf16 value
        at_residual(s);
        at_mma_pb<false>(dq, s, ks, kb);  // and its residual
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
    uint32_t *red = reinterpret_cast<uint32_t *>(d_s + Lp);  // [5][4] block maxima
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
    uint32_t dmax = 0;
    for (int i = threadIdx.x; i < Lp; i += AT_THREADS) {
        const bool v = i < L;
        lse_s[i] = v ? __ldg(a.lse + ((long long)g * H + h) * a.C + i) : 0.0f;
        d_s[i] = v ? __ldg(a.dsum + ((long long)g * H + h) * a.C + i) : 0.0f;
        dmax = max(dmax, __float_as_uint(fabsf(d_s[i])));
    }
    at_cp_wait(0);  // every query: the scales of Q and dO span them all
    uint32_t mx[5] = {at_tile_absmax<AT_THREADS>(qs, Lp), at_tile_absmax<AT_THREADS>(ks, AT_BLK),
                      at_tile_absmax<AT_THREADS>(vs, AT_BLK), at_tile_absmax<AT_THREADS>(dos, Lp), dmax};
    at_block_max<5, AT_THREADS / 32>(mx, red);
    const AtScales sc = at_scales(mx, a.scale);
    at_tile_to_f16<AT_THREADS>(qs, Lp, sc.q);
    at_tile_to_f16<AT_THREADS>(ks, AT_BLK, sc.k);
    at_tile_to_f16<AT_THREADS>(vs, AT_BLK, sc.v);
    at_tile_to_f16<AT_THREADS>(dos, Lp, sc.dO);
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, t = lane & 3;
    uint32_t ka[4][4], va[4][4];
    at_afrag(ka, ks, warp * 16);
    at_afrag(va, vs, warp * 16);
    float dk[8][4], dv[8][4];
    at_zero(dk);
    at_zero(dv);
    // query blocks of 32, which holds S^T and dP^T in half the registers
#pragma unroll 1
    for (int qb = 0; qb < Lp; qb += 32) {
        float st[4][4], dpt[4][4];
        at_zero(st);
        at_zero(dpt);
        at_mma_abt<true, 4>(st, ka, qs, qb);   // K Q^T: [16 keys x 32 queries]
        at_mma_abt<true, 4>(dpt, va, dos, qb); // V dO^T
#pragma unroll
        for (int nt = 0; nt < 4; ++nt)
#pragma unroll
            for (int j = 0; j < 4; ++j) {
                const int q = qb + nt * 8 + 2 * t + (j & 1);
                st[nt][j] = q < L ? __expf(st[nt][j] * sc.s - lse_s[q]) : 0.0f;  // P^T
                dpt[nt][j] = st[nt][j] * (dpt[nt][j] * sc.dp - d_s[q] * sc.d);   // dS^T, scaled
            }
        at_mma_pb<true, 4>(dv, st, dos, qb);
        at_mma_pb<true, 4>(dk, dpt, qs, qb);
    }
    __nv_bfloat16 *dst = a.dqkv + (long long)g * a.C * ld;
    at_store(dk, sc.dk, dst, ld, k0 + warp * 16, L, (H + h) * AT_DK);
    at_store(dv, sc.dv, dst, ld, k0 + warp * 16, L, (2 * H + h) * AT_DK);
}

// ------------------------------------------------------------------ backward, groups of <= 128 tokens
// One CTA of 8 warps per (head, group) with L <= 128: S, P, dP and dS are formed
// once for all queries and keys instead of in both kernels above.  Warp w owns
// queries [16 w, 16 w + 16).  Per block of 64 keys: S = Q K^T, dP = dO V^T,
// P = exp(S / sqrt(dk) - lse), dS = P (dP - D) (zero for queries or keys past
// L), dQ += dS K in registers; P and dS (fp16, as the MMAs round them) go to
// shared memory, and warps 0-3 form dV = P^T dO and warps 4-7 dK = dS^T Q for
// the block's 64 keys (16 a warp), summed over the queries in increasing order.
constexpr int AF_THREADS = 256;
constexpr int AF_ROWS = 128;

// acc[8][4] (16 keys x 64) += A^T B: A = 16 key columns (from acol) of a shared
// [query][key] tile, B = a shared [query][64] tile, over queries [0, nq) in
// steps of 16 (A fragments by ldmatrix.trans: A's rows are the tile's columns);
// fp16 operands.
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
            at_mma<true>(acc[2 * dp], a[0], a[1], a[2], a[3], b[0], b[1]);
            at_mma<true>(acc[2 * dp + 1], a[0], a[1], a[2], a[3], b[2], b[3]);
        }
    }
}

// A warp's 16 x 8 NT fp32 tile as fp16 into rows row0.. and columns col0.. of a
// shared [rows][AT_PITCH] tile.
template <int NT>
__device__ __forceinline__ void at_put(__nv_bfloat16 *tile, int row0, int col0, const float (&v)[NT][4]) {
    const int lane = threadIdx.x & 31, g = lane >> 2, t = lane & 3;
#pragma unroll
    for (int h = 0; h < 2; ++h)
#pragma unroll
        for (int nt = 0; nt < NT; ++nt)
            *reinterpret_cast<uint32_t *>(tile + (row0 + g + 8 * h) * AT_PITCH + col0 + nt * 8 + 2 * t) =
                at_pack<true>(v[nt][2 * h], v[nt][2 * h + 1]);
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
    uint32_t *red = reinterpret_cast<uint32_t *>(lse_s + AF_ROWS);  // [5][8] block maxima
    const __nv_bfloat16 *src = a.qkv + (long long)g * a.C * ld;
    const long long ob = (long long)g * a.C * ldo;
    at_cp_rows_n<AF_THREADS>(ps, a.o + ob, ldo, 0, AF_ROWS, L, h * AT_DK);
    at_cp_rows_n<AF_THREADS>(qs, src, ld, 0, AF_ROWS, L, h * AT_DK);
    at_cp_rows_n<AF_THREADS>(dos, a.dout + ob, ldo, 0, AF_ROWS, L, h * AT_DK);
    at_cp_rows_n<AF_THREADS>(ks, src, ld, 0, AF_ROWS, L, (H + h) * AT_DK);
    at_cp_rows_n<AF_THREADS>(vs, src, ld, 0, AF_ROWS, L, (2 * H + h) * AT_DK);
    at_cp_commit();
    for (int i = threadIdx.x; i < AF_ROWS; i += AF_THREADS)
        lse_s[i] = i < L ? __ldg(a.lse + ((long long)g * H + h) * a.C + i) : 0.0f;
    at_cp_wait(0);
    uint32_t mx[5];
    {
        const int r = threadIdx.x >> 1, c0 = (threadIdx.x & 1) * 32;
        float acc = 0.0f;
#pragma unroll 8
        for (int c = 0; c < 32; ++c)
            acc += __bfloat162float(dos[r * AT_PITCH + c0 + c]) * __bfloat162float(ps[r * AT_PITCH + c0 + c]);
        acc += __shfl_xor_sync(0xffffffffu, acc, 1);
        if ((threadIdx.x & 1) == 0) dsh[r] = acc;
        mx[4] = __float_as_uint(fabsf(acc));
    }
    mx[0] = at_tile_absmax<AF_THREADS>(qs, Lp);
    mx[1] = at_tile_absmax<AF_THREADS>(ks, Lp);
    mx[2] = at_tile_absmax<AF_THREADS>(vs, Lp);
    mx[3] = at_tile_absmax<AF_THREADS>(dos, Lp);
    at_block_max<5, AF_THREADS / 32>(mx, red);
    const AtScales sc = at_scales(mx, a.scale);
    at_tile_to_f16<AF_THREADS>(qs, Lp, sc.q);
    at_tile_to_f16<AF_THREADS>(ks, Lp, sc.k);
    at_tile_to_f16<AF_THREADS>(vs, Lp, sc.v);
    at_tile_to_f16<AF_THREADS>(dos, Lp, sc.dO);
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
        dd[h2] = dsh[r] * sc.d;
    }
    float dq[8][4];
    at_zero(dq);
    for (int kb = 0; kb < Lp; kb += AT_BLK) {
        // in two halves of 32 keys, which holds S and dP in half the registers
#pragma unroll 1
        for (int k32 = 0; k32 < AT_BLK; k32 += 32) {
            uint32_t fa[4][4];
            float s[4][4], dp[4][4];
            at_zero(s);
            at_zero(dp);
            at_afrag(fa, qs, row0);
            at_mma_abt<true, 4>(s, fa, ks, kb + k32);
            at_afrag(fa, dos, row0);
            at_mma_abt<true, 4>(dp, fa, vs, kb + k32);
#pragma unroll
            for (int nt = 0; nt < 4; ++nt)
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const int key = kb + k32 + nt * 8 + 2 * t + (j & 1);
                    const bool in = key < L && rv[j >> 1];
                    const float p = in ? __expf(s[nt][j] * sc.s - lse[j >> 1]) : 0.0f;
                    s[nt][j] = p;                                                  // P
                    dp[nt][j] = in ? p * (dp[nt][j] * sc.dp - dd[j >> 1]) : 0.0f;  // dS, scaled
                }
            at_mma_pb<true, 4>(dq, dp, ks, kb + k32);
            at_put<4>(ps, row0, k32, s);
            at_put<4>(dss, row0, k32, dp);
        }
        __syncthreads();
        {
            float acc[8][4];
            at_zero(acc);
            const int key0 = (warp & 3) * 16;  // the warp's 16 keys of the block
            if (warp < 4) {
                at_mma_tb(acc, ps, key0, dos, Lp);   // dV = P^T dO
                at_store(acc, sc.dv, a.dqkv + (long long)g * a.C * ld, ld, kb + key0, L, (2 * H + h) * AT_DK);
            } else {
                at_mma_tb(acc, dss, key0, qs, Lp);   // dK = dS^T Q / sqrt(dk)
                at_store(acc, sc.dk, a.dqkv + (long long)g * a.C * ld, ld, kb + key0, L, (H + h) * AT_DK);
            }
        }
        __syncthreads();  // P and dS of this block are read; the next block rewrites them
    }
    at_store(dq, sc.dq, a.dqkv + (long long)g * a.C * ld, ld, row0, L, h * AT_DK);
}

size_t at_smem_fwd(int C) {
    const int Cp = (C + AT_BLK - 1) / AT_BLK * AT_BLK;
    return (size_t)(AT_BLK + 2 * Cp) * AT_PITCH * 2;
}
size_t at_smem_dq(int C) {
    const int Cp = (C + AT_BLK - 1) / AT_BLK * AT_BLK;
    return (size_t)(3 * AT_BLK + 2 * Cp) * AT_PITCH * 2 + AT_BLK * 4;
}
size_t at_smem_fused() {
    return (size_t)6 * AF_ROWS * AT_PITCH * 2 + 2 * (size_t)AF_ROWS * 4 + 5 * (AF_THREADS / 32) * 4;
}
size_t at_smem_dkv(int C) {
    const int Cp = (C + AT_BLK - 1) / AT_BLK * AT_BLK;
    return (size_t)(2 * AT_BLK + 2 * Cp) * AT_PITCH * 2 + 2 * (size_t)Cp * 4 + 5 * (AT_THREADS / 32) * 4;
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
