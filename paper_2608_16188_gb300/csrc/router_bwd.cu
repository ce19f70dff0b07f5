// router_bwd.cu -- the router backward: the gradient of <dY, y> through the
// gates with the routing (chosen experts, slots) held fixed, which completes
// the adaptation gradient of the gating network (Section 3.1: the visual
// module, router included, is what gets adapted; Section 2.1: gates are a
// softmax of the router logits).
//
//   dgate_j  = <dY[t,n], Ye[t, e_j, s_j]>  for a kept choice, 0 if dropped
//   dlogit   = softmax backward over the k selected logits (renormalised gates)
//              or over all E logits (VMOE_NO_RENORM)
//   dX[t,n] += W_r[t] dlogit[t,n]
//   dW_r[t]  = x[t]^T dlogit[t],  dbias[t] = sum_n dlogit[t,n]
//
// Kernel 1 (router_grad): one warp per token.  The dot products stream dY and
// the k expert-output rows with 16-byte vectors and a fixed butterfly
// reduction; the dX update reads W_r[t] transposed from shared memory, staged
// once per task segment of a persistent CTA.  With renormalised gates dlogit
// has k non-zeros, so the update is k scaled columns of W_r, not an E-term
// contraction.
//
// Kernel 2 (router_dw), bf16 problems: dW_r = x^T dlogit on the tensor cores,
// tcgen05 for E = 32 or 64 and d a multiple of 128 (router_dw_tc.cu), else the
// mma.sync kernel below.  x is exact in bf16; dlogit (fp32) is split into three
// bf16 parts while it is staged, so every partial product is exact in fp32 and
// the MMAs accumulate in fp32.  The token (reduction) dimension is split over
// the CTAs of a thread-block cluster and the partial tiles are summed through
// distributed shared memory in rank order, so the result is deterministic.
// fp32 problems use a CUDA-core tile kernel instead.  No atomics anywhere.
#include <cooperative_groups.h>
#include <math.h>

#include <algorithm>

#include "common.cuh"

namespace cg = cooperative_groups;

namespace vmoe {

int launch_router_dw_tc(const Dims &p, const __nv_bfloat16 *x, const float *dl, float *dw, float *dbias,
                        cudaStream_t s);  // router_dw_tc.cu

namespace {

// ---------------------------------------------------------------------------
// Vector helpers: 8 consecutive elements as floats.
template <typename T>
__device__ __forceinline__ void load8(const T *p, float *o);  // read-only data
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
__device__ __forceinline__ void load8_rw(const T *p, float *o);  // data this kernel writes
template <>
__device__ __forceinline__ void load8_rw<__nv_bfloat16>(const __nv_bfloat16 *p, float *o) {
    bf16x8_to_f32(*reinterpret_cast<const uint4 *>(p), o);
}
template <>
__device__ __forceinline__ void load8_rw<float>(const float *p, float *o) {
    const float4 a = reinterpret_cast<const float4 *>(p)[0];
    const float4 b = reinterpret_cast<const float4 *>(p)[1];
    o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
    o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
}

template <typename T>
__device__ __forceinline__ void store8(T *p, const float *v);
template <>
__device__ __forceinline__ void store8<__nv_bfloat16>(__nv_bfloat16 *p, const float *v) {
    *reinterpret_cast<uint4 *>(p) = f32_to_bf16x8(v);
}
template <>
__device__ __forceinline__ void store8<float>(float *p, const float *v) {
    reinterpret_cast<float4 *>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4 *>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
}

// ---------------------------------------------------------------------------
// Kernel 1: dgate, dlogits and the dX update, one warp per token.
constexpr int RG_THREADS = 512;
constexpr int RG_WARPS = RG_THREADS / 32;
constexpr int RG_UNROLL = 2;
constexpr size_t RG_SMEM_CAP = 200 * 1024;

// Shared memory: per-warp dlogit rows (VMOE_NO_RENORM), then W_r[t]^T, one row
// per expert with pitch wt_pitch(d) floats.  Within each block of 256 columns the
// columns are permuted so that the 8 columns 8L..8L+7 a lane reads sit at 4L..4L+3
// and 128+4L..128+4L+3: the lanes of a warp then read two runs of consecutive
// 16-byte words, free of bank conflicts.
__host__ __device__ inline int wt_pitch(int d) { return ((d + 255) & ~255) + 4; }
__device__ __forceinline__ int wt_col(int i) {  // physical position of column i
    const int w = i & 255, q = w & 7;
    return (i & ~255) + ((w >> 3) << 2) + (q < 4 ? q : 124 + q);
}
__device__ __forceinline__ int wt_col8(int v) {  // first half of columns v..v+7, v % 8 == 0
    return (v & ~255) + ((v & 255) >> 1);
}
inline size_t rg_smem_rows(const Dims &p) {
    return (p.flags & VMOE_NO_RENORM) ? (size_t)RG_WARPS * p.E * sizeof(float) : 0;
}
inline size_t rg_smem_w(const Dims &p) { return (size_t)p.E * wt_pitch(p.d) * sizeof(float); }

// W_r[t] ([d][E], fp32) into shared memory as W^T with row pitch dp.  Kept out
// of line so its load batch does not raise the token loop's register count.
__device__ __noinline__ void stage_wt(const float *__restrict__ wrt, float *WT, int d, int E,
                                      int dp) {
    if ((E & 7) == 0) {
        // thread = one row i, 8 experts at a time: one 32-byte sector per load
        // pair, consecutive i across a warp (conflict-free transposing stores)
        const int E8 = E >> 3;
        for (int i = threadIdx.x; i < d; i += RG_THREADS) {
            const float4 *src = reinterpret_cast<const float4 *>(wrt + (long long)i * E);
            for (int e8 = 0; e8 < E8; e8 += RG_UNROLL) {
                float4 buf[RG_UNROLL][2];
#pragma unroll
                for (int u = 0; u < RG_UNROLL; ++u)
                    if (e8 + u < E8) {
                        buf[u][0] = __ldg(src + 2 * (e8 + u));
                        buf[u][1] = __ldg(src + 2 * (e8 + u) + 1);
                    }
#pragma unroll
                for (int u = 0; u < RG_UNROLL; ++u)
                    if (e8 + u < E8) {
                        float *col = WT + (8 * (e8 + u)) * dp + wt_col(i);
                        col[0 * dp] = buf[u][0].x;
                        col[1 * dp] = buf[u][0].y;
                        col[2 * dp] = buf[u][0].z;
                        col[3 * dp] = buf[u][0].w;
                        col[4 * dp] = buf[u][1].x;
                        col[5 * dp] = buf[u][1].y;
                        col[6 * dp] = buf[u][1].z;
                        col[7 * dp] = buf[u][1].w;
                    }
            }
        }
    } else {
        for (int i = threadIdx.x; i < d; i += RG_THREADS)
            for (int e = 0; e < E; ++e) WT[e * dp + wt_col(i)] = __ldg(wrt + (long long)i * E + e);
    }
}

// Per-token steps shared by both forms of kernel 1.
//
// gate_backward: reduces the lane partials of dgate_j (fixed butterfly), writes
// dgate and the dlogit row, and returns in c[j] the dlogit of expert e_j
// (renormalised gates; VMOE_NO_RENORM leaves the dense row in dlrow).  Returns
// whether the dX update has any non-zero term.
template <int KMAX>
__device__ __forceinline__ bool gate_backward(int k, int E, bool norenorm, int lane, long long tn,
                                              float (&dg)[KMAX], const float (&gt)[KMAX],
                                              const int (&ei)[KMAX], const float *logits,
                                              float *dgate, float *dlogits, float *dlrow,
                                              float (&c)[KMAX]) {
    float s = 0.0f;
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
        if (j >= k) continue;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) dg[j] += __shfl_xor_sync(0xffffffffu, dg[j], o);
        s = fmaf(gt[j], dg[j], s);
    }
    {
        float mine = 0.0f;
#pragma unroll
        for (int j = 0; j < KMAX; ++j)
            if (j == lane) mine = dg[j];
        if (lane < k) dgate[tn * k + lane] = mine;
    }
    float *dl = dlogits + tn * E;
    bool any = false;
#pragma unroll
    for (int j = 0; j < KMAX; ++j) {
        c[j] = j < k ? gt[j] * (dg[j] - s) : 0.0f;
        any |= c[j] != 0.0f;
    }
    if (!norenorm) {
        for (int e = lane; e < E; e += 32) {
            float v = 0.0f;
#pragma unroll
            for (int j = 0; j < KMAX; ++j)
                if (j < k && ei[j] == e) v = c[j];
            dl[e] = v;
        }
        return any;
    }
    const float *l = logits + tn * E;
    float mx = -INFINITY;
    for (int e = lane; e < E; e += 32) mx = fmaxf(mx, __ldg(l + e));
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float sum = 0.0f;
    for (int e = lane; e < E; e += 32) sum += expf(__ldg(l + e) - mx);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    for (int e = lane; e < E; e += 32) {
        float g = 0.0f;
#pragma unroll
        for (int j = 0; j < KMAX; ++j)
            if (j < k && ei[j] == e) g = dg[j];
        const float v = expf(__ldg(l + e) - mx) / sum * (g - s);
        dl[e] = v;
        dlrow[e] = v;
    }
    __syncwarp();
    return true;
}

// dx_terms: r[0..7] = sum over the dX terms of dlogit_e * W_r[v + q][e] for the
// 8 columns v..v+7: the k chosen experts (renormalised gates) or all E.
template <int KMAX, bool WSMEM>
__device__ __forceinline__ void dx_terms(float (&r)[8], int v, int ne, bool norenorm,
                                         const float *dlrow, const int (&ei)[KMAX],
                                         const float (&c)[KMAX], const float *WT, int dp,
                                         const float *wrt, int E) {
#pragma unroll
    for (int q = 0; q < 8; ++q) r[q] = 0.0f;
    for (int jj = 0; jj < ne; ++jj) {
        int e = jj;
        float cj = 0.0f;
        if (norenorm) {
            cj = dlrow[jj];
        } else {
#pragma unroll
            for (int j = 0; j < KMAX; ++j)
                if (j == jj) {
                    e = ei[j];
                    cj = c[j];
                }
        }
        float w[8];
        if (WSMEM) {
            const float *wp = WT + e * dp + wt_col8(v);
            const float4 a = *reinterpret_cast<const float4 *>(wp);
            const float4 b = *reinterpret_cast<const float4 *>(wp + 128);
            w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w;
            w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
        } else {
#pragma unroll
            for (int q = 0; q < 8; ++q) w[q] = __ldg(wrt + (long long)(v + q) * E + e);
        }
#pragma unroll
        for (int q = 0; q < 8; ++q) r[q] = fmaf(cj, w[q], r[q]);
    }
}

// Generic form (any dtype, k, d).  Persistent: CTA b takes tokens
// [TN b / grid, TN (b + 1) / grid) of the task-major token order, in task
// segments; W_r[t]^T is staged per segment.
template <typename T, int KMAX, bool WSMEM>
__global__ void __launch_bounds__(RG_THREADS, KMAX <= 2 ? 2 : 1)
router_grad_kernel(Dims p, const T *__restrict__ dy, const T *__restrict__ ye,
                   const float *__restrict__ logits, const int32_t *__restrict__ idx,
                   const float *__restrict__ gate, const int32_t *__restrict__ slot,
                   const float *__restrict__ wr, float *__restrict__ dgate,
                   float *__restrict__ dlogits, T *dx) {
    extern __shared__ __align__(16) float rg_smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int d = p.d, E = p.E, k = p.k, N = p.N;
    const bool norenorm = (p.flags & VMOE_NO_RENORM) != 0;
    const int dp = wt_pitch(d);
    float *dlrow = rg_smem + warp * E;
    float *WT = rg_smem + (norenorm ? RG_WARPS * E : 0);
    const long long TN = (long long)p.T * N;
    const long long beg = TN * blockIdx.x / gridDim.x;
    const long long end = TN * (blockIdx.x + 1) / gridDim.x;
    for (long long seg = beg; seg < end;) {
        const int t = (int)(seg / N);
        const long long seg_end = min(end, (long long)(t + 1) * N);
        const float *wrt = wr + (long long)t * d * E;
        if (WSMEM) {
            __syncthreads();  // the previous segment's readers are done
            stage_wt(wrt, WT, d, E, dp);
            __syncthreads();
        }
        for (long long tn = seg + warp; tn < seg_end; tn += RG_WARPS) {
            const T *dyr = dy + tn * d;
            int ei[KMAX], sl[KMAX];
            float gt[KMAX], dg[KMAX];
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                ei[j] = 0;
                sl[j] = -1;
                gt[j] = 0.0f;
                dg[j] = 0.0f;
                if (j < k) {
                    ei[j] = __ldg(idx + tn * k + j);
                    sl[j] = __ldg(slot + tn * k + j);
                    gt[j] = __ldg(gate + tn * k + j);
                }
            }
            // dgate_j = <dY, Ye[e_j, s_j]>: per-lane fp32 partial sums
            for (int v = lane * 8; v < d; v += 256) {
                float fa[8];
                load8<T>(dyr + v, fa);
#pragma unroll
                for (int j = 0; j < KMAX; ++j) {
                    if (sl[j] < 0) continue;
                    float fb[8];
                    load8<T>(ye + (((long long)t * E + ei[j]) * p.C + sl[j]) * d + v, fb);
#pragma unroll
                    for (int q = 0; q < 8; ++q) dg[j] = fmaf(fa[q], fb[q], dg[j]);
                }
            }
            float c[KMAX];
            const bool any = gate_backward<KMAX>(k, E, norenorm, lane, tn, dg, gt, ei, logits,
                                                 dgate, dlogits, dlrow, c);
            // dX += W_r dlogit, summed in fp32 and added to dX with one rounding
            if (dx != nullptr && any) {
                T *xr = dx + tn * d;
                const int ne = norenorm ? E : k;
                for (int v = lane * 8; v < d; v += 256) {
                    float r[8], o[8];
                    dx_terms<KMAX, WSMEM>(r, v, ne, norenorm, dlrow, ei, c, WT, dp, wrt, E);
                    load8_rw<T>(xr + v, o);
#pragma unroll
                    for (int q = 0; q < 8; ++q) o[q] += r[q];
                    store8<T>(xr + v, o);
                }
            }
            if (norenorm) __syncwarp();  // dlrow is rewritten by the next token
        }
        seg = seg_end;
    }
}

// Fast form: bf16, k <= 2, d <= 256 NCH.  One CTA per SM with up to 128
// registers a thread, so every load of a token -- the dY row, its k expert-output
// rows and its dX row -- is in flight at once (one memory round trip per token),
// and the next token's routing is fetched while this one is reduced.
template <int NCH, int KMAX, bool WSMEM>
__global__ void __launch_bounds__(RG_THREADS, 1)
router_grad_fast_kernel(Dims p, const __nv_bfloat16 *__restrict__ dy,
                        const __nv_bfloat16 *__restrict__ ye, const float *__restrict__ logits,
                        const int32_t *__restrict__ idx, const float *__restrict__ gate,
                        const int32_t *__restrict__ slot, const float *__restrict__ wr,
                        float *__restrict__ dgate, float *__restrict__ dlogits,
                        __nv_bfloat16 *dx) {
    extern __shared__ __align__(16) float rg_smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int d = p.d, E = p.E, k = p.k, N = p.N;
    const bool norenorm = (p.flags & VMOE_NO_RENORM) != 0;
    const int dp = wt_pitch(d);
    float *dlrow = rg_smem + warp * E;
    float *WT = rg_smem + (norenorm ? RG_WARPS * E : 0);
    const long long TN = (long long)p.T * N;
    const long long beg = TN * blockIdx.x / gridDim.x;
    const long long end = TN * (blockIdx.x + 1) / gridDim.x;
    for (long long seg = beg; seg < end;) {
        const int t = (int)(seg / N);
        const long long seg_end = min(end, (long long)(t + 1) * N);
        const float *wrt = wr + (long long)t * d * E;
        if (WSMEM) {
            __syncthreads();
            stage_wt(wrt, WT, d, E, dp);
            __syncthreads();
        }
        const __nv_bfloat16 *yet = ye + (long long)t * E * p.C * d;
        long long tn = seg + warp;
        int ei[KMAX], sl[KMAX];
        float gt[KMAX];
#pragma unroll
        for (int j = 0; j < KMAX; ++j) {
            ei[j] = 0;
            sl[j] = -1;
            gt[j] = 0.0f;
            if (tn < seg_end && j < k) {
                ei[j] = __ldg(idx + tn * k + j);
                sl[j] = __ldg(slot + tn * k + j);
                gt[j] = __ldg(gate + tn * k + j);
            }
        }
        for (; tn < seg_end; tn += RG_WARPS) {
            uint4 a[NCH], b[KMAX][NCH], xo[NCH];
#pragma unroll
            for (int ch = 0; ch < NCH; ++ch) {
                const int v = lane * 8 + 256 * ch;
                if (v < d) a[ch] = __ldg(reinterpret_cast<const uint4 *>(dy + tn * d + v));
            }
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                if (sl[j] < 0) continue;
                const __nv_bfloat16 *row = yet + ((long long)ei[j] * p.C + sl[j]) * d;
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch) {
                    const int v = lane * 8 + 256 * ch;
                    if (v < d) b[j][ch] = __ldg(reinterpret_cast<const uint4 *>(row + v));
                }
            }
            if (dx != nullptr) {
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch) {
                    const int v = lane * 8 + 256 * ch;
                    if (v < d) xo[ch] = *reinterpret_cast<const uint4 *>(dx + tn * d + v);
                }
            }
            // the next token's routing
            const long long tn2 = tn + RG_WARPS;
            int ei2[KMAX], sl2[KMAX];
            float gt2[KMAX];
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                ei2[j] = 0;
                sl2[j] = -1;
                gt2[j] = 0.0f;
                if (tn2 < seg_end && j < k) {
                    ei2[j] = __ldg(idx + tn2 * k + j);
                    sl2[j] = __ldg(slot + tn2 * k + j);
                    gt2[j] = __ldg(gate + tn2 * k + j);
                }
            }
            float dg[KMAX];
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                dg[j] = 0.0f;
                if (sl[j] < 0) continue;
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch) {
                    if (lane * 8 + 256 * ch >= d) continue;
                    float fa[8], fb[8];
                    bf16x8_to_f32(a[ch], fa);
                    bf16x8_to_f32(b[j][ch], fb);
#pragma unroll
                    for (int q = 0; q < 8; ++q) dg[j] = fmaf(fa[q], fb[q], dg[j]);
                }
            }
            float c[KMAX];
            const bool any = gate_backward<KMAX>(k, E, norenorm, lane, tn, dg, gt, ei, logits,
                                                 dgate, dlogits, dlrow, c);
            if (dx != nullptr && any) {
                const int ne = norenorm ? E : k;
#pragma unroll
                for (int ch = 0; ch < NCH; ++ch) {
                    const int v = lane * 8 + 256 * ch;
                    if (v >= d) continue;
                    float r[8], o[8];
                    dx_terms<KMAX, WSMEM>(r, v, ne, norenorm, dlrow, ei, c, WT, dp, wrt, E);
                    bf16x8_to_f32(xo[ch], o);
#pragma unroll
                    for (int q = 0; q < 8; ++q) o[q] += r[q];
                    *reinterpret_cast<uint4 *>(dx + tn * d + v) = f32_to_bf16x8(o);
                }
            }
            if (norenorm) __syncwarp();
#pragma unroll
            for (int j = 0; j < KMAX; ++j) {
                ei[j] = ei2[j];
                sl[j] = sl2[j];
                gt[j] = gt2[j];
            }
        }
        seg = seg_end;
    }
}

// ---------------------------------------------------------------------------
// Kernel 2 (bf16): dW_r = x^T dlogit and dbias on the tensor cores.
constexpr int DW_MT = 2;            // m16 tiles (of d rows) per warp
constexpr int DW_WARPS = 4;         // DW_WARPS x DW_MT x 16 = DW_BD rows
constexpr int DW_THREADS = 32 * DW_WARPS;
constexpr int DW_BD = 128;          // rows of d per CTA
constexpr int DW_BE = 32;           // experts per CTA
constexpr int DW_KC = 32;           // tokens per stage
constexpr int DW_STAGES = 3;
constexpr int DW_SPLIT = 4;         // cluster size: the token range is split 4 ways
constexpr int DW_XP = DW_BD + 8;    // x row pitch (bf16): 272 B, conflict-free ldmatrix
constexpr int DW_PP = DW_KC + 8;    // dlogit-part row pitch (bf16): 80 B, conflict-free
constexpr int DW_RP = DW_BE + 1;    // fp32 partial-tile row pitch

struct DwSmem {
    __nv_bfloat16 x[DW_STAGES][DW_KC][DW_XP];     // token rows of the d-slice
    float dl[DW_STAGES][DW_KC][DW_BE];            // dlogit rows as loaded (fp32)
    __nv_bfloat16 part[3][DW_BE][DW_PP];          // their three bf16 parts, expert-major
    float bias[DW_WARPS][DW_BE];
    float bias_sum[DW_BE];
};
static_assert(sizeof(DwSmem) <= 48 * 1024, "static shared memory");
static_assert(DW_WARPS * DW_MT * 16 == DW_BD, "warp tiling of the d-slice");
static_assert(DW_BD * DW_RP * sizeof(float) <= sizeof(DwSmem::x), "partial tile reuses x");

__device__ __forceinline__ void cp_async16(void *smem, const void *gmem, bool valid) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
    const int n = valid ? 16 : 0;  // 0 source bytes: the 16 bytes are zero-filled
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async4(void *smem, const void *gmem, bool valid) {
    const uint32_t s = (uint32_t)__cvta_generic_to_shared(smem);
    const int n = valid ? 4 : 0;
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;\n" ::"r"(s), "l"(gmem), "r"(n));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N)); }

__device__ __forceinline__ void ldsm_x4(uint32_t (&r)[4], const void *smem) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(a));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t (&r)[4], const void *smem) {
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(smem);
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];\n"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]) : "r"(a));
}

// grid (DW_SPLIT, ceil(d / DW_BD), T * ceil(E / DW_BE)), cluster (DW_SPLIT, 1, 1).
// Warp w owns rows [32 w, 32 w + 32) of the CTA's d-slice (two m16 tiles, so
// each dlogit fragment read from shared memory feeds two products) and all 32
// experts.
__global__ void __cluster_dims__(DW_SPLIT, 1, 1) __launch_bounds__(DW_THREADS)
router_dw_mma_kernel(Dims p, const __nv_bfloat16 *__restrict__ x,
                     const float *__restrict__ dlg, float *__restrict__ dw,
                     float *__restrict__ dbias) {
    __shared__ __align__(128) DwSmem sm;
    cg::cluster_group cluster = cg::this_cluster();
    const int rank = (int)cluster.block_rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int d = p.d, E = p.E, N = p.N;
    const int etiles = (E + DW_BE - 1) / DW_BE;
    const int t = blockIdx.z / etiles;
    const int e0 = (blockIdx.z - t * etiles) * DW_BE;
    const int d0 = blockIdx.y * DW_BD;
    const int n_beg = (int)((long long)N * rank / DW_SPLIT);
    const int n_end = (int)((long long)N * (rank + 1) / DW_SPLIT);
    const int nchunks = (n_end - n_beg + DW_KC - 1) / DW_KC;
    const __nv_bfloat16 *xt = x + (long long)t * N * d;
    const float *dlt = dlg + (long long)t * N * E;
    const bool do_bias = dbias != nullptr && blockIdx.y == 0;

    auto load_x = [&](int chunk, int stage) {
        // 32 token rows x 16 vectors of 8 bf16
#pragma unroll
        for (int u = 0; u < DW_KC * 16 / DW_THREADS; ++u) {
            const int v = tid + u * DW_THREADS;
            const int r = v >> 4, cv = (v & 15) * 8;
            const int n = n_beg + chunk * DW_KC + r;
            const bool ok = n < n_end && d0 + cv < d;
            const __nv_bfloat16 *src = ok ? xt + (long long)n * d + d0 + cv : xt;
            cp_async16(&sm.x[stage][r][cv], src, ok);
        }
    };
    // dlogit rows of a chunk: 32 tokens x 32 experts, 16-byte copies when E % 4 == 0
    const bool vec_dl = (E & 3) == 0;
    auto load_dl = [&](int chunk, int stage) {
        if (vec_dl) {
#pragma unroll
            for (int u = 0; u < DW_KC * 8 / DW_THREADS; ++u) {
                const int v = tid + u * DW_THREADS;
                const int r = v >> 3, c4 = (v & 7) * 4;
                const int n = n_beg + chunk * DW_KC + r;
                const bool ok = n < n_end && e0 + c4 < E;
                cp_async16(&sm.dl[stage][r][c4], ok ? dlt + (long long)n * E + e0 + c4 : dlt, ok);
            }
        } else {
#pragma unroll
            for (int u = 0; u < DW_KC * DW_BE / DW_THREADS; ++u) {
                const int v = tid + u * DW_THREADS;
                const int r = v >> 5, c = v & 31;
                const int n = n_beg + chunk * DW_KC + r;
                const bool ok = n < n_end && e0 + c < E;
                cp_async4(&sm.dl[stage][r][c], ok ? dlt + (long long)n * E + e0 + c : dlt, ok);
            }
        }
    };
    // the split: warp w takes token rows [8 w, 8 w + 8) of the chunk, lane = expert
    // column, so each part of a lane's 8 tokens is one 16-byte shared store
    // (rows 80 bytes apart: the 8 lanes of a quarter-warp hit distinct banks)
    static_assert(DW_KC == 8 * DW_WARPS, "one 8-token row group per warp");
    const int pc = lane;
    float bias_acc = 0.0f;

    float acc[DW_MT][4][4];
#pragma unroll
    for (int mt = 0; mt < DW_MT; ++mt)
#pragma unroll
        for (int a = 0; a < 4; ++a)
#pragma unroll
            for (int b = 0; b < 4; ++b) acc[mt][a][b] = 0.0f;

    // prologue: chunks 0 .. STAGES-2
#pragma unroll
    for (int st = 0; st < DW_STAGES - 1; ++st) {
        if (st < nchunks) {
            load_x(st, st);
            load_dl(st, st);
        }
        cp_async_commit();
    }
    for (int ch = 0; ch < nchunks; ++ch) {
        const int stage = ch % DW_STAGES;
        cp_async_wait<DW_STAGES - 2>();  // this thread's copies of chunk ch have landed
        __syncthreads();  // everyone's copies of chunk ch visible; iteration ch - 1 finished
        {
            const int nx = ch + DW_STAGES - 1;  // refills the stage iteration ch - 1 read
            if (nx < nchunks) {
                load_x(nx, nx % DW_STAGES);
                load_dl(nx, nx % DW_STAGES);
            }
            cp_async_commit();
        }
        {
            uint32_t ph[4], pm[4], pl[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const float v0 = sm.dl[stage][8 * warp + 2 * u][pc];
                const float v1 = sm.dl[stage][8 * warp + 2 * u + 1][pc];
                __nv_bfloat16 h0, m0, l0, h1, m1, l1;
                split3(v0, h0, m0, l0);
                split3(v1, h1, m1, l1);
                ph[u] = pack2(h0, h1);
                pm[u] = pack2(m0, m1);
                pl[u] = pack2(l0, l1);
                bias_acc += v0;
                bias_acc += v1;
            }
            *reinterpret_cast<uint4 *>(&sm.part[0][pc][8 * warp]) = make_uint4(ph[0], ph[1], ph[2], ph[3]);
            *reinterpret_cast<uint4 *>(&sm.part[1][pc][8 * warp]) = make_uint4(pm[0], pm[1], pm[2], pm[3]);
            *reinterpret_cast<uint4 *>(&sm.part[2][pc][8 * warp]) = make_uint4(pl[0], pl[1], pl[2], pl[3]);
        }
        __syncthreads();  // parts visible
        // two-level sum: this chunk's products, then into the running total
        float cacc[DW_MT][4][4];
#pragma unroll
        for (int mt = 0; mt < DW_MT; ++mt)
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) cacc[mt][a][b] = 0.0f;
#pragma unroll
        for (int ks = 0; ks < DW_KC; ks += 16) {
            const int mi = lane >> 3, r = lane & 7;
            uint32_t a[DW_MT][4];
#pragma unroll
            for (int mt = 0; mt < DW_MT; ++mt)
                ldsm_x4_t(a[mt], &sm.x[stage][ks + (mi >> 1) * 8 + r]
                                     [(warp * DW_MT + mt) * 16 + (mi & 1) * 8]);
#pragma unroll
            for (int part = 0; part < 3; ++part) {
#pragma unroll
                for (int np = 0; np < 2; ++np) {
                    uint32_t b[4];
                    ldsm_x4(b, &sm.part[part][np * 16 + (mi >> 1) * 8 + r][ks + (mi & 1) * 8]);
#pragma unroll
                    for (int mt = 0; mt < DW_MT; ++mt) {
                        mma_bf16_16816(cacc[mt][2 * np], a[mt][0], a[mt][1], a[mt][2], a[mt][3],
                                       b[0], b[1]);
                        mma_bf16_16816(cacc[mt][2 * np + 1], a[mt][0], a[mt][1], a[mt][2],
                                       a[mt][3], b[2], b[3]);
                    }
                }
            }
        }
#pragma unroll
        for (int mt = 0; mt < DW_MT; ++mt)
#pragma unroll
            for (int a = 0; a < 4; ++a)
#pragma unroll
                for (int b = 0; b < 4; ++b) acc[mt][a][b] += cacc[mt][a][b];
    }
    cp_async_wait<0>();
    __syncthreads();

    // partial tile into shared memory (reusing the x stages), then the cluster sum
    float *red = reinterpret_cast<float *>(&sm.x[0][0][0]);
    {
        const int g = lane >> 2, q = lane & 3;
#pragma unroll
        for (int mt = 0; mt < DW_MT; ++mt)
#pragma unroll
            for (int nt = 0; nt < 4; ++nt) {
                const int m = (warp * DW_MT + mt) * 16 + g, n = nt * 8 + 2 * q;
                red[m * DW_RP + n] = acc[mt][nt][0];
                red[m * DW_RP + n + 1] = acc[mt][nt][1];
                red[(m + 8) * DW_RP + n] = acc[mt][nt][2];
                red[(m + 8) * DW_RP + n + 1] = acc[mt][nt][3];
            }
    }
    if (do_bias) sm.bias[warp][pc] = bias_acc;  // warp w's tokens 8w..8w+7 of every chunk
    __syncthreads();
    if (do_bias && tid < DW_BE) {
        float b = 0.0f;
#pragma unroll
        for (int w = 0; w < DW_WARPS; ++w) b += sm.bias[w][tid];
        sm.bias_sum[tid] = b;
    }
    cluster.sync();
    // rank r writes rows [32 r, 32 r + 32) of the tile, summing ranks 0..3 in order
    float *dwt = dw + (long long)t * d * E;
    constexpr int ROWS = DW_BD / DW_SPLIT;
    for (int v = tid; v < ROWS * DW_BE; v += DW_THREADS) {
        const int m = rank * ROWS + v / DW_BE, n = v % DW_BE;
        float sum = 0.0f;
#pragma unroll
        for (int q = 0; q < DW_SPLIT; ++q) sum += cluster.map_shared_rank(red, q)[m * DW_RP + n];
        if (d0 + m < d && e0 + n < E) dwt[(long long)(d0 + m) * E + e0 + n] = sum;
    }
    if (do_bias && rank == 0 && tid < DW_BE && e0 + tid < E) {
        float b = 0.0f;
#pragma unroll
        for (int q = 0; q < DW_SPLIT; ++q) b += cluster.map_shared_rank(sm.bias_sum, q)[tid];
        dbias[(long long)t * E + e0 + tid] = b;
    }
    cluster.sync();  // every rank's shared memory stays alive until the remote reads are done
}

// ---------------------------------------------------------------------------
// Kernel 2 (fp32 problems): the same product on CUDA cores, 64 x 64 tiles,
// 4 x 4 accumulators per thread, a two-level sum over tokens (per chunk of 32,
// then across chunks: rounding error grows with sqrt(32) + sqrt(N / 32)).
constexpr int RT = 64;
constexpr int RKC = 32;
constexpr int RD_THREADS = 256;

__global__ void __launch_bounds__(RD_THREADS)
router_dw_simt_kernel(Dims p, const float *__restrict__ x, const float *__restrict__ dl,
                      float *__restrict__ dw, float *__restrict__ dbias) {
    __shared__ __align__(16) float xs[RKC][RT];
    __shared__ __align__(16) float ds[RKC][RT];
    const int t = blockIdx.z, i0 = blockIdx.x * RT, e0 = blockIdx.y * RT;
    const int tid = threadIdx.x, ti = tid / 16, tj = tid % 16;
    const int d = p.d, E = p.E, N = p.N;
    const float *xt = x + (long long)t * N * d;
    const float *dlt = dl + (long long)t * N * E;
    float acc[4][4] = {};
    float bacc = 0.0f;
    const bool do_bias = dbias != nullptr && blockIdx.x == 0 && tid < RT && e0 + tid < E;
    for (int n0 = 0; n0 < N; n0 += RKC) {
        for (int i = tid; i < RKC * RT; i += RD_THREADS) {
            const int r = i / RT, c = i % RT;
            const int n = n0 + r;
            xs[r][c] = (n < N && i0 + c < d) ? xt[(long long)n * d + i0 + c] : 0.0f;
            ds[r][c] = (n < N && e0 + c < E) ? dlt[(long long)n * E + e0 + c] : 0.0f;
        }
        __syncthreads();
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

// ---------------------------------------------------------------------------
template <typename T, int KMAX, bool WSMEM>
int launch_grad(const Dims &p, const float *wr, const float *logits, const int32_t *idx,
                const float *gate, const int32_t *slot, const T *dy, const T *ye, float *dgate,
                float *dlogits, T *dx, size_t smem, cudaStream_t s) {
    auto kern = router_grad_kernel<T, KMAX, WSMEM>;
    // attribute and occupancy per (device, shared-memory size)
    static std::atomic<int> smem_limit[64];
    static std::atomic<uint64_t> occupancy[64];  // per device: (smem << 32) | CTAs per SM
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return VMOE_ERR_CUDA;
    if (smem > 48 * 1024)
        if (const int st = raise_smem_limit((const void *)kern, smem_limit, (int)smem)) return st;
    const uint64_t o = occupancy[dev].load(std::memory_order_relaxed);
    int per_sm = (int)(o & 0xffffffffu);
    if (per_sm < 1 || (o >> 32) != (uint64_t)smem) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, RG_THREADS, smem) !=
                cudaSuccess ||
            per_sm < 1)
            return VMOE_ERR_CUDA;
        occupancy[dev].store(((uint64_t)smem << 32) | (uint32_t)per_sm, std::memory_order_relaxed);
    }
    const long long tokens = (long long)p.T * p.N;
    long long grid = (long long)per_sm * num_sms();
    grid = std::min(grid, (tokens + RG_WARPS - 1) / RG_WARPS);
    kern<<<(unsigned)grid, RG_THREADS, smem, s>>>(p, dy, ye, logits, idx, gate, slot, wr, dgate,
                                                  dlogits, dx);
    return launch_result();
}

template <int NCH, int KMAX, bool WSMEM>
int launch_grad_fast(const Dims &p, const float *wr, const float *logits, const int32_t *idx,
                     const float *gate, const int32_t *slot, const __nv_bfloat16 *dy,
                     const __nv_bfloat16 *ye, float *dgate, float *dlogits, __nv_bfloat16 *dx,
                     size_t smem, cudaStream_t s) {
    auto kern = router_grad_fast_kernel<NCH, KMAX, WSMEM>;
    static std::atomic<int> smem_limit[64];
    static std::atomic<uint64_t> occupancy[64];  // per device: (smem << 32) | CTAs per SM
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return VMOE_ERR_CUDA;
    if (smem > 48 * 1024)
        if (const int st = raise_smem_limit((const void *)kern, smem_limit, (int)smem)) return st;
    const uint64_t o = occupancy[dev].load(std::memory_order_relaxed);
    int per_sm = (int)(o & 0xffffffffu);
    if (per_sm < 1 || (o >> 32) != (uint64_t)smem) {
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kern, RG_THREADS, smem) !=
                cudaSuccess ||
            per_sm < 1)
            return VMOE_ERR_CUDA;
        occupancy[dev].store(((uint64_t)smem << 32) | (uint32_t)per_sm, std::memory_order_relaxed);
    }
    const long long tokens = (long long)p.T * p.N;
    long long grid = (long long)per_sm * num_sms();
    grid = std::min(grid, (tokens + RG_WARPS - 1) / RG_WARPS);
    kern<<<(unsigned)grid, RG_THREADS, smem, s>>>(p, dy, ye, logits, idx, gate, slot, wr, dgate,
                                                  dlogits, dx);
    return launch_result();
}

template <int NCH, int KMAX>
int launch_grad_fast_w(const Dims &p, const float *wr, const float *logits, const int32_t *idx,
                       const float *gate, const int32_t *slot, const __nv_bfloat16 *dy,
                       const __nv_bfloat16 *ye, float *dgate, float *dlogits, __nv_bfloat16 *dx,
                       cudaStream_t s) {
    const size_t rows = rg_smem_rows(p);
    if (dx != nullptr && rows + rg_smem_w(p) <= RG_SMEM_CAP)
        return launch_grad_fast<NCH, KMAX, true>(p, wr, logits, idx, gate, slot, dy, ye, dgate,
                                                 dlogits, dx, rows + rg_smem_w(p), s);
    return launch_grad_fast<NCH, KMAX, false>(p, wr, logits, idx, gate, slot, dy, ye, dgate,
                                              dlogits, dx, rows, s);
}

template <int KMAX>
int launch_grad_fast_n(const Dims &p, const float *wr, const float *logits, const int32_t *idx,
                       const float *gate, const int32_t *slot, const __nv_bfloat16 *dy,
                       const __nv_bfloat16 *ye, float *dgate, float *dlogits, __nv_bfloat16 *dx,
                       cudaStream_t s) {
    const int nch = (p.d + 255) / 256;
    if (nch <= 1)
        return launch_grad_fast_w<1, KMAX>(p, wr, logits, idx, gate, slot, dy, ye, dgate, dlogits, dx, s);
    if (nch <= 2)
        return launch_grad_fast_w<2, KMAX>(p, wr, logits, idx, gate, slot, dy, ye, dgate, dlogits, dx, s);
    if (nch <= 3)
        return launch_grad_fast_w<3, KMAX>(p, wr, logits, idx, gate, slot, dy, ye, dgate, dlogits, dx, s);
    return launch_grad_fast_w<4, KMAX>(p, wr, logits, idx, gate, slot, dy, ye, dgate, dlogits, dx, s);
}

template <typename T, int KMAX>
int launch_grad_k(const Dims &p, const float *wr, const float *logits, const int32_t *idx,
                  const float *gate, const int32_t *slot, const T *dy, const T *ye, float *dgate,
                  float *dlogits, T *dx, cudaStream_t s) {
    const size_t rows = rg_smem_rows(p);
    if (dx != nullptr && rows + rg_smem_w(p) <= RG_SMEM_CAP)
        return launch_grad<T, KMAX, true>(p, wr, logits, idx, gate, slot, dy, ye, dgate, dlogits,
                                          dx, rows + rg_smem_w(p), s);
    return launch_grad<T, KMAX, false>(p, wr, logits, idx, gate, slot, dy, ye, dgate, dlogits, dx,
                                       rows, s);
}

template <typename T>
int run(const Dims &p, const void *x, const float *wr, const float *logits, const int32_t *idx,
        const float *gate, const int32_t *slot, const void *dy, const void *ye, float *dgate,
        float *dlogits, float *dw, float *dbias, void *dx, cudaStream_t s) {
    const T *dyt = (const T *)dy, *yet = (const T *)ye;
    T *dxt = (T *)dx;
    int st;
    trace_before(s, "router_grad");
    if (p.bf16 && p.k <= 2 && p.d <= 1024) {
        const __nv_bfloat16 *dyb = (const __nv_bfloat16 *)dy, *yeb = (const __nv_bfloat16 *)ye;
        __nv_bfloat16 *dxb = (__nv_bfloat16 *)dx;
        st = p.k <= 1 ? launch_grad_fast_n<1>(p, wr, logits, idx, gate, slot, dyb, yeb, dgate,
                                              dlogits, dxb, s)
                      : launch_grad_fast_n<2>(p, wr, logits, idx, gate, slot, dyb, yeb, dgate,
                                              dlogits, dxb, s);
    } else if (p.k <= 1)
        st = launch_grad_k<T, 1>(p, wr, logits, idx, gate, slot, dyt, yet, dgate, dlogits, dxt, s);
    else if (p.k <= 2)
        st = launch_grad_k<T, 2>(p, wr, logits, idx, gate, slot, dyt, yet, dgate, dlogits, dxt, s);
    else if (p.k <= 4)
        st = launch_grad_k<T, 4>(p, wr, logits, idx, gate, slot, dyt, yet, dgate, dlogits, dxt, s);
    else
        st = launch_grad_k<T, 8>(p, wr, logits, idx, gate, slot, dyt, yet, dgate, dlogits, dxt, s);
    trace_after(s);
    if (st != VMOE_OK) return st;
    trace_before(s, "router_dw");
    if (p.bf16 && (st = launch_router_dw_tc(p, (const __nv_bfloat16 *)x, dlogits, dw, dbias, s)) !=
                      VMOE_ERR_UNSUPPORTED) {
        trace_after(s);
        return st;
    }
    if (p.bf16) {
        dim3 grid(DW_SPLIT, (p.d + DW_BD - 1) / DW_BD, p.T * ((p.E + DW_BE - 1) / DW_BE));
        router_dw_mma_kernel<<<grid, DW_THREADS, 0, s>>>(p, (const __nv_bfloat16 *)x, dlogits, dw,
                                                         dbias);
    } else {
        dim3 grid((p.d + RT - 1) / RT, (p.E + RT - 1) / RT, p.T);
        router_dw_simt_kernel<<<grid, RD_THREADS, 0, s>>>(p, (const float *)x, dlogits, dw, dbias);
    }
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
