// gemm_tc_bwd.cu -- backward launches of the tcgen05 grouped GEMM:
//   dA + GELU': dH = (dYe W2^T) * GELU'(H)  (A: dYe K-major; B: W2 [f,d] read K-major)
//   dX:         dXe = dH W1^T               (A: dH K-major;  B: W1 [d,f] read K-major)
//   dW1:        dW1 = Xe^T dH               (both MN-major, K = load)
//   dW2:        dW2 = A^T dYe               (both MN-major, K = load)
#include <vector>

#include "gemm_tc2.cuh"
#include "planner.cuh"

namespace vmoe {

int plan_shares(int n, const double *work, const int32_t *minimum, const int32_t *saturation,
                int32_t budget, int32_t *shares);                      // planner.cu

namespace tc {
int pair_clusters(const void *kern, size_t smem) {
    // per device and kernel: the kernels are few, a small table does
    struct Entry {
        std::atomic<const void *> kern;
        std::atomic<int> n;
    };
    static Entry cache[64][8];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    for (auto &e : cache[dev])
        if (e.kern.load(std::memory_order_acquire) == kern) return e.n.load(std::memory_order_relaxed);
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(2 * (unsigned)num_sms());
    cfg.blockDim = dim3(THREADS);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, kern, &cfg) != cudaSuccess || n <= 0) return 0;
    static std::mutex mu;
    std::lock_guard<std::mutex> lock(mu);
    for (auto &e : cache[dev]) {
        const void *k = e.kern.load(std::memory_order_relaxed);
        if (k == kern) break;
        if (k == nullptr) {
            e.n.store(n, std::memory_order_relaxed);
            e.kern.store(kern, std::memory_order_release);
            break;
        }
    }
    return n;
}
}  // namespace tc

using namespace tc;

int launch_expert_bwd_bf16(const Dims &p, const __nv_bfloat16 *xe, const __nv_bfloat16 *h,
                           const __nv_bfloat16 *act, const __nv_bfloat16 *w1,
                           const __nv_bfloat16 *w2, const __nv_bfloat16 *dye,
                           const int32_t *load, __nv_bfloat16 *dxe, __nv_bfloat16 *dw1,
                           __nv_bfloat16 *dw2, __nv_bfloat16 *dh, cudaStream_t s) {
    // dH is kept as a bf16 pair: the workspace holds, per group, dH_hi in rows
    // [0, C) and the residual dH_lo = dH - dH_hi in rows [C, 2C).  dX uses dH_hi;
    // dW1 = Xe^T dH_hi + Xe^T dH_lo, which keeps short weight-gradient sums
    // (groups with a few rows, where terms cancel) at fp32-like accuracy.
    const long long C = p.C, f = p.f;
    __nv_bfloat16 *dh_hi = dh, *dh_lo = dh + C * f;
    int st = row_gemm<EPI_DGELU, false>(p, dye, p.d, w2, p.f, load, dh_hi, dh_lo, h, s,
                                        "tc_da_dgelu", 2 * C * f, C * f);
    if (st != VMOE_OK) return st;
    if ((st = row_gemm<EPI_STORE, false>(p, dh_hi, p.f, w1, p.d, load, dxe, nullptr, nullptr, s,
                                         "tc_dx", 0, 0, 2 * C * f)) != VMOE_OK)
        return st;
    if ((st = wgrad_gemm(p, xe, p.d, dh, p.f, load, dw1, s, "tc_dw1", true)) != VMOE_OK) return st;
    return wgrad_gemm(p, act, p.f, dye, p.d, load, dw2, s, "tc_dw2");
}

// The backward under a dH budget (the expert groups' temporary memory, Section
// 3.2.1): when the workspace cannot hold dH for every group, the groups are
// placed in slices by the cross-task DP planner, each group's footprint being
// its dH rows (load rows of dH_hi, then load rows of the residual), in units of
// BW_UNIT rows; the slice's groups are packed into the workspace at 8-row
// offsets, and dA, dX and dW1 run per slice.  dW2 needs no dH and runs once.
// The loads are read back to the host first (one stream synchronisation).
// dW2 is launched before any planning, and the DP hands out one slice at a
// time: the host places the groups of slice s + 1 while the GPU runs slice s
// (and, for the first slice, dW2).  Each slice's plan (group list and first
// rows) reaches the head of the workspace through a small kernel whose
// parameters carry it, so no host copy waits for the stream.
constexpr int BW_UNIT = 8;
constexpr int PLAN_CHUNK = 256;

size_t bwd_plan_bytes(const Dims &p) { return (((size_t)2 * p.G() * sizeof(int32_t)) + 255) & ~(size_t)255; }

size_t bwd_min_workspace(const Dims &p) {
    const size_t unit_rows = ((size_t)2 * p.C + BW_UNIT - 1) / BW_UNIT * BW_UNIT;
    return bwd_plan_bytes(p) + unit_rows * p.f * sizeof(__nv_bfloat16);
}

namespace {
// Up to PLAN_CHUNK plan entries of one slice, by value: entry pos + i is group
// g[i], whose dH rows start at row[i] of the workspace.
struct PlanChunk {
    int32_t n, pos, G;
    int32_t g[PLAN_CHUNK];
    int32_t row[PLAN_CHUNK];
};

__global__ void __launch_bounds__(PLAN_CHUNK) plan_write_kernel(const __grid_constant__ PlanChunk c,
                                                               int32_t *__restrict__ plan) {
    const int i = threadIdx.x;
    if (i < c.n) {
        plan[c.pos + i] = c.g[i];
        plan[c.G + c.pos + i] = c.row[i];
    }
}
}  // namespace

int launch_expert_bwd_bf16_sliced(const Dims &p, const __nv_bfloat16 *xe, const __nv_bfloat16 *h,
                                  const __nv_bfloat16 *act, const __nv_bfloat16 *w1,
                                  const __nv_bfloat16 *w2, const __nv_bfloat16 *dye,
                                  const int32_t *load, __nv_bfloat16 *dxe, __nv_bfloat16 *dw1,
                                  __nv_bfloat16 *dw2, void *workspace, size_t workspace_bytes,
                                  cudaStream_t s, int *nslices_out) {
    const int G = p.G();
    const size_t plan_bytes = bwd_plan_bytes(p);
    if (workspace_bytes < bwd_min_workspace(p)) return VMOE_ERR_INVALID;
    long long rows = (long long)((workspace_bytes - plan_bytes) / ((size_t)p.f * sizeof(__nv_bfloat16)));
    if (rows > 0x7fffffffLL) rows = 0x7fffffffLL;  // compact row offsets are int32
    std::vector<int32_t> hload(G);
    if (cudaMemcpyAsync(hload.data(), load, sizeof(int32_t) * G, cudaMemcpyDeviceToHost, s) !=
            cudaSuccess ||
        cudaStreamSynchronize(s) != cudaSuccess)
        return VMOE_ERR_CUDA;
    std::vector<int64_t> w(G);
    std::vector<double> r(G);
    long long total_units = 0;
    for (int g = 0; g < G; ++g) {
        const int L = hload[g] < 0 ? 0 : (hload[g] > p.C ? p.C : hload[g]);
        hload[g] = L;
        w[g] = (2LL * L + BW_UNIT - 1) / BW_UNIT;
        r[g] = (double)L;
        total_units += w[g];
    }
    // no slice needs more than every group's footprint: that bounds the DP table
    long long cap_units = rows / BW_UNIT;
    if (cap_units > total_units) cap_units = total_units;
    SlicePlanner planner;
    int st = planner.init(G, w.data(), r.data(), cap_units, 0.0, 0.0);
    if (st != VMOE_OK) return st;
    // dW2 first: it needs no dH, and it runs while the first slice is planned
    if ((st = wgrad_gemm(p, act, p.f, dye, p.d, load, dw2, s, "tc_dw2")) != VMOE_OK) return st;
    int32_t *dplan = reinterpret_cast<int32_t *>(workspace);
    __nv_bfloat16 *dh = reinterpret_cast<__nv_bfloat16 *>(static_cast<uint8_t *>(workspace) + plan_bytes);
    // dW1 of a slice on SM pairs, optionally (VMOE_SHARES=1) with each group's
    // column tiles on a share of the pairs from the fill-clamp-refill allocation
    // (Section 3.2.2): work = its tiles x (output bytes + load x input bytes per
    // row), at least one pair, at most one pair per tile; slices with more
    // groups than pairs keep the round-robin schedule.
    const bool use_shares = shares_enabled() && pair_enabled() && p.d % 256 == 0 && p.f % 256 == 0 &&
                            p.C <= 4 * BK;
    const int pairs = use_shares ? pair_wgrad_capacity<true>(p.C) : 0;
    auto slice_schedule = [&](const std::vector<int> &slice, PairSchedule &sc) {
        sc.enabled = 0;
        const int n = (int)slice.size();
        if (pairs <= 0 || n > pairs || pairs > MAX_PAIRS) return;
        const int units = p.f / 256, tiles_m = p.d / 256;
        std::vector<double> work(n);
        std::vector<int32_t> mn(n, 1), sat(n, units), share(n);
        for (int i = 0; i < n; ++i) {
            const double L = hload[slice[i]];
            work[i] = units * ((double)tiles_m * 256 * 256 * 2 + L * ((double)p.d * 2 + 4 * 256));
        }
        if (plan_shares(n, work.data(), mn.data(), sat.data(), pairs, share.data()) < 0) return;
        int c = 0;
        for (int i = 0; i < n; ++i)
            for (int j = 0; j < share[i]; ++j, ++c) {
                const int lo = j * units / share[i], hi = (j + 1) * units / share[i];
                sc.first[c] = i * units + lo;
                sc.count[c] = hi - lo;
            }
        for (; c < MAX_PAIRS; ++c) sc.first[c] = sc.count[c] = 0;
        sc.enabled = 1;
    };
    std::vector<int> slice;
    int pos = 0, ns = 0;
    while (st == VMOE_OK && planner.next(slice)) {
        const int n = (int)slice.size();
        // this slice's plan entries [pos, pos + n) on the device
        PlanChunk c;
        c.G = G;
        long long row = 0;
        for (int k0 = 0; k0 < n && st == VMOE_OK; k0 += PLAN_CHUNK) {
            c.pos = pos + k0;
            c.n = n - k0 < PLAN_CHUNK ? n - k0 : PLAN_CHUNK;
            for (int i = 0; i < c.n; ++i) {
                c.g[i] = slice[k0 + i];
                c.row[i] = (int32_t)row;
                row += w[slice[k0 + i]] * BW_UNIT;
            }
            trace_before(s, "bwd_plan");
            plan_write_kernel<<<1, PLAN_CHUNK, 0, s>>>(c, dplan);
            st = launch_result();
            trace_after(s);
        }
        if (st != VMOE_OK) break;
        Slice sl;
        sl.glist = dplan + pos;
        sl.crow = dplan + G + pos;
        sl.n = n;
        sl.rows = rows;
        sl.compact = CMP_D;
        st = row_gemm<EPI_DGELU, false>(p, dye, p.d, w2, p.f, load, dh, dh, h, s, "tc_da_dgelu", 0, 0, 0,
                                        sl);
        if (st != VMOE_OK) break;
        sl.compact = CMP_A;
        st = row_gemm<EPI_STORE, false>(p, dh, p.f, w1, p.d, load, dxe, nullptr, nullptr, s, "tc_dx", 0,
                                        0, 0, sl);
        if (st != VMOE_OK) break;
        sl.compact = CMP_B;
        PairSchedule sc;
        slice_schedule(slice, sc);
        st = wgrad_gemm(p, xe, p.d, dh, p.f, load, dw1, s, "tc_dw1", true, sl, &sc);
        pos += n;
        ++ns;
    }
    if (nslices_out) *nslices_out = ns;
    return st;
}

// Attention experts, backward: dO = dYe W_o^T, dW_o = O^T dYe, the attention
// core's dQ, dK, dV (attention.cu) into dQKV, dXe = dQKV W_qkv^T and
// dW_qkv = Xe^T dQKV.  The workspace holds dO [G, C, H dk] and dQKV
// [G, C, 3 H dk] (bf16), then D [G, H, C] (fp32).
size_t attn_bwd_workspace(const Dims &p, int H) {
    const size_t hd = (size_t)H * 64, rows = (size_t)p.G() * p.C;
    return rows * hd * 2 + rows * 3 * hd * 2 + (size_t)p.G() * H * p.C * 4;
}

int launch_attn_expert_bwd(const Dims &p, int H, const __nv_bfloat16 *xe, const __nv_bfloat16 *qkv,
                           const __nv_bfloat16 *o, const float *lse, const __nv_bfloat16 *wqkv,
                           const __nv_bfloat16 *wo, const __nv_bfloat16 *dye, const int32_t *load,
                           __nv_bfloat16 *dxe, __nv_bfloat16 *dwqkv, __nv_bfloat16 *dwo, void *workspace,
                           cudaStream_t s) {
    const int hd = H * 64;
    const size_t rows = (size_t)p.G() * p.C;
    __nv_bfloat16 *dout = static_cast<__nv_bfloat16 *>(workspace);
    __nv_bfloat16 *dqkv = dout + rows * hd;
    float *dsum = reinterpret_cast<float *>(dqkv + rows * 3 * hd);
    int st = row_gemm<EPI_STORE, false>(p, dye, p.d, wo, hd, load, dout, nullptr, nullptr, s, "attn_dout");
    if (st != VMOE_OK) return st;
    if ((st = wgrad_gemm(p, o, hd, dye, p.d, load, dwo, s, "attn_dwo")) != VMOE_OK) return st;
    if ((st = launch_attn_core_bwd(p.G(), p.C, H, load, qkv, o, lse, dout, dsum, dqkv, s)) != VMOE_OK)
        return st;
    if ((st = row_gemm<EPI_STORE, false>(p, dqkv, 3 * hd, wqkv, p.d, load, dxe, nullptr, nullptr, s,
                                         "attn_dxe")) != VMOE_OK)
        return st;
    return wgrad_gemm(p, xe, p.d, dqkv, 3 * hd, load, dwqkv, s, "attn_dwqkv");
}

}  // namespace vmoe
