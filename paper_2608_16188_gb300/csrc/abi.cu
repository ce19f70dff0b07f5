// abi.cu -- the extern "C" entry points of libvmoe: argument checks, capacity
// rule, dtype selection, the device status word and the kernel trace.
#include <math.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <vector>

#include "common.cuh"

namespace vmoe {

// One status word per device that loads the library.  Kernels that give up a
// bounded wait OR a vmoe_status into it; vmoe_device_status reads it.
static __device__ int g_status_word = 0;

int *device_status_word() {
    static std::atomic<int *> addr[64];  // per device; the same value from every thread
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return nullptr;
    int *a = addr[dev].load(std::memory_order_acquire);
    if (!a) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_status_word) != cudaSuccess) return nullptr;
        a = static_cast<int *>(p);
        addr[dev].store(a, std::memory_order_release);
    }
    return a;
}

bool pdl_enabled() {
    static const bool on = [] {
        const char *v = getenv("VMOE_PDL");
        return !(v && v[0] == '0');
    }();
    return on;
}

bool pair_enabled() {
    static const bool on = [] {
        const char *v = getenv("VMOE_PAIR");
        return !(v && v[0] == '0');
    }();
    return on;
}

bool shares_enabled() {
    static const bool on = [] {
        const char *v = getenv("VMOE_SHARES");
        return v && v[0] == '1';
    }();
    return on;
}

bool route_tc_enabled() {
    static const bool on = [] {
        const char *v = getenv("VMOE_ROUTE_TC");
        return v && v[0] == '1';
    }();
    return on;
}

bool row_pair_enabled() {
    static const bool on = [] {
        const char *v = getenv("VMOE_ROW_PAIR");
        return v && v[0] == '1';
    }();
    return on;
}

int num_sms() {
    static std::atomic<int> sms[64];  // per device; the same value from every thread
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 1;
    int n = sms[dev].load(std::memory_order_relaxed);
    if (!n) {
        int v = 0;
        cudaDeviceGetAttribute(&v, cudaDevAttrMultiProcessorCount, dev);
        n = v > 0 ? v : 1;
        sms[dev].store(n, std::memory_order_relaxed);
    }
    return n;
}

// ---------------------------------------------------------------------------
// Kernel trace: host-thread-local list of (name, start event, stop event).
struct TraceRec {
    const char *name;
    cudaEvent_t start, stop;
};
struct Trace {
    bool on = false;
    int max_records = 0;
    int count = 0;
    std::vector<TraceRec> recs;  // event pool, reused across enables
};
static thread_local Trace g_trace;

void trace_before(cudaStream_t s, const char *kernel_name) {
    Trace &t = g_trace;
    if (!t.on || t.count >= t.max_records) return;
    TraceRec &r = t.recs[t.count];
    r.name = kernel_name;
    cudaEventRecord(r.start, s);
}

void trace_after(cudaStream_t s) {
    Trace &t = g_trace;
    if (!t.on || t.count >= t.max_records) return;
    cudaEventRecord(t.recs[t.count].stop, s);
    t.count++;
}

}  // namespace vmoe

using namespace vmoe;

static int capacity_of(const vmoe_problem *p) {
    if (p->capacity > 0) return p->capacity;
    double c = ceil(p->capacity_factor * (double)p->k * (double)p->N / (double)p->E);
    if (c < 1.0) c = 1.0;
    if (c > (double)p->N) c = (double)p->N;
    return (int)c;
}

// Checks the problem statement; fills `d`.  Returns VMOE_OK or an error.
static int check_problem(const vmoe_problem *p, Dims *d) {
    if (!p) return VMOE_ERR_INVALID;
    if (p->T < 1 || p->N < 1 || p->E < 1 || p->k < 1 || p->d_model < 1 || p->d_ff < 1)
        return VMOE_ERR_INVALID;
    if (p->k > p->E || p->k > 8) return VMOE_ERR_INVALID;
    if (p->dtype != VMOE_F32 && p->dtype != VMOE_BF16) return VMOE_ERR_INVALID;
    if (p->capacity < 0) return VMOE_ERR_INVALID;
    if (p->capacity == 0 && !(p->capacity_factor > 0.0 && isfinite(p->capacity_factor)))
        return VMOE_ERR_INVALID;
    if (p->flags & ~(uint32_t)(VMOE_LOGITS_IN | VMOE_NO_RENORM | VMOE_GELU_TANH))
        return VMOE_ERR_INVALID;
    if (p->E > 256) return VMOE_ERR_UNSUPPORTED;
    if ((long long)p->T * p->E > 1024) return VMOE_ERR_UNSUPPORTED;
    if (p->d_model % 8 != 0) return VMOE_ERR_UNSUPPORTED;
    // 32-bit element offsets inside one group / one task are assumed.
    if ((long long)p->N * p->d_model >= (1LL << 31)) return VMOE_ERR_UNSUPPORTED;
    if ((long long)p->d_model * p->d_ff >= (1LL << 31)) return VMOE_ERR_UNSUPPORTED;
    int C = capacity_of(p);
    if ((long long)C * p->d_ff >= (1LL << 31)) return VMOE_ERR_UNSUPPORTED;
    d->T = p->T;
    d->N = p->N;
    d->d = p->d_model;
    d->f = p->d_ff;
    d->E = p->E;
    d->k = p->k;
    d->C = C;
    d->flags = p->flags;
    d->bf16 = p->dtype == VMOE_BF16;
    return VMOE_OK;
}

static bool aligned16(const void *ptr) { return ((uintptr_t)ptr & 15u) == 0; }
static bool dev_ok(const void *ptr) { return ptr != nullptr && aligned16(ptr); }
static bool opt_ok(const void *ptr) { return ptr == nullptr || aligned16(ptr); }

static int check_expert_shape(const Dims &d) {
    if (d.bf16 && (d.d % 128 != 0 || d.f % 128 != 0)) return VMOE_ERR_UNSUPPORTED;
    if (!d.bf16 && (d.d % 4 != 0 || d.f % 4 != 0)) return VMOE_ERR_UNSUPPORTED;
    return VMOE_OK;
}

extern "C" {

int vmoe_version(void) { return VMOE_VERSION; }

const char *vmoe_status_string(int status) {
    switch (status) {
        case VMOE_OK: return "VMOE_OK";
        case VMOE_ERR_INVALID: return "VMOE_ERR_INVALID: invalid argument";
        case VMOE_ERR_UNSUPPORTED: return "VMOE_ERR_UNSUPPORTED: unsupported shape";
        case VMOE_ERR_CUDA: return "VMOE_ERR_CUDA: CUDA runtime error";
        case VMOE_ERR_DEVICE_TIMEOUT: return "VMOE_ERR_DEVICE_TIMEOUT: a kernel gave up a bounded wait";
        default: return "unknown vmoe status";
    }
}

int vmoe_problem_capacity(const vmoe_problem *p) {
    Dims d;
    int st = check_problem(p, &d);
    return st == VMOE_OK ? d.C : st;
}

int vmoe_route(const vmoe_problem *p, const void *x, const float *w_router,
               const float *logit_bias, float *logits, int32_t *expert_idx, float *gate,
               int32_t *slot, int32_t *load, void *cuda_stream) {
    Dims d;
    int st = check_problem(p, &d);
    if (st != VMOE_OK) return st;
    bool given = (p->flags & VMOE_LOGITS_IN) != 0;
    if (!given && (!dev_ok(x) || !dev_ok(w_router))) return VMOE_ERR_INVALID;
    if (!opt_ok(logit_bias) || !dev_ok(logits) || !dev_ok(expert_idx) || !dev_ok(gate) ||
        !dev_ok(slot) || !dev_ok(load))
        return VMOE_ERR_INVALID;
    return launch_route(d, given ? nullptr : x, w_router, logit_bias, logits, expert_idx, gate,
                        slot, load, (cudaStream_t)cuda_stream);
}

int vmoe_dispatch(const vmoe_problem *p, const void *src, const float *weight,
                  const int32_t *expert_idx, const int32_t *slot, const int32_t *load,
                  void *dst, void *cuda_stream) {
    Dims d;
    int st = check_problem(p, &d);
    if (st != VMOE_OK) return st;
    if (!dev_ok(src) || !opt_ok(weight) || !dev_ok(expert_idx) || !dev_ok(slot) ||
        !dev_ok(load) || !dev_ok(dst))
        return VMOE_ERR_INVALID;
    return launch_dispatch(d, src, weight, expert_idx, slot, load, dst, (cudaStream_t)cuda_stream);
}

int vmoe_combine(const vmoe_problem *p, const void *src, const float *weight,
                 const int32_t *expert_idx, const int32_t *slot, void *dst, void *cuda_stream) {
    Dims d;
    int st = check_problem(p, &d);
    if (st != VMOE_OK) return st;
    if (!dev_ok(src) || !opt_ok(weight) || !dev_ok(expert_idx) || !dev_ok(slot) || !dev_ok(dst))
        return VMOE_ERR_INVALID;
    return launch_combine(d, src, weight, expert_idx, slot, dst, (cudaStream_t)cuda_stream);
}

int vmoe_router_bwd(const vmoe_problem *p, const void *x, const float *w_router,
                    const float *logits, const int32_t *expert_idx, const float *gate,
                    const int32_t *slot, const void *dy, const void *ye, float *dgate,
                    float *dlogits, float *dw_router, float *dbias, void *dx,
                    void *cuda_stream) {
    Dims d;
    int st = check_problem(p, &d);
    if (st != VMOE_OK) return st;
    if (!dev_ok(x) || !dev_ok(expert_idx) || !dev_ok(gate) || !dev_ok(slot) || !dev_ok(dy) ||
        !dev_ok(ye) || !dev_ok(dgate) || !dev_ok(dlogits) || !dev_ok(dw_router) ||
        !opt_ok(dbias) || !opt_ok(dx))
        return VMOE_ERR_INVALID;
    if (dx ? !dev_ok(w_router) : !opt_ok(w_router)) return VMOE_ERR_INVALID;
    if ((p->flags & VMOE_NO_RENORM) ? !dev_ok(logits) : !opt_ok(logits)) return VMOE_ERR_INVALID;
    return launch_router_bwd(d, x, w_router, logits, expert_idx, gate, slot, dy, ye, dgate,
                             dlogits, dw_router, dbias, dx, (cudaStream_t)cuda_stream);
}

int vmoe_expert_fwd(const vmoe_problem *p, const void *xe, const void *w1, const void *w2,
                    const int32_t *load, void *h, void *a, void *ye, void *cuda_stream) {
    Dims d;
    int st = check_problem(p, &d);
    if (st != VMOE_OK) return st;
    if ((st = check_expert_shape(d)) != VMOE_OK) return st;
    if (!dev_ok(xe) || !dev_ok(w1) || !dev_ok(w2) || !dev_ok(load) || !dev_ok(h) ||
        !dev_ok(a) || !dev_ok(ye))
        return VMOE_ERR_INVALID;
    cudaStream_t s = (cudaStream_t)cuda_stream;
    if (d.bf16)
        return launch_expert_fwd_bf16(
            d, (const __nv_bfloat16 *)xe, (const __nv_bfloat16 *)w1, (const __nv_bfloat16 *)w2,
            load, (__nv_bfloat16 *)h, (__nv_bfloat16 *)a, (__nv_bfloat16 *)ye, s);
    return launch_expert_fwd_f32(d, (const float *)xe, (const float *)w1, (const float *)w2, load,
                                 (float *)h, (float *)a, (float *)ye, s);
}

size_t vmoe_expert_bwd_workspace_size(const vmoe_problem *p) {
    Dims d;
    if (check_problem(p, &d) != VMOE_OK) return 0;
    // bf16: dH as a (bf16 part, bf16 residual) pair per element; fp32: dH itself.
    size_t per_elem = d.bf16 ? 2 * 2 : 4;
    return (size_t)d.T * d.E * d.C * d.f * per_elem;
}

size_t vmoe_expert_bwd_min_workspace_size(const vmoe_problem *p) {
    Dims d;
    if (check_problem(p, &d) != VMOE_OK) return 0;
    return d.bf16 ? bwd_min_workspace(d) : vmoe_expert_bwd_workspace_size(p);
}

int vmoe_expert_bwd(const vmoe_problem *p, const void *xe, const void *h, const void *a,
                    const void *w1, const void *w2, const void *dye, const int32_t *load,
                    void *dxe, void *dw1, void *dw2, void *workspace, size_t workspace_bytes,
                    void *cuda_stream) {
    Dims d;
    int st = check_problem(p, &d);
    if (st != VMOE_OK) return st;
    if ((st = check_expert_shape(d)) != VMOE_OK) return st;
    if (!dev_ok(xe) || !dev_ok(h) || !dev_ok(a) || !dev_ok(w1) || !dev_ok(w2) || !dev_ok(dye) ||
        !dev_ok(load) || !dev_ok(dxe) || !dev_ok(dw1) || !dev_ok(dw2) || !dev_ok(workspace))
        return VMOE_ERR_INVALID;
    cudaStream_t s = (cudaStream_t)cuda_stream;
    if (workspace_bytes < vmoe_expert_bwd_workspace_size(p)) {
        // a smaller workspace: the backward in slices (bf16 only)
        if (!d.bf16 || workspace_bytes < bwd_min_workspace(d)) return VMOE_ERR_INVALID;
        return launch_expert_bwd_bf16_sliced(
            d, (const __nv_bfloat16 *)xe, (const __nv_bfloat16 *)h, (const __nv_bfloat16 *)a,
            (const __nv_bfloat16 *)w1, (const __nv_bfloat16 *)w2, (const __nv_bfloat16 *)dye, load,
            (__nv_bfloat16 *)dxe, (__nv_bfloat16 *)dw1, (__nv_bfloat16 *)dw2, workspace,
            workspace_bytes, s, nullptr);
    }
    if (d.bf16)
        return launch_expert_bwd_bf16(
            d, (const __nv_bfloat16 *)xe, (const __nv_bfloat16 *)h, (const __nv_bfloat16 *)a,
            (const __nv_bfloat16 *)w1, (const __nv_bfloat16 *)w2, (const __nv_bfloat16 *)dye, load,
            (__nv_bfloat16 *)dxe, (__nv_bfloat16 *)dw1, (__nv_bfloat16 *)dw2,
            (__nv_bfloat16 *)workspace, s);
    return launch_expert_bwd_f32(d, (const float *)xe, (const float *)h, (const float *)a,
                                 (const float *)w1, (const float *)w2, (const float *)dye, load,
                                 (float *)dxe, (float *)dw1, (float *)dw2, (float *)workspace, s);
}

// Attention experts: bf16, head dimension 64, an even number of heads (the
// projection GEMMs need H * 64 to be a multiple of 128), d % 128 == 0, C <= 512.
static int check_attn(const vmoe_problem *p, int heads, Dims *d) {
    int st = check_problem(p, d);
    if (st != VMOE_OK) return st;
    if (heads < 1) return VMOE_ERR_INVALID;
    if (!d->bf16 || heads % 2 != 0 || d->d % 128 != 0 || !attn_core_supported(d->C, 64))
        return VMOE_ERR_UNSUPPORTED;
    if ((long long)d->C * 3 * heads * 64 >= (1LL << 31)) return VMOE_ERR_UNSUPPORTED;
    return VMOE_OK;
}

int vmoe_attn_expert_fwd(const vmoe_problem *p, int heads, const void *xe, const void *wqkv,
                         const void *wo, const int32_t *load, void *qkv, void *o, float *lse, void *ye,
                         void *cuda_stream) {
    Dims d;
    int st = check_attn(p, heads, &d);
    if (st != VMOE_OK) return st;
    if (!dev_ok(xe) || !dev_ok(wqkv) || !dev_ok(wo) || !dev_ok(load) || !dev_ok(qkv) || !dev_ok(o) ||
        !dev_ok(lse) || !dev_ok(ye))
        return VMOE_ERR_INVALID;
    return launch_attn_expert_fwd(d, heads, (const __nv_bfloat16 *)xe, (const __nv_bfloat16 *)wqkv,
                                  (const __nv_bfloat16 *)wo, load, (__nv_bfloat16 *)qkv, (__nv_bfloat16 *)o,
                                  lse, (__nv_bfloat16 *)ye, (cudaStream_t)cuda_stream);
}

size_t vmoe_attn_expert_bwd_workspace_size(const vmoe_problem *p, int heads) {
    Dims d;
    if (check_attn(p, heads, &d) != VMOE_OK) return 0;
    return attn_bwd_workspace(d, heads);
}

int vmoe_attn_expert_bwd(const vmoe_problem *p, int heads, const void *xe, const void *qkv,
                         const void *o, const float *lse, const void *wqkv, const void *wo,
                         const void *dye, const int32_t *load, void *dxe, void *dwqkv, void *dwo,
                         void *workspace, size_t workspace_bytes, void *cuda_stream) {
    Dims d;
    int st = check_attn(p, heads, &d);
    if (st != VMOE_OK) return st;
    if (!dev_ok(xe) || !dev_ok(qkv) || !dev_ok(o) || !dev_ok(lse) || !dev_ok(wqkv) || !dev_ok(wo) ||
        !dev_ok(dye) || !dev_ok(load) || !dev_ok(dxe) || !dev_ok(dwqkv) || !dev_ok(dwo) ||
        !dev_ok(workspace))
        return VMOE_ERR_INVALID;
    if (workspace_bytes < attn_bwd_workspace(d, heads)) return VMOE_ERR_INVALID;
    return launch_attn_expert_bwd(d, heads, (const __nv_bfloat16 *)xe, (const __nv_bfloat16 *)qkv,
                                  (const __nv_bfloat16 *)o, lse, (const __nv_bfloat16 *)wqkv,
                                  (const __nv_bfloat16 *)wo, (const __nv_bfloat16 *)dye, load,
                                  (__nv_bfloat16 *)dxe, (__nv_bfloat16 *)dwqkv, (__nv_bfloat16 *)dwo,
                                  workspace, (cudaStream_t)cuda_stream);
}

int vmoe_device_status(int reset) {
    if (cudaDeviceSynchronize() != cudaSuccess) return VMOE_ERR_CUDA;
    int *addr = device_status_word();
    if (!addr) return VMOE_ERR_CUDA;
    int v = 0;
    if (cudaMemcpy(&v, addr, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        return VMOE_ERR_CUDA;
    if (reset) {
        int z = 0;
        if (cudaMemcpy(addr, &z, sizeof(int), cudaMemcpyHostToDevice) != cudaSuccess)
            return VMOE_ERR_CUDA;
    }
    return v;
}

int vmoe_trace_enable(int max_records) {
    if (max_records < 1 || max_records > (1 << 20)) return VMOE_ERR_INVALID;
    Trace &t = g_trace;
    while ((int)t.recs.size() < max_records) {
        TraceRec r;
        r.name = nullptr;
        if (cudaEventCreate(&r.start) != cudaSuccess) return VMOE_ERR_CUDA;
        if (cudaEventCreate(&r.stop) != cudaSuccess) {
            cudaEventDestroy(r.start);
            return VMOE_ERR_CUDA;
        }
        t.recs.push_back(r);
    }
    t.max_records = max_records;
    t.count = 0;
    t.on = true;
    return VMOE_OK;
}

int vmoe_trace_disable(void) {
    g_trace.on = false;
    return g_trace.count;
}

int vmoe_trace_get(int i, const char **kernel_name, float *ms) {
    Trace &t = g_trace;
    if (i < 0 || i >= t.count || !kernel_name || !ms) return VMOE_ERR_INVALID;
    if (cudaEventSynchronize(t.recs[i].stop) != cudaSuccess) return VMOE_ERR_CUDA;
    if (cudaEventElapsedTime(ms, t.recs[i].start, t.recs[i].stop) != cudaSuccess)
        return VMOE_ERR_CUDA;
    *kernel_name = t.recs[i].name;
    return VMOE_OK;
}

}  // extern "C"
