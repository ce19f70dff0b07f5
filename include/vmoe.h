/*
 * vmoe.h -- C ABI of libvmoe: one adaptation step of T concurrent V-MoE expert
 * layers on one NVIDIA GB300 (sm_103a).
 *
 * The method is AdaSprite's multi-task V-MoE co-adaptation (arxiv 2608.16188):
 * the experts of T V-MoEs form one pool (Section 2.2, "MoE merging"); each
 * task keeps its own router and experts and its tokens are routed to their
 * most relevant experts (Section 2.1) under per-expert capacity limits
 * (Challenge #1 in Section 1, Section 2.3.1); the experts of all tasks run
 * concurrently (Section 3.2, expert parallelism) and only the visual
 * experts are adapted (Section 3.1, specification-based tuning).  Here every
 * stage is one grouped launch over all T*E (task, expert) groups.
 *
 * One step is:
 *   vmoe_route     logits = x W_r + bias; softmax; top-k; capacity scan
 *   vmoe_dispatch  Xe  = gather(x)               (padding rows zero)
 *   vmoe_expert_fwd H = Xe W1, A = GELU(H), Ye = A W2
 *   vmoe_combine   y   = sum_j gate_j * Ye[e_j, s_j]
 *   vmoe_dispatch  dYe = gate * gather(dY)
 *   vmoe_expert_bwd dH = (dYe W2^T) * GELU'(H), dXe = dH W1^T,
 *                  dW1 = Xe^T dH, dW2 = A^T dYe
 *   vmoe_combine   dX  = sum_j dXe[e_j, s_j]
 *   vmoe_router_bwd dgate, dlogits, dW_r, dbias; dX += dlogits W_r^T
 *
 * Conventions for every entry point:
 *  - Ownership: every array argument is caller-owned DEVICE memory (except
 *    the vmoe_problem struct, read on the host), row-major and contiguous in
 *    the layout stated, with a base address aligned to 16 bytes.  The library
 *    allocates no device memory and keeps no state between calls other than
 *    the device status word (vmoe_device_status) and the optional trace.
 *  - Execution: calls enqueue kernels on `cuda_stream` (a cudaStream_t; NULL
 *    is the legacy default stream) and return without synchronising.
 *  - Errors: arguments are checked on the host before any launch; an invalid
 *    argument returns VMOE_ERR_INVALID and an unsupported shape
 *    VMOE_ERR_UNSUPPORTED, in both cases with nothing launched.  A failed
 *    launch returns VMOE_ERR_CUDA.  Device data is trusted: loads are clamped
 *    to [0, C], and expert indices or slots out of range are undefined
 *    behaviour.
 *  - Determinism: results are bitwise reproducible run to run (no atomics in
 *    any reduction, fixed summation orders).
 *  - Host threads: entry points may be called from several host threads at
 *    once, each with its own stream and arrays; the kernel trace is kept per
 *    host thread.  The exception is vmoe_expert_bwd_static_scratch, whose
 *    calls share one device array (see there).
 *  - Dtypes: x, dY, weights and all activations use p->dtype (fp32 or bf16);
 *    W_r, bias, logits and gates are always fp32.  bf16 contractions
 *    accumulate in fp32 on the tcgen05 tensor cores; fp32 runs on CUDA cores.
 *
 * Shapes (t < T tasks, n < N tokens per task, e < E experts per task,
 * j < k choices, s < C capacity slots, g = t*E + e):
 *   x, y, dY, dX [T,N,d]   W_r [T,d,E]   bias [T,E]   logits [T,N,E]
 *   expert_idx, gate, slot [T,N,k]   load [T,E]
 *   Xe, Ye, dYe, dXe [T,E,C,d]   H, A [T,E,C,f]
 *   W1, dW1 [T,E,d,f]   W2, dW2 [T,E,f,d]
 */
#ifndef VMOE_H
#define VMOE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define VMOE_VERSION 1

typedef enum {
    VMOE_OK = 0,
    VMOE_ERR_INVALID = -1,        /* bad argument; nothing launched */
    VMOE_ERR_UNSUPPORTED = -2,    /* valid but unsupported shape; nothing launched */
    VMOE_ERR_CUDA = -3,           /* a CUDA runtime call or launch failed */
    VMOE_ERR_DEVICE_TIMEOUT = -4  /* a kernel gave up a bounded wait (vmoe_device_status) */
} vmoe_status;

typedef enum { VMOE_F32 = 0, VMOE_BF16 = 1 } vmoe_dtype;

enum {
    VMOE_LOGITS_IN = 1u << 0, /* vmoe_route reads `logits` instead of computing them */
    VMOE_NO_RENORM = 1u << 1, /* gate = softmax probability (V-MoE); default renormalises over top-k */
    VMOE_GELU_TANH = 1u << 2  /* tanh-approximate GELU; default is the exact erf form */
};

/* The problem statement: T tasks, each with N tokens of width d_model, its own
 * router and E experts of hidden width d_ff; top-k routing with capacity
 * C = ceil(capacity_factor * k * N / E) clamped to [1, N], or `capacity` when
 * it is > 0.  Limits: T, N, E >= 1; 1 <= k <= min(E, 8); E <= 256;
 * T*E <= 1024; d_model % 8 == 0.  The bf16 expert path also needs d_model and
 * d_ff to be multiples of 128 (VMOE_ERR_UNSUPPORTED otherwise). */
typedef struct {
    int32_t T, N, d_model, d_ff, E, k;
    double capacity_factor;
    int32_t capacity;
    vmoe_dtype dtype;
    uint32_t flags;
} vmoe_problem;

/* Library version (VMOE_VERSION). */
int vmoe_version(void);

/* Human-readable name of a vmoe_status value (static storage). */
const char *vmoe_status_string(int status);

/* The capacity C the library uses for `p` (capacity rule above), or a negative
 * vmoe_status if `p` is invalid.  Host only; no device work. */
int vmoe_problem_capacity(const vmoe_problem *p);

/* Routing: top-k softmax gating with per-expert capacity (Section 2.1 routing
 * to the most relevant experts; capacity limits of Challenge #1; sequential
 * assignment of Section 3.3.1).
 *   x          [T,N,d] p->dtype           input tokens (unused with VMOE_LOGITS_IN; may be NULL then)
 *   w_router   [T,d,E] fp32               per-task router (unused with VMOE_LOGITS_IN)
 *   logit_bias [T,E]   fp32, nullable     per-task additive logit bias
 *   logits     [T,N,E] fp32               output, or input with VMOE_LOGITS_IN
 *   expert_idx [T,N,k] int32 out          the k largest logits, descending, ties to the lower index
 *   gate       [T,N,k] fp32 out           softmax probability of each choice, divided by the
 *                                         top-k probability mass unless VMOE_NO_RENORM
 *   slot       [T,N,k] int32 out          position in the expert's buffer, -1 if dropped: in
 *                                         choice-major order (all first choices in token order,
 *                                         then all second choices, ...) the s-th assignment to an
 *                                         expert gets slot s while s < C
 *   load       [T,E]   int32 out          kept assignments per expert = min(count, C)
 * Logits are accumulated in fp32.  A NaN logit is treated as -inf when the
 * experts are chosen (indices stay in range); its gates are unspecified. */
int vmoe_route(const vmoe_problem *p, const void *x, const float *w_router,
               const float *logit_bias, float *logits, int32_t *expert_idx, float *gate,
               int32_t *slot, int32_t *load, void *cuda_stream);

/* Dispatch (permute into expert-contiguous buffers for the grouped expert
 * launch of Section 3.2): dst[t,e,s,:] = w * src[t,n,:] for the kept choice
 * (n, j) with expert_idx = e and slot = s, w = weight[t,n,j] or 1 if weight
 * is NULL; rows s >= load[t,e] of dst are written as zero.
 *   src [T,N,d] p->dtype, weight [T,N,k] fp32 nullable, expert_idx/slot [T,N,k],
 *   load [T,E], dst [T,E,C,d] p->dtype (every element written).
 * The weighted product is formed in fp32 and rounded to p->dtype. */
int vmoe_dispatch(const vmoe_problem *p, const void *src, const float *weight,
                  const int32_t *expert_idx, const int32_t *slot, const int32_t *load,
                  void *dst, void *cuda_stream);

/* Expert FFN forward over all T*E groups in one grouped launch per layer
 * (Section 2.1: the ViT MLP block becomes experts; no bias terms):
 *   H = Xe W1, A = GELU(H), Ye = A W2, per group g for its rows s < load[g].
 *   xe [T,E,C,d], w1 [T,E,d,f], w2 [T,E,f,d], load [T,E] int32
 *   h, a [T,E,C,f] out, ye [T,E,C,d] out -- rows s >= load[g] are not written.
 * Rows s >= load[g] of xe are padding: their contents (NaN included) reach no
 * output.  load[g] is clamped to [0, C].
 * bf16: fp32 accumulation; A is GELU of the fp32 accumulator, H and A are
 * stored rounded to bf16. */
int vmoe_expert_fwd(const vmoe_problem *p, const void *xe, const void *w1, const void *w2,
                    const int32_t *load, void *h, void *a, void *ye, void *cuda_stream);

/* Device bytes of scratch vmoe_expert_bwd needs for `p`, or 0 if `p` is
 * invalid.  Host only.  It holds dH: T*E*C*d_ff fp32 elements for fp32
 * problems; for bf16, 2*T*E*C*d_ff bf16 elements, dH kept as a bf16 value plus
 * its bf16 residual so the weight gradients of small groups stay accurate. */
size_t vmoe_expert_bwd_workspace_size(const vmoe_problem *p);

/* The smallest workspace vmoe_expert_bwd accepts for `p`, or 0 if `p` is
 * invalid.  Host only.  fp32: the full size above.  bf16: one group's dH (2C
 * rows, rounded up to 8) plus 8*T*E bytes (rounded up to 256) for the plan of a
 * sliced run -- see vmoe_expert_bwd. */
size_t vmoe_expert_bwd_min_workspace_size(const vmoe_problem *p);

/* Expert FFN backward (adaptation of the expert weights, Section 3.1), the
 * gradient of <dY, y> through the expert path with routing and gates fixed:
 *   dH = (dYe W2^T) * GELU'(H), dXe = dH W1^T, dW1 = Xe^T dH, dW2 = A^T dYe,
 * the weight gradients summing over each group's rows s < load[g].
 *   xe [T,E,C,d], h, a [T,E,C,f] (from vmoe_expert_fwd), w1, w2, dye [T,E,C,d]
 *   (= vmoe_dispatch(dY, gate)), load [T,E]
 *   dxe [T,E,C,d] out (rows >= load not written), dw1 [T,E,d,f] out, dw2 [T,E,f,d] out
 *   (every element written; zero for a group with load 0)
 *   Rows s >= load[g] of xe, h, a and dye are padding: their contents (NaN
 *   included) reach no output.
 *   workspace: caller-owned device scratch, 16-byte aligned, its contents
 *   clobbered.  With vmoe_expert_bwd_workspace_size(p) bytes or more, dH of
 *   every group fits and the call is asynchronous.  bf16 problems also accept
 *   less, down to vmoe_expert_bwd_min_workspace_size(p): the groups are then
 *   placed in slices whose dH fits (the cross-task DP of vmoe_plan_slices,
 *   Section 3.2.1, each group's footprint its dH rows, its lifespan its load)
 *   and dA, dX and dW1 run slice by slice.  That path reads `load` back to the
 *   host first and synchronises `cuda_stream` (once); it then launches dW2 and
 *   plans one slice at a time, each slice's kernels queued as soon as it is
 *   placed, and returns when the last slice is queued.  The results are
 *   bitwise the same either way.  Less than the minimum, or NULL, returns
 *   VMOE_ERR_INVALID. */
int vmoe_expert_bwd(const vmoe_problem *p, const void *xe, const void *h, const void *a,
                    const void *w1, const void *w2, const void *dye, const int32_t *load,
                    void *dxe, void *dw1, void *dw2, void *workspace, size_t workspace_bytes,
                    void *cuda_stream);

/* Size in bytes of the device array behind vmoe_expert_bwd_static_scratch. */
#define VMOE_STATIC_SCRATCH_BYTES (64u << 20)

/* vmoe_expert_bwd without a caller-supplied workspace, for callers that cannot
 * allocate device memory: a plug-in whose host framework owns every device
 * buffer, or a deployment that allows no device allocation after start-up.
 * The paper has no counterpart; this is a packaging choice of the library.
 *   Arguments, layouts and results are those of vmoe_expert_bwd.  The dH
 *   scratch is a 64 MiB array compiled into the library, which every GPU that
 *   loads the library holds until the process exits; the call itself allocates
 *   nothing.  When vmoe_expert_bwd_workspace_size(p) <= VMOE_STATIC_SCRATCH_BYTES,
 *   dH of every group fits and the call is asynchronous like vmoe_expert_bwd.
 *   Otherwise a bf16 problem runs in slices planned to fit the array (as
 *   vmoe_expert_bwd with a smaller workspace): that path reads `load` back to
 *   the host and synchronises `cuda_stream`.  The call returns
 *   VMOE_ERR_UNSUPPORTED, with nothing launched, only when even
 *   vmoe_expert_bwd_min_workspace_size(p) exceeds the array: an fp32 problem
 *   whose dH is larger than the array, or a bf16 problem one of whose groups
 *   alone does not fit.  The first call on a device looks up the array's
 *   device address (cudaGetSymbolAddress) with that device current and caches
 *   it; make that first call before any stream capture.  Every call on a
 *   device shares the one array, which keeps whatever the last call left in
 *   it, so calls whose kernels overlap on the GPU (other streams, other host
 *   threads) race and corrupt each other's dH; issue them in order on one
 *   stream. */
int vmoe_expert_bwd_static_scratch(const vmoe_problem *p, const void *xe, const void *h,
                                   const void *a, const void *w1, const void *w2, const void *dye,
                                   const int32_t *load, void *dxe, void *dw1, void *dw2,
                                   void *cuda_stream);

/* Attention experts (Section 2.1: V-MoE expertizes the ViT's attention as well
 * as its MLP; Section 3.2.1's memory estimator gives such an expert buffers of
 * order T d_k for Q / K / V and T^2 for the scores).  The paper gives no more;
 * the library's reading: each (task, expert) group g owns W_qkv [d, 3 H 64]
 * (column blocks Q | K | V, head h at columns h * 64 of each) and W_o [H 64, d],
 * and runs H-head softmax attention, head dimension 64, among its L = load[g]
 * routed tokens only (the rows [0, L) of xe, as dispatched by vmoe_dispatch):
 *   QKV = Xe W_qkv;  per head  S = Q_h K_h^T / 8,  P = softmax over the L keys
 *   (row maximum subtracted),  O_h = P V_h;  Ye = O W_o,
 * then vmoe_combine gate-weights Ye back to token order as for the FFN.
 * bf16 only, H even, d % 128 == 0, C <= 512 (else VMOE_ERR_UNSUPPORTED);
 * p->d_ff is not used.  Sums accumulate in fp32; P is rounded to bf16 for the
 * P V product; no atomics.  Rows s >= load[g] of xe (and of dye, qkv, o in the
 * backward) are padding, reach no output and are not written.
 *   xe [T,E,C,d], wqkv [T,E,d,3H64], wo [T,E,H64,d] in; qkv [T,E,C,3H64],
 *   o [T,E,C,H64] bf16 and lse [T,E,H,C] fp32 (each row's log-sum-exp of the
 *   scaled scores, kept for the backward) out; ye [T,E,C,d] out. */
int vmoe_attn_expert_fwd(const vmoe_problem *p, int heads, const void *xe, const void *wqkv,
                         const void *wo, const int32_t *load, void *qkv, void *o, float *lse, void *ye,
                         void *cuda_stream);

/* Workspace of vmoe_attn_expert_bwd in bytes (dO and dQKV in bf16, then the row
 * sums D of dO * O in fp32), or 0 for an invalid or unsupported problem. */
size_t vmoe_attn_expert_bwd_workspace_size(const vmoe_problem *p, int heads);

/* Backward of vmoe_attn_expert_fwd with routing and gates fixed: the gradient
 * of <dYe, Ye> per group,
 *   dO = dYe W_o^T,  dW_o = O^T dYe,  D = rowsum(dO * O) per head,
 *   dS = P * (dO_h V_h^T - D),  dQ_h = dS K_h / 8,  dK_h = dS^T Q_h / 8,  dV_h = P^T dO_h,
 *   dXe = dQKV W_qkv^T,  dW_qkv = Xe^T dQKV,
 * P rebuilt from qkv and lse, D formed from the stored o.  The attention core's
 * products take fp16 operands, each staged tile of Q, K, V and dO scaled by a
 * power of two (exact for bf16 values), so P and dS enter dV, dQ and dK with 11
 * significant bits; for C > 128, dQ = dS K instead takes dS as a bf16 value
 * plus its bf16 residual.  Sums accumulate in fp32.  Inputs as written by the
 * forward (xe, qkv, o, lse) and dye [T,E,C,d] (vmoe_dispatch of dY with the
 * gates); outputs dxe [T,E,C,d]
 * (rows >= load not written), dwqkv [T,E,d,3H64] and dwo [T,E,H64,d] (zero for an
 * empty group).  workspace: caller-owned device scratch of at least
 * vmoe_attn_expert_bwd_workspace_size(p, heads) bytes (else VMOE_ERR_INVALID),
 * its contents clobbered.  Asynchronous on `cuda_stream`. */
int vmoe_attn_expert_bwd(const vmoe_problem *p, int heads, const void *xe, const void *qkv,
                         const void *o, const float *lse, const void *wqkv, const void *wo,
                         const void *dye, const int32_t *load, void *dxe, void *dwqkv, void *dwo,
                         void *workspace, size_t workspace_bytes, void *cuda_stream);

/* Combine back to token order: dst[t,n,:] = sum over kept choices j (slot >= 0)
 * of w * src[t, expert_idx_j, slot_j, :], w = weight[t,n,j] or 1 if NULL,
 * summed in fp32 in the order j = 0..k-1 and rounded once; a token with every
 * choice dropped gets zero.
 *   src [T,E,C,d], weight [T,N,k] fp32 nullable, expert_idx/slot [T,N,k],
 *   dst [T,N,d] out.  The forward uses weight = gate, the backward (dX) NULL. */
int vmoe_combine(const vmoe_problem *p, const void *src, const float *weight,
                 const int32_t *expert_idx, const int32_t *slot, void *dst, void *cuda_stream);

/* Router backward (Section 3.1 adapts the visual module, its gating network
 * included; Section 2.1 defines the gates as a softmax of the router logits).
 * With the routing held fixed (expert_idx, slot from vmoe_route), the gradient
 * of <dY, y> with y = sum_j gate_j Ye[e_j, s_j]:
 *   dgate[t,n,j]   = <dY[t,n], Ye[t,e_j,s_j]> for a kept choice, 0 if dropped;
 *   dlogits[t,n,e] = softmax backward: with s = sum_j gate_j dgate_j,
 *     renormalised gates:  dlogits[e_j] = gate_j (dgate_j - s), 0 elsewhere;
 *     VMOE_NO_RENORM:      dlogits[e]   = p_e (dgate(e) - s), p = softmax(logits)
 *                          and dgate(e) = dgate_j if e = e_j, else 0;
 *   dw_router[t]   = x[t]^T dlogits[t]      (sum over the N tokens of task t);
 *   dbias[t,e]     = sum_n dlogits[t,n,e];
 *   dx[t,n,:]     += W_r[t] dlogits[t,n]    (summed in fp32, rounded once).
 * Inputs: x, dY [T,N,d] and Ye [T,E,C,d] in p->dtype (Ye is the expert output
 * of vmoe_expert_fwd); w_router [T,d,E], logits [T,N,E], gate [T,N,k] fp32;
 * expert_idx, slot [T,N,k] int32.  w_router may be NULL only when dx is NULL;
 * logits is read only with VMOE_NO_RENORM (else it may be NULL).
 * Outputs (overwritten): dgate [T,N,k], dlogits [T,N,E], dw_router [T,d,E]
 * fp32; dbias [T,E] fp32, nullable.  dx [T,N,d] in p->dtype is read and
 * updated in place (the dX of vmoe_combine, which then holds the input
 * gradient through both the experts and the router); NULL skips it.
 * Sums run in fixed orders; no atomics. */
int vmoe_router_bwd(const vmoe_problem *p, const void *x, const float *w_router,
                    const float *logits, const int32_t *expert_idx, const float *gate,
                    const int32_t *slot, const void *dy, const void *ye, float *dgate,
                    float *dlogits, float *dw_router, float *dbias, void *dx,
                    void *cuda_stream);

/* Cross-task slice planner (Section 3.2.1, fragmentation-aware expert
 * grouping; host code, no GPU).  Items (experts) i = 0..n-1 have a memory
 * footprint weight[i] >= 0 and a lifespan lifespan[i]; the value of an item is
 * v_i = weight[i] / M - eta * lifespan[i], M = budget if budget > 0, else
 * capacity.  A 0/1-knapsack DP, dp[i][j] = max(dp[i-1][j], dp[i-1][j - w_i] +
 * v_i), picks the slice of largest total value whose weight fits `capacity`;
 * the chosen items leave and the DP runs again until every item is placed.
 * Items enter the DP in shortest-job-first order (lifespan, then index) and
 * keep that order inside a slice; an item is taken only when strictly better;
 * if nothing is chosen, the first remaining item forms a slice alone;
 * zero-weight items join the first slice.
 * Output: order[n], the items slice by slice; slice_start[n + 1], where slice s
 * is order[slice_start[s] .. slice_start[s + 1]).  Returns the number of slices,
 * VMOE_ERR_INVALID (null pointers, negative weight, NaN lifespan) or
 * VMOE_ERR_UNSUPPORTED (an item heavier than capacity, or a DP table above 2^30
 * entries). */
int vmoe_plan_slices(int n, const int64_t *weight, const double *lifespan, int64_t capacity,
                     double eta, double budget, int32_t *order, int32_t *slice_start);

/* Resource shares of co-running experts (Section 3.2.2, lifespan-aware
 * aligning; host code, no GPU): the fill-clamp-refill allocation of `budget`
 * units among n experts -- each is seeded with minimum[i]; what is left is
 * shared out in proportion to work[i] among the experts below their
 * saturation[i]; an expert above its saturation is clamped to it and what it
 * gave up is shared out again, until nothing is left or every expert with work
 * is saturated.  An expert with work 0 keeps its minimum.  The real-valued
 * shares are then rounded to whole units: floored, and the units still
 * missing from their total given one each to the largest fractional parts
 * (ties to the lower index), so minimum[i] <= shares[i] <= saturation[i].
 * float64 arithmetic, sums in index order.
 * Output: shares[n].  Returns the number of units allocated (budget, or less
 * when the saturations do not reach it), VMOE_ERR_INVALID (null pointers,
 * negative or NaN work, negative minimum, saturation below minimum) or
 * VMOE_ERR_UNSUPPORTED (the minima exceed the budget). */
int vmoe_plan_shares(int n, const double *work, const int32_t *minimum, const int32_t *saturation,
                     int32_t budget, int32_t *shares);

/* Device status word of the current device: 0 when clean, otherwise a
 * vmoe_status (VMOE_ERR_DEVICE_TIMEOUT after a kernel gave up a bounded
 * wait).  Synchronises the current device.  `reset` != 0 clears the word. */
int vmoe_device_status(int reset);

/* Self-test of the failure path: launches one kernel that waits on a device
 * barrier nothing ever signals, through the same bounded wait the grouped GEMM
 * uses, and gives up after `limit_ns` nanoseconds (1 ns .. 1 s).  The wait
 * running out sets the device status word to VMOE_ERR_DEVICE_TIMEOUT (read and
 * cleared with vmoe_device_status) and the kernel returns normally, leaving the
 * context usable.  Returns VMOE_OK after the launch, VMOE_ERR_INVALID for a
 * limit out of range. */
int vmoe_selftest_bounded_wait(long long limit_ns, void *cuda_stream);

/* Kernel trace (host-side tracing aid).  While enabled on the calling host
 * thread, every kernel the library launches is bracketed by two CUDA events
 * recorded on its stream; at most `max_records` launches are kept.
 * vmoe_trace_disable stops recording and returns the number of records;
 * vmoe_trace_get synchronises on record i and returns its kernel name (static
 * storage) and duration in milliseconds.  Returns VMOE_OK or a vmoe_status. */
int vmoe_trace_enable(int max_records);
int vmoe_trace_disable(void);
int vmoe_trace_get(int i, const char **kernel_name, float *ms);

#ifdef __cplusplus
}
#endif
#endif /* VMOE_H */
