/*
 * vmoe_oracle.c -- TEST INFRASTRUCTURE, NOT PRODUCT CODE.
 *
 * A plain, slow, fp64 CPU definition of one adaptation step of T concurrent
 * V-MoE expert layers (AdaSprite, arxiv 2608.16188):
 *   router logits -> softmax + top-k gating -> per-expert capacity scan ->
 *   dispatch into [T,E,C,d] expert buffers -> expert FFN (Linear-GELU-Linear)
 *   forward -> weighted combine back to token order, the backward of the
 *   expert path (dX, dW1, dW2) with routing and gates held constant, and the
 *   router backward (dgate, dlogits, dW_r, dbias and the router's share of dX)
 *   with the routing held fixed.
 *
 * Only the test suite, the smoke check and the benchmark's CPU-baseline leg
 * may load this file.  It shares no code, header or constant with the CUDA
 * library; every loop below is the textbook definition written out, with no
 * blocking, fusion or reordering of any sum.  OpenMP only splits loops over
 * independent tokens or (task, expert) groups; no reduction order changes.
 *
 * Where the paper is silent, the reading taken is stated at the function
 * (the paper prints no gating formula, no capacity formula and no worked
 * example; it cites V-MoE and Switch routing for them).
 *
 * Layouts (row-major, contiguous):
 *   x, y, dY, dX : [T, N, d]          W_r : [T, d, E]      bias : [T, E]
 *   logits       : [T, N, E]          idx, gate, slot : [T, N, k]
 *   load         : [T, E]             Xe, Ye, dYe, dXe : [T*E, C, d]
 *   H, A, dH     : [T*E, C, f]        W1, dW1 : [T*E, d, f]   W2, dW2 : [T*E, f, d]
 * Rows >= load of the per-group activation buffers are written as zero here.
 */
#include <math.h>
#include <stdint.h>
#include <stddef.h>
#include <string.h>

#define ORACLE_FLAG_NO_RENORM 2u
#define ORACLE_FLAG_GELU_TANH 4u

/* Per-expert capacity.  Challenge #1 (Section 1) and Section 2.3.1 name
 * "capacity limits" (Switch routing) as the standard way to bound expert load
 * but print no formula.  Reading: C = ceil(cf * k * N / E), clamped to [1, N],
 * evaluated in double as ((cf * k) * N) / E; an explicit positive override
 * wins. */
int oracle_capacity(int N, int E, int k, double capacity_factor, int capacity_override)
{
    if (capacity_override > 0) return capacity_override;
    double c = ceil(capacity_factor * (double)k * (double)N / (double)E);
    if (c < 1.0) c = 1.0;
    if (c > (double)N) c = (double)N;
    return (int)c;
}

/* Router logits (Section 2.1: tokens are routed "to the most relevant
 * experts"; each task has its own router, Section 2.2 keeps model-specific
 * parts per model): logits[t,n,e] = sum_i x[t,n,i] * W_r[t,i,e] + bias[t,e]. */
void oracle_router_logits(int T, int N, int d, int E, const double *x, const double *w_router,
                          const double *bias /* nullable */, double *logits)
{
    long total = (long)T * N;
#pragma omp parallel for schedule(static)
    for (long tn = 0; tn < total; ++tn) {
        int t = (int)(tn / N);
        const double *xr = x + tn * d;
        const double *wr = w_router + (long)t * d * E;
        for (int e = 0; e < E; ++e) {
            double s = 0.0;
            for (int i = 0; i < d; ++i) s += xr[i] * wr[(long)i * E + e];
            if (bias) s += bias[(long)t * E + e];
            logits[tn * E + e] = s;
        }
    }
}

/* Softmax + top-k gating for one token (Section 2.1 routing; the formula is
 * V-MoE's, which the paper cites without restating).  Readings:
 *  - the k experts are the k largest logits, taken one at a time, ties to the
 *    lowest expert index (selection on logits, not on rounded probabilities);
 *  - p = softmax over all E logits with the maximum subtracted;
 *  - gate_j = p[e_j] / sum_{i<k} p[e_i] (renormalised top-k mass), or p[e_j]
 *    when ORACLE_FLAG_NO_RENORM is set (V-MoE's own convention). */
static void topk_gate_one(int E, int k, unsigned flags, const double *l, int32_t *idx, double *gate)
{
    double mx = l[0];
    for (int e = 1; e < E; ++e)
        if (l[e] > mx) mx = l[e];
    double sum = 0.0;
    for (int e = 0; e < E; ++e) sum += exp(l[e] - mx);

    for (int j = 0; j < k; ++j) {
        int best = -1;
        for (int e = 0; e < E; ++e) {
            int taken = 0;
            for (int i = 0; i < j; ++i)
                if (idx[i] == e) taken = 1;
            if (taken) continue;
            if (best < 0 || l[e] > l[best]) best = e; /* strict '>' keeps the lower index on ties */
        }
        idx[j] = best;
    }
    double kept = 0.0;
    for (int j = 0; j < k; ++j) kept += exp(l[idx[j]] - mx) / sum;
    for (int j = 0; j < k; ++j) {
        double p = exp(l[idx[j]] - mx) / sum;
        gate[j] = (flags & ORACLE_FLAG_NO_RENORM) ? p : p / kept;
    }
}

/* Routing for all tasks: top-k gating per token, then the capacity scan.
 * Section 3.3.1 states that tokens are assigned to experts sequentially; with
 * capacity limits (Challenge #1) the overflow is dropped.  Reading of the
 * order: choice-major -- every token's first choice in token order, then every
 * token's second choice, and so on.  The s-th assignment that reaches expert
 * e gets slot s if s < C, else slot -1 (dropped); load[t,e] = min(count, C). */
void oracle_route(int T, int N, int E, int k, int C, unsigned flags, const double *logits,
                  int32_t *idx, double *gate, int32_t *slot, int32_t *load)
{
    long total = (long)T * N;
#pragma omp parallel for schedule(static)
    for (long tn = 0; tn < total; ++tn)
        topk_gate_one(E, k, flags, logits + tn * E, idx + tn * k, gate + tn * k);

    for (int t = 0; t < T; ++t) {
        int32_t *cnt = load + (long)t * E;
        for (int e = 0; e < E; ++e) cnt[e] = 0;
        for (int j = 0; j < k; ++j) {
            for (int n = 0; n < N; ++n) {
                long a = ((long)t * N + n) * k + j;
                int e = idx[a];
                slot[a] = (cnt[e] < C) ? cnt[e] : -1;
                cnt[e] += 1;
            }
        }
        for (int e = 0; e < E; ++e)
            if (cnt[e] > C) cnt[e] = C;
    }
}

/* Dispatch (Section 3.2, expert parallelism over the merged pool of
 * Section 2.2): dst[t,e,s,:] = w * src[t,n,:] for the kept assignment (n, j)
 * with idx = e and slot = s, where w = weight[t,n,j] or 1 when weight is NULL.
 * Every other row of dst is zero. */
void oracle_dispatch(int T, int N, int d, int E, int k, int C, const double *src,
                     const double *weight /* nullable */, const int32_t *idx, const int32_t *slot,
                     double *dst)
{
    memset(dst, 0, sizeof(double) * (size_t)T * E * C * d);
    for (int t = 0; t < T; ++t)
        for (int n = 0; n < N; ++n)
            for (int j = 0; j < k; ++j) {
                long a = ((long)t * N + n) * k + j;
                if (slot[a] < 0) continue;
                double w = weight ? weight[a] : 1.0;
                double *row = dst + (((long)t * E + idx[a]) * C + slot[a]) * d;
                const double *in = src + ((long)t * N + n) * d;
                for (int i = 0; i < d; ++i) row[i] = w * in[i];
            }
}

/* GELU and its derivative.  The paper does not name the activation of the
 * expert MLP; reading: exact erf GELU, GELU(h) = h/2 * (1 + erf(h/sqrt 2)),
 * GELU'(h) = Phi(h) + h*phi(h); or the tanh form of Hendrycks & Gimpel with
 * its analytic derivative when ORACLE_FLAG_GELU_TANH is set. */
static double gelu(double h, unsigned flags)
{
    if (flags & ORACLE_FLAG_GELU_TANH) {
        double c = sqrt(2.0 / M_PI);
        return 0.5 * h * (1.0 + tanh(c * (h + 0.044715 * h * h * h)));
    }
    return 0.5 * h * (1.0 + erf(h / sqrt(2.0)));
}

static double gelu_deriv(double h, unsigned flags)
{
    if (flags & ORACLE_FLAG_GELU_TANH) {
        double c = sqrt(2.0 / M_PI);
        double u = c * (h + 0.044715 * h * h * h);
        double th = tanh(u);
        return 0.5 * (1.0 + th) + 0.5 * h * (1.0 - th * th) * c * (1.0 + 3.0 * 0.044715 * h * h);
    }
    double Phi = 0.5 * (1.0 + erf(h / sqrt(2.0)));
    double phi = exp(-0.5 * h * h) / sqrt(2.0 * M_PI);
    return Phi + h * phi;
}

/* Expert FFN forward per (task, expert) group g with L = load[g] rows
 * (Section 2.1: the MLP block of a ViT becomes a set of experts; no biases,
 * reading): H = Xe W1, A = GELU(H), Ye = A W2.  Rows >= L are zero. */
void oracle_expert_fwd(int G, int C, int d, int f, unsigned flags, const double *xe,
                       const double *w1, const double *w2, const int32_t *load,
                       double *h, double *a, double *ye)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int g = 0; g < G; ++g) {
        int L = load[g];
        const double *X = xe + (long)g * C * d;
        const double *W1 = w1 + (long)g * d * f;
        const double *W2 = w2 + (long)g * f * d;
        double *Hg = h + (long)g * C * f;
        double *Ag = a + (long)g * C * f;
        double *Yg = ye + (long)g * C * d;
        memset(Hg, 0, sizeof(double) * (size_t)C * f);
        memset(Ag, 0, sizeof(double) * (size_t)C * f);
        memset(Yg, 0, sizeof(double) * (size_t)C * d);
        for (int s = 0; s < L; ++s) {
            for (int i = 0; i < d; ++i) { /* H[s,:] += X[s,i] * W1[i,:] */
                double xv = X[(long)s * d + i];
                for (int c = 0; c < f; ++c) Hg[(long)s * f + c] += xv * W1[(long)i * f + c];
            }
            for (int c = 0; c < f; ++c) Ag[(long)s * f + c] = gelu(Hg[(long)s * f + c], flags);
            for (int c = 0; c < f; ++c) { /* Ye[s,:] += A[s,c] * W2[c,:] */
                double av = Ag[(long)s * f + c];
                for (int i = 0; i < d; ++i) Yg[(long)s * d + i] += av * W2[(long)c * d + i];
            }
        }
    }
}

/* Combine: dst[t,n,:] = sum over kept choices j (slot >= 0), in order
 * j = 0..k-1, of w * src[t, idx_j, slot_j, :], w = weight[t,n,j] or 1 when
 * weight is NULL.  A token whose every choice was dropped gets zero. */
void oracle_combine(int T, int N, int d, int E, int k, int C, const double *src,
                    const double *weight /* nullable */, const int32_t *idx, const int32_t *slot,
                    double *dst)
{
    long total = (long)T * N;
#pragma omp parallel for schedule(static)
    for (long tn = 0; tn < total; ++tn) {
        int t = (int)(tn / N);
        double *out = dst + tn * d;
        for (int i = 0; i < d; ++i) out[i] = 0.0;
        for (int j = 0; j < k; ++j) {
            long a = tn * k + j;
            if (slot[a] < 0) continue;
            double w = weight ? weight[a] : 1.0;
            const double *row = src + (((long)t * E + idx[a]) * C + slot[a]) * d;
            for (int i = 0; i < d; ++i) out[i] += w * row[i];
        }
    }
}

/* Expert FFN backward per group (specification-based tuning, Section 3.1:
 * only the visual module is adapted, so the expert weights get gradients).
 * It is the gradient of <dY, y> through the expert path with gates and
 * routing held constant, given dYe = dispatch(dY, gate):
 *   dA = dYe W2^T, dH = dA * GELU'(H), dXe = dH W1^T,
 *   dW1 = Xe^T dH, dW2 = A^T dYe  (sums over the L = load[g] rows only).
 * Rows >= L of dH and dXe are zero; a group with L = 0 gets dW1 = dW2 = 0. */
void oracle_expert_bwd(int G, int C, int d, int f, unsigned flags, const double *xe,
                       const double *h, const double *a, const double *w1, const double *w2,
                       const double *dye, const int32_t *load, double *dh, double *dxe,
                       double *dw1, double *dw2)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int g = 0; g < G; ++g) {
        int L = load[g];
        const double *X = xe + (long)g * C * d;
        const double *Hg = h + (long)g * C * f;
        const double *Ag = a + (long)g * C * f;
        const double *W1 = w1 + (long)g * d * f;
        const double *W2 = w2 + (long)g * f * d;
        const double *DY = dye + (long)g * C * d;
        double *DH = dh + (long)g * C * f;
        double *DX = dxe + (long)g * C * d;
        double *DW1 = dw1 + (long)g * d * f;
        double *DW2 = dw2 + (long)g * f * d;
        memset(DH, 0, sizeof(double) * (size_t)C * f);
        memset(DX, 0, sizeof(double) * (size_t)C * d);
        memset(DW1, 0, sizeof(double) * (size_t)d * f);
        memset(DW2, 0, sizeof(double) * (size_t)f * d);
        for (int s = 0; s < L; ++s) {
            for (int c = 0; c < f; ++c) { /* dA[s,c] = sum_i dYe[s,i] W2[c,i] */
                double acc = 0.0;
                for (int i = 0; i < d; ++i) acc += DY[(long)s * d + i] * W2[(long)c * d + i];
                DH[(long)s * f + c] = acc * gelu_deriv(Hg[(long)s * f + c], flags);
            }
            for (int i = 0; i < d; ++i) { /* dXe[s,i] = sum_c dH[s,c] W1[i,c] */
                double acc = 0.0;
                for (int c = 0; c < f; ++c) acc += DH[(long)s * f + c] * W1[(long)i * f + c];
                DX[(long)s * d + i] = acc;
            }
        }
        for (int i = 0; i < d; ++i) /* dW1[i,c] = sum_s Xe[s,i] dH[s,c] */
            for (int s = 0; s < L; ++s) {
                double xv = X[(long)s * d + i];
                for (int c = 0; c < f; ++c) DW1[(long)i * f + c] += xv * DH[(long)s * f + c];
            }
        for (int c = 0; c < f; ++c) /* dW2[c,i] = sum_s A[s,c] dYe[s,i] */
            for (int s = 0; s < L; ++s) {
                double av = Ag[(long)s * f + c];
                for (int i = 0; i < d; ++i) DW2[(long)c * d + i] += av * DY[(long)s * d + i];
            }
    }
}

/* Number of threads the OpenMP runtime would use (reported by the CPU
 * baseline). */
int oracle_num_threads(void)
{
#ifdef _OPENMP
    extern int omp_get_max_threads(void);
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Router backward (the adaptation gradient of the gating network: the router
 * belongs to the visual module that specification-based tuning adapts,
 * Section 3.1).  Routing -- the chosen experts and the slots -- is piecewise
 * constant in the logits and is held fixed; the gates are differentiable:
 *   dgate_j = <dY[t,n], Ye[t, e_j, s_j]> for a kept choice, 0 for a dropped one
 *             (y does not depend on a dropped choice's gate);
 *   renormalised gates (the default) are the softmax of the k selected logits,
 *     dlogit[e_j] = w_j (dgate_j - sum_i w_i dgate_i), 0 for unselected experts;
 *   V-MoE gates (ORACLE_FLAG_NO_RENORM) are the full softmax p,
 *     dlogit[e] = p_e (g_e - sum_j w_j dgate_j), g_e = dgate_j if e = e_j else 0;
 *   logits = x W_r + bias, so dW_r[t] = sum_n x[t,n]^T dlogit[t,n],
 *     dbias[t] = sum_n dlogit[t,n], dx_router[t,n] = W_r[t] dlogit[t,n]. */
void oracle_router_bwd(int T, int N, int d, int E, int k, int C, unsigned flags, const double *x,
                       const double *w_router, const double *logits, const int32_t *idx,
                       const double *gate, const int32_t *slot, const double *dy, const double *ye,
                       double *dgate, double *dlogits, double *dw_router, double *dbias,
                       double *dx_router)
{
    long total = (long)T * N;
#pragma omp parallel for schedule(static)
    for (long tn = 0; tn < total; ++tn) {
        int t = (int)(tn / N);
        const double *dyr = dy + tn * d;
        double *dl = dlogits + tn * E;
        double *dg = dgate + tn * k;
        for (int j = 0; j < k; ++j) {
            long a = tn * k + j;
            dg[j] = 0.0;
            if (slot[a] < 0) continue;
            const double *row = ye + (((long)t * E + idx[a]) * C + slot[a]) * d;
            for (int i = 0; i < d; ++i) dg[j] += dyr[i] * row[i];
        }
        double s = 0.0;
        for (int j = 0; j < k; ++j) s += gate[tn * k + j] * dg[j];
        for (int e = 0; e < E; ++e) dl[e] = 0.0;
        if (flags & ORACLE_FLAG_NO_RENORM) {
            const double *l = logits + tn * E;
            double mx = l[0];
            for (int e = 1; e < E; ++e)
                if (l[e] > mx) mx = l[e];
            double sum = 0.0;
            for (int e = 0; e < E; ++e) sum += exp(l[e] - mx);
            for (int e = 0; e < E; ++e) {
                double g = 0.0;
                for (int j = 0; j < k; ++j)
                    if (idx[tn * k + j] == e) g = dg[j];
                dl[e] = exp(l[e] - mx) / sum * (g - s);
            }
        } else {
            for (int j = 0; j < k; ++j) dl[idx[tn * k + j]] = gate[tn * k + j] * (dg[j] - s);
        }
        double *dxr = dx_router + tn * d;
        const double *wr = w_router + (long)t * d * E;
        for (int i = 0; i < d; ++i) {
            double acc = 0.0;
            for (int e = 0; e < E; ++e) acc += wr[(long)i * E + e] * dl[e];
            dxr[i] = acc;
        }
    }
#pragma omp parallel for schedule(static)
    for (int t = 0; t < T; ++t) {
        double *dw = dw_router + (long)t * d * E;
        for (long i = 0; i < (long)d * E; ++i) dw[i] = 0.0;
        for (int e = 0; e < E; ++e) dbias[(long)t * E + e] = 0.0;
        for (int n = 0; n < N; ++n) {
            const double *xr = x + ((long)t * N + n) * d;
            const double *dl = dlogits + ((long)t * N + n) * E;
            for (int i = 0; i < d; ++i)
                for (int e = 0; e < E; ++e) dw[(long)i * E + e] += xr[i] * dl[e];
            for (int e = 0; e < E; ++e) dbias[(long)t * E + e] += dl[e];
        }
    }
}
