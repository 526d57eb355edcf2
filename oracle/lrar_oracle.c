/*
 * lrar_oracle.c -- fp64 CPU oracle for the depth-attention mix of
 * "Low-Rank Attention Residuals" (arxiv 2607.09694).
 *
 * TEST INFRASTRUCTURE ONLY.  This is the plain, slow, obviously-correct
 * statement of what the GPU library computes, used to check it.  Only the
 * test suite, the smoke check and the benchmark's CPU-baseline leg load it.
 * It shares no code, header, table or helper with the CUDA library, and the
 * CUDA library never calls it.
 *
 * Every quantity is evaluated in double precision, token by token, straight
 * from the paper's definitions:
 *   Eq. (8)  lr_key_norm        kbar_i = RMSNorm(k_i), parameter-free (§3.2, App. A.5)
 *   Eq. (9)  lr_attnres_weight  alpha_i = softmax_i(q^T kbar_i), no temperature (§3.2)
 *   Eq. (10) lr_attnres_output  h = sum_i alpha_i o_i (§3.2)
 *   Eq. (12) fused_projection   P-LR keys are a separate input tensor of the mix
 *                                (§3.3); oracle_projection evaluates Eq. (11)-(12)
 *                                itself: [o; k] = [W_O; W_K] a
 *   Eq. (14) sliced_key         S-LR key = last r coordinates of o_i (§3.4)
 *   Eq. (2)  attnres_weight     AttnRes key = o_i itself, r = d (§3.1)
 *   Eq. (5), (6)                Block AttnRes summaries are plain sums (§3.1)
 * The paper prints no gradient formulas.  The backward functions apply the
 * chain rule to those equations one step at a time: the vector-Jacobian
 * product of the weighted sum, of the softmax, of the dot-product score and
 * of the RMSNorm, in that order.
 *
 * Readings where the paper is silent (all explicit arguments here):
 *   - the RMSNorm epsilon is an argument (the paper states none);
 *   - RMSNorm has no gain (the parameter-free convention of App. A.5);
 *   - scores carry no 1/sqrt(r) temperature (Eq. 9 is a plain dot product);
 *   - tail_r is 0-based [d-r, d) (Eq. 14's 1-based d-r+1..d);
 *   - gradients flow through the keys (no stop-gradient is mentioned).
 *
 * Element types: 0 = float64, 1 = float32, 2 = bfloat16 (raw 16-bit words).
 * Widening to double is exact in every case.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum { OR_FULL = 0, OR_SLICED = 1, OR_PROJECTED = 2 };
enum { OR_F64 = 0, OR_F32 = 1, OR_BF16 = 2 };

/* Decode stored element idx of an array of the given type.  A bfloat16 word
 * is the upper half of an IEEE binary32 word. */
static double elem(const void *base, int dtype, int64_t idx) {
    if (dtype == OR_F64) return ((const double *)base)[idx];
    if (dtype == OR_F32) return (double)((const float *)base)[idx];
    uint32_t w = (uint32_t)((const uint16_t *)base)[idx] << 16;
    float f;
    memcpy(&f, &w, sizeof f);
    return (double)f;
}

static int nthreads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

static int thread_id(void) {
#ifdef _OPENMP
    return omp_get_thread_num();
#else
    return 0;
#endif
}

void oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

int oracle_get_threads(void) { return nthreads(); }

/* Value o_i of token x, coordinate j (values are stacked [n, T, d]). */
static double value_at(const void *values, int dtype, int64_t T, int d, int i, int64_t x, int j) {
    return elem(values, dtype, ((int64_t)i * T + x) * d + j);
}

/* Routing key k_i of token x:
 *   PROJECTED: the learned key of Eq. (12), stored [n, T, r];
 *   SLICED:    tail_r(o_i) of Eq. (14), coordinates d-r..d-1 of the value;
 *   FULL:      the AttnRes key of Eq. (2), the whole value (r = d). */
static void fetch_key(int variant, int dtype, const void *values, const void *keys,
                      int64_t T, int d, int r, int i, int64_t x, double *k) {
    for (int j = 0; j < r; ++j) {
        if (variant == OR_PROJECTED)
            k[j] = elem(keys, dtype, ((int64_t)i * T + x) * r + j);
        else if (variant == OR_SLICED)
            k[j] = value_at(values, dtype, T, d, i, x, d - r + j);
        else
            k[j] = value_at(values, dtype, T, d, i, x, j);
    }
}

/* Eq. (8): parameter-free RMSNorm, kbar = k / sqrt(mean_j k_j^2 + eps).
 * Returns the scale rho = 1 / sqrt(mean_j k_j^2 + eps). */
static double rmsnorm(const double *k, int r, double eps, double *kbar) {
    double sumsq = 0.0;
    for (int j = 0; j < r; ++j) sumsq += k[j] * k[j];
    double rho = 1.0 / sqrt(sumsq / (double)r + eps);
    for (int j = 0; j < r; ++j) kbar[j] = rho * k[j];
    return rho;
}

/* Per-thread scratch for one token. */
typedef struct {
    double *k;      /* [n*r] raw keys      */
    double *kbar;   /* [n*r] normed keys   */
    double *rho;    /* [n]                 */
    double *s;      /* [n] scores          */
    double *alpha;  /* [n] weights         */
    double *g;      /* [n] dL/dalpha       */
    double *ds;     /* [n] dL/ds           */
    double *dk;     /* [r] dL/dk_i         */
    double *dh;     /* [d] upstream grad   */
} scratch_t;

static int scratch_alloc(scratch_t *w, int n, int d, int r) {
    w->k = malloc(sizeof(double) * (size_t)n * r);
    w->kbar = malloc(sizeof(double) * (size_t)n * r);
    w->rho = malloc(sizeof(double) * n);
    w->s = malloc(sizeof(double) * n);
    w->alpha = malloc(sizeof(double) * n);
    w->g = malloc(sizeof(double) * n);
    w->ds = malloc(sizeof(double) * n);
    w->dk = malloc(sizeof(double) * r);
    w->dh = malloc(sizeof(double) * d);
    return (w->k && w->kbar && w->rho && w->s && w->alpha && w->g && w->ds && w->dk && w->dh) ? 0 : -1;
}

static void scratch_free(scratch_t *w) {
    free(w->k); free(w->kbar); free(w->rho); free(w->s); free(w->alpha);
    free(w->g); free(w->ds); free(w->dk); free(w->dh);
}

/* Eq. (8)-(9) for one token: keys, RMSNorm, scores, two-pass softmax.
 * Returns lse = log sum_i exp(s_i). */
static double route_token(int variant, int dtype, const void *values, const void *keys,
                          const double *q, int n, int64_t T, int d, int r, double eps,
                          int64_t x, scratch_t *w) {
    for (int i = 0; i < n; ++i) {
        double *ki = w->k + (size_t)i * r;
        double *kbi = w->kbar + (size_t)i * r;
        fetch_key(variant, dtype, values, keys, T, d, r, i, x, ki);
        w->rho[i] = rmsnorm(ki, r, eps, kbi);
        double s = 0.0;
        for (int j = 0; j < r; ++j) s += q[j] * kbi[j];
        w->s[i] = s;
    }
    double m = w->s[0];
    for (int i = 1; i < n; ++i) if (w->s[i] > m) m = w->s[i];
    double Z = 0.0;
    for (int i = 0; i < n; ++i) Z += exp(w->s[i] - m);
    for (int i = 0; i < n; ++i) w->alpha[i] = exp(w->s[i] - m) / Z;
    return m + log(Z);
}

static int check_args(int variant, int dtype, const void *values, const void *keys, const double *q,
                      int n, int64_t T, int d, int r, double eps) {
    if (variant < OR_FULL || variant > OR_PROJECTED) return -1;
    if (dtype < OR_F64 || dtype > OR_BF16) return -1;
    if (!values || !q || n < 1 || T < 0 || d < 1 || r < 1 || r > d || !(eps > 0.0)) return -1;
    if (variant == OR_FULL && r != d) return -1;
    if (variant == OR_PROJECTED && !keys) return -1;
    return 0;
}

/*
 * Forward pass, Eq. (8)-(10), for the listed tokens (tokens == NULL: all T).
 *   values [n, T, d], keys [n, T, r] (PROJECTED only), q [r]
 *   h      [n_tok, d]   output (required)
 *   lse    [n_tok]      output, may be NULL
 *   alpha  [n_tok, n]   output, may be NULL
 */
int oracle_forward(int variant, int dtype, const void *values, const void *keys, const double *q,
                   int n, int64_t T, int d, int r, double eps,
                   const int64_t *tokens, int64_t n_tok,
                   double *h, double *lse, double *alpha) {
    if (check_args(variant, dtype, values, keys, q, n, T, d, r, eps)) return -1;
    if (!tokens) n_tok = T;
    if (n_tok < 0 || !h) return -1;
    int err = 0;
#pragma omp parallel reduction(| : err)
    {
        scratch_t w;
        int ok = scratch_alloc(&w, n, d, r) == 0;
        if (!ok) err |= 1;
        /* every thread reaches the work-sharing loop, even without scratch */
        {
#pragma omp for schedule(static)
            for (int64_t u = 0; u < n_tok; ++u) {
                int64_t x = tokens ? tokens[u] : u;
                if (!ok || x < 0 || x >= T) { err |= 1; continue; }
                double l = route_token(variant, dtype, values, keys, q, n, T, d, r, eps, x, &w);
                for (int j = 0; j < d; ++j) {           /* Eq. (10) */
                    double acc = 0.0;
                    for (int i = 0; i < n; ++i) acc += w.alpha[i] * value_at(values, dtype, T, d, i, x, j);
                    h[u * d + j] = acc;
                }
                if (lse) lse[u] = l;
                if (alpha) for (int i = 0; i < n; ++i) alpha[u * n + i] = w.alpha[i];
            }
        }
        scratch_free(&w);
    }
    return err ? -1 : 0;
}

/*
 * Backward pass: gradients of L = sum_x <dh_x, h_x> through Eq. (8)-(10)
 * for the listed tokens (tokens == NULL: all T).
 *   dh       [T, d]  upstream gradient, same element type as values
 *   dvalues  [n, n_tok, d] output or NULL (SLICED/FULL include the key path)
 *   dkeys    [n, n_tok, r] output or NULL (PROJECTED only)
 *   dq       [r] output or NULL: sum over the listed tokens
 *   ds       [n_tok, n] output or NULL: dL/ds_i (score gradients)
 */
int oracle_backward(int variant, int dtype, const void *values, const void *keys, const double *q,
                    int n, int64_t T, int d, int r, double eps, const void *dh,
                    const int64_t *tokens, int64_t n_tok,
                    double *dvalues, double *dkeys, double *dq, double *ds, double *dq_abs) {
    if (check_args(variant, dtype, values, keys, q, n, T, d, r, eps) || !dh) return -1;
    if (!tokens) n_tok = T;
    if (n_tok < 0) return -1;
    int nt = nthreads();
    /* per thread: r partial sums of dq, then r sums of |ds_i kbar_ij| (the
     * magnitude of the terms dq adds up, for judging its rounding) */
    double *dq_part = calloc((size_t)nt * 2 * r, sizeof(double));
    if (!dq_part) return -1;
    int err = 0;
#pragma omp parallel reduction(| : err)
    {
        scratch_t w;
        double *dqp = dq_part + (size_t)thread_id() * 2 * r;
        double *dqa = dqp + r;
        int ok = scratch_alloc(&w, n, d, r) == 0;
        if (!ok) err |= 1;
        /* every thread reaches the work-sharing loop, even without scratch */
        {
#pragma omp for schedule(static)
            for (int64_t u = 0; u < n_tok; ++u) {
                int64_t x = tokens ? tokens[u] : u;
                if (!ok || x < 0 || x >= T) { err |= 1; continue; }
                route_token(variant, dtype, values, keys, q, n, T, d, r, eps, x, &w);
                for (int j = 0; j < d; ++j) w.dh[j] = elem(dh, dtype, x * (int64_t)d + j);

                /* Eq. (10): h = sum_i alpha_i o_i, so dL/do_i = alpha_i dh and
                 * dL/dalpha_i = <dh, o_i>. */
                for (int i = 0; i < n; ++i) {
                    double g = 0.0;
                    for (int j = 0; j < d; ++j) g += w.dh[j] * value_at(values, dtype, T, d, i, x, j);
                    w.g[i] = g;
                }
                /* Eq. (9), softmax Jacobian: dL/ds_i = alpha_i (g_i - sum_k alpha_k g_k). */
                double gbar = 0.0;
                for (int k = 0; k < n; ++k) gbar += w.alpha[k] * w.g[k];
                for (int i = 0; i < n; ++i) w.ds[i] = w.alpha[i] * (w.g[i] - gbar);

                if (dvalues)
                    for (int i = 0; i < n; ++i)
                        for (int j = 0; j < d; ++j)
                            dvalues[((int64_t)i * n_tok + u) * d + j] = w.alpha[i] * w.dh[j];

                for (int i = 0; i < n; ++i) {
                    const double *ki = w.k + (size_t)i * r;
                    const double *kbi = w.kbar + (size_t)i * r;
                    double rho = w.rho[i];
                    /* Score s_i = q . kbar_i: dL/dq += ds_i kbar_i, dL/dkbar_i = ds_i q. */
                    for (int j = 0; j < r; ++j) {
                        dqp[j] += w.ds[i] * kbi[j];
                        dqa[j] += fabs(w.ds[i] * kbi[j]);
                    }
                    /* Eq. (8), RMSNorm: kbar = rho k with rho = (k.k/r + eps)^(-1/2),
                     * so d kbar_a / d k_b = rho [a==b] + k_a drho/dk_b and
                     * drho/dk_b = -rho^3 k_b / r.  Apply the transpose to dkbar. */
                    double k_dot_dkbar = 0.0;
                    for (int a = 0; a < r; ++a) k_dot_dkbar += ki[a] * (w.ds[i] * q[a]);
                    for (int b = 0; b < r; ++b)
                        w.dk[b] = rho * (w.ds[i] * q[b]) - (rho * rho * rho / (double)r) * ki[b] * k_dot_dkbar;
                    /* Route the key gradient to the tensor the key was read from. */
                    if (variant == OR_PROJECTED) {
                        if (dkeys)
                            for (int j = 0; j < r; ++j) dkeys[((int64_t)i * n_tok + u) * r + j] = w.dk[j];
                    } else if (dvalues) {
                        int off = (variant == OR_SLICED) ? d - r : 0;
                        for (int j = 0; j < r; ++j) dvalues[((int64_t)i * n_tok + u) * d + off + j] += w.dk[j];
                    }
                }
                if (ds) for (int i = 0; i < n; ++i) ds[u * n + i] = w.ds[i];
            }
        }
        scratch_free(&w);
    }
    for (int j = 0; j < r; ++j) {
        double acc = 0.0, mag = 0.0;
        for (int t = 0; t < nt; ++t) {
            acc += dq_part[(size_t)t * 2 * r + j];
            mag += dq_part[(size_t)t * 2 * r + r + j];
        }
        if (dq) dq[j] = acc;
        if (dq_abs) dq_abs[j] = mag;
    }
    free(dq_part);
    return err ? -1 : 0;
}

/*
 * Source-set sizes n_t = |S_t| for residual read site t in 1..M+1 (§3.1).
 * Full AttnRes, Eq. (4): S_t = {0, ..., t-1}.
 * Block AttnRes with c outputs per block: the embedding, each completed block
 * summary (Eq. 5), and the partial-block summary (Eq. 6) when it is non-empty.
 * Outputs o_1..o_{t-1} have been written before site t.
 */
int oracle_full_num_sources(int t) { return t; }

int oracle_block_num_sources(int t, int c) {
    if (t < 1 || c < 1) return -1;
    int written = t - 1;
    int completed = written / c;
    int partial = written - completed * c;
    return 1 + completed + (partial > 0 ? 1 : 0);
}

/*
 * Block AttnRes source stack at site t, Eq. (5)-(6):
 *   sources[0]   = o_0 (the embedding, its own source)
 *   sources[1+b] = sum of o_i over block b: members i = b*c+1 .. b*c+c
 * where the last slot is the partial block when (t-1) is not a multiple of c.
 *   outputs [t, T, w] holds o_0 .. o_{t-1}; sources [n_t, T, w] (double).
 * Works for values (w = d) and, under the P-LR reading that a summary's key
 * is the sum of its members' keys, for keys (w = r).  Returns n_t, or -1.
 */
int oracle_block_sources(int dtype, const void *outputs, int t, int64_t T, int w, int c, double *sources) {
    if (!outputs || !sources || t < 1 || T < 0 || w < 1 || c < 1) return -1;
    int nt = oracle_block_num_sources(t, c);
    memset(sources, 0, sizeof(double) * (size_t)nt * T * w);
    for (int i = 0; i < t; ++i) {
        int slot = (i == 0) ? 0 : 1 + (i - 1) / c;
        for (int64_t e = 0; e < T * (int64_t)w; ++e)
            sources[(int64_t)slot * T * w + e] += elem(outputs, dtype, (int64_t)i * T * w + e);
    }
    return nt;
}

/*
 * Gradient of the Block assembly: each output o_i receives the gradient of
 * the one summary it is summed into (o_0 receives that of slot 0).
 *   dsources [n_t, T, w], doutputs [t, T, w] (both double).
 */
int oracle_block_fanout(const double *dsources, int t, int64_t T, int w, int c, double *doutputs) {
    if (!dsources || !doutputs || t < 1 || T < 0 || w < 1 || c < 1) return -1;
    for (int i = 0; i < t; ++i) {
        int slot = (i == 0) ? 0 : 1 + (i - 1) / c;
        memcpy(doutputs + (int64_t)i * T * w, dsources + (int64_t)slot * T * w, sizeof(double) * (size_t)T * w);
    }
    return 0;
}

/*
 * Routing diagnostics of §4.5-4.6 for the listed tokens:
 *   neff  [n_tok]: N_eff = exp(H(alpha)), Eq. (16), with 0 log 0 = 0
 *   mean_alpha [n]: alpha averaged over the listed tokens (heatmap row)
 * Either output may be NULL.
 */
int oracle_diagnostics(int variant, int dtype, const void *values, const void *keys, const double *q,
                       int n, int64_t T, int d, int r, double eps,
                       const int64_t *tokens, int64_t n_tok, double *neff, double *mean_alpha) {
    if (check_args(variant, dtype, values, keys, q, n, T, d, r, eps)) return -1;
    if (!tokens) n_tok = T;
    if (n_tok < 0) return -1;
    double *alpha = malloc(sizeof(double) * (size_t)(n_tok > 0 ? n_tok : 1) * n);
    double *h = malloc(sizeof(double) * (size_t)(n_tok > 0 ? n_tok : 1) * d);
    if (!alpha || !h) { free(alpha); free(h); return -1; }
    int rc = oracle_forward(variant, dtype, values, keys, q, n, T, d, r, eps, tokens, n_tok, h, NULL, alpha);
    if (rc == 0) {
        for (int64_t u = 0; u < n_tok && neff; ++u) {
            double H = 0.0;
            for (int i = 0; i < n; ++i) {
                double a = alpha[u * n + i];
                if (a > 0.0) H -= a * log(a);
            }
            neff[u] = exp(H);
        }
        if (mean_alpha) {
            for (int i = 0; i < n; ++i) {
                double acc = 0.0;
                for (int64_t u = 0; u < n_tok; ++u) acc += alpha[u * n + i];
                mean_alpha[i] = n_tok > 0 ? acc / (double)n_tok : 0.0;
            }
        }
    }
    free(alpha);
    free(h);
    return rc;
}

/*
 * P-LR fused output projection, Eq. (11)-(12) (§3.3), for the listed tokens:
 *   y[u][j] = sum_c w[j][c] a[x_u][c],   j = 0..nrows-1,
 * where rows 0..d-1 of w are the ordinary output projection W_O (so y's first
 * d columns are the sub-layer output o) and rows d..d+r-1 are the key rows
 * W_K (the P-LR key k).  Eq. (13)'s embedding key is the case d = 0.
 *   a [T, m], w [nrows, m] (element type dtype), y [n_tok, nrows] float64.
 */
int oracle_projection(int dtype, const void *a, const void *w, int64_t T, int m, int nrows,
                      const int64_t *tokens, int64_t n_tok, double *y) {
    if (!a || !w || !y || T < 0 || m < 1 || nrows < 1) return -1;
    if (dtype < OR_F64 || dtype > OR_BF16) return -1;
    if (!tokens) n_tok = T;
    if (n_tok < 0) return -1;
    for (int64_t u = 0; u < n_tok; ++u)
        if (tokens && (tokens[u] < 0 || tokens[u] >= T)) return -1;
#pragma omp parallel for schedule(static)
    for (int64_t u = 0; u < n_tok; ++u) {
        const int64_t x = tokens ? tokens[u] : u;
        for (int j = 0; j < nrows; ++j) {
            double acc = 0.0;
            for (int c = 0; c < m; ++c) acc += elem(w, dtype, (int64_t)j * m + c) * elem(a, dtype, x * m + c);
            y[u * nrows + j] = acc;
        }
    }
    return 0;
}
