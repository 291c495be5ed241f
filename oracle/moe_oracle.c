/*
 * moe_oracle.c -- plain fp64 CPU oracle of the DBRX-style MoE layer.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline leg of the benchmark may load this library.  It shares no code,
 * header or constant with the CUDA path.
 *
 * The layer (arxiv 2506.23635, Sec. 2.1 and Table 1 notes (d),(e)): each token
 * is sent to 4 of 16 feed-forward experts; an expert holds three matrices
 * v1, w1, w2 of size D_embed x D_ffn; the selected experts' outputs are
 * combined by a weighted sum (Table 2 caption; Sec. 4.2 "Busy Full Loading"
 * zeroes the unselected experts in that sum).  The paper does not print the
 * router or the GLU formula; the readings used here are:
 *
 *   logits[t,e] = sum_d x[t,d] * Wr[d,e]                       (no bias)
 *   p[t,:]      = softmax(logits[t,:]) over all E experts
 *   idx[t,0..K) = the K largest logits, descending, ties -> lower expert id
 *   g[t,k]      = p[t,idx[t,k]] / sum_j p[t,idx[t,j]]          (sum_k g = 1)
 *   a_f = sum_d x_d W1[e,f,d],  b_f = sum_d x_d V1[e,f,d]
 *   h_f = SiLU(a_f) * b_f,  SiLU(z) = z / (1 + exp(-z))
 *   y_d = sum_f h_f W2[e,d,f]
 *   out[t,d] = sum_k g[t,k] * y^(k)_d
 *
 * Layouts: x [T,D]; Wr [D,E]; W1, V1 [E,F,D]; W2 [E,D,F], row-major.
 * Storage types: 0 = float32, 1 = bfloat16 (uint16 bit pattern).  Every
 * stored value is widened exactly to double; nothing is rounded afterwards.
 *
 * Parity status: every function below is pinned by the CPU tests
 * (brute-force top-k, closed-form expert outputs, invariants).
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_F32 0
#define ORC_BF16 1
#define ORC_F64 2 /* internal: an already widened double array */

static double orc_load(const void *base, int dtype, size_t i)
{
    if (dtype == ORC_F64) return ((const double *)base)[i];
    if (dtype == ORC_BF16) {
        uint32_t u = (uint32_t)((const uint16_t *)base)[i] << 16;
        float f;
        memcpy(&f, &u, sizeof f);
        return (double)f;
    }
    return (double)((const float *)base)[i];
}

static size_t orc_elem_size(int dtype)
{
    return dtype == ORC_BF16 ? 2u : (dtype == ORC_F64 ? 8u : 4u);
}

/* Router logits, reading C1: a plain product with no bias. */
void orc_router_logits(int T, int D, int E, const void *x, int xdt,
                       const void *wr, int wdt, double *logits)
{
    for (int t = 0; t < T; ++t)
        for (int e = 0; e < E; ++e) {
            double s = 0.0;
            for (int d = 0; d < D; ++d)
                s += orc_load(x, xdt, (size_t)t * D + d) *
                     orc_load(wr, wdt, (size_t)d * E + e);
            logits[(size_t)t * E + e] = s;
        }
}

/* Softmax over all E experts, top-K selection, gate renormalisation
 * (Sec. 2.1 "selects 4 out of 16"; readings C1, C2, C5). */
void orc_topk_gates(int T, int E, int K, const double *logits, int32_t *idx,
                    double *gate)
{
    double *p = (double *)malloc(sizeof(double) * (size_t)E);
    char *taken = (char *)malloc((size_t)E);
    for (int t = 0; t < T; ++t) {
        const double *l = logits + (size_t)t * E;
        double m = l[0];
        for (int e = 1; e < E; ++e)
            if (l[e] > m) m = l[e];
        double z = 0.0;
        for (int e = 0; e < E; ++e) {
            p[e] = exp(l[e] - m);
            z += p[e];
        }
        for (int e = 0; e < E; ++e) p[e] /= z;

        memset(taken, 0, (size_t)E);
        double psel = 0.0;
        for (int k = 0; k < K; ++k) {
            int best = -1;
            for (int e = 0; e < E; ++e) {
                if (taken[e]) continue;
                /* strict '>' keeps the lower index on ties */
                if (best < 0 || l[e] > l[best]) best = e;
            }
            taken[best] = 1;
            idx[(size_t)t * K + k] = best;
            psel += p[best];
        }
        for (int k = 0; k < K; ++k)
            gate[(size_t)t * K + k] = p[idx[(size_t)t * K + k]] / psel;
    }
    free(p);
    free(taken);
}

/* Dispatch (reading C6): slots s = t*K + k are ordered by expert, and within
 * an expert by ascending s.  counts[e] = #slots of expert e, offsets is the
 * exclusive prefix sum (E+1 entries), perm[j] = slot at sorted position j,
 * inv_perm[s] = sorted position of slot s. */
void orc_dispatch(int T, int K, int E, const int32_t *idx, int32_t *counts,
                  int32_t *offsets, int32_t *perm, int32_t *inv_perm)
{
    int S = T * K;
    for (int e = 0; e < E; ++e) counts[e] = 0;
    for (int s = 0; s < S; ++s) counts[idx[s]] += 1;
    offsets[0] = 0;
    for (int e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + counts[e];
    int pos = 0;
    for (int e = 0; e < E; ++e)
        for (int s = 0; s < S; ++s)
            if (idx[s] == e) {
                perm[pos] = s;
                inv_perm[s] = pos;
                ++pos;
            }
}

/* One expert applied to one token (Table 1 notes (d),(e); reading C3).
 * w1e, v1e point at the expert's [F,D] matrices, w2e at its [D,F] matrix.
 * h (F) and y (D) receive the GLU hidden vector and the expert output. */
void orc_expert_ffn(int D, int F, const double *xt, const void *w1e,
                    const void *v1e, const void *w2e, int wdt, double *h,
                    double *y)
{
    #pragma omp parallel for schedule(static)
    for (int f = 0; f < F; ++f) {
        double a = 0.0, b = 0.0;
        for (int d = 0; d < D; ++d) {
            a += xt[d] * orc_load(w1e, wdt, (size_t)f * D + d);
            b += xt[d] * orc_load(v1e, wdt, (size_t)f * D + d);
        }
        h[f] = a / (1.0 + exp(-a)) * b;
    }
    #pragma omp parallel for schedule(static)
    for (int d = 0; d < D; ++d) {
        double s = 0.0;
        for (int f = 0; f < F; ++f)
            s += h[f] * orc_load(w2e, wdt, (size_t)d * F + f);
        y[d] = s;
    }
}

static const void *orc_expert_ptr(const void *w, int wdt, size_t per_expert,
                                  int e)
{
    return (const char *)w + (size_t)e * per_expert * orc_elem_size(wdt);
}

/* The sparse layer for the tokens listed in tokens[0..n_tok) (any subset of
 * [0,T)).  out is [n_tok, D]; idx_out [n_tok,K] and gate_out [n_tok,K] are
 * optional (may be NULL).  If residual is non-NULL ([T,D] doubles) it is
 * added to the output row.  Returns 0, or -1 on an out-of-range token. */
int orc_layer_tokens(int T, int D, int F, int E, int K, int n_tok,
                     const int32_t *tokens, const void *x, int xdt,
                     const void *wr, const void *w1, const void *v1,
                     const void *w2, int wdt, const double *residual,
                     double *out, int32_t *idx_out, double *gate_out)
{
    double *xt = (double *)malloc(sizeof(double) * (size_t)D);
    double *lg = (double *)malloc(sizeof(double) * (size_t)E);
    double *h = (double *)malloc(sizeof(double) * (size_t)F);
    double *y = (double *)malloc(sizeof(double) * (size_t)D);
    int32_t *idx = (int32_t *)malloc(sizeof(int32_t) * (size_t)K);
    double *g = (double *)malloc(sizeof(double) * (size_t)K);
    int rc = 0;
    for (int i = 0; i < n_tok; ++i) {
        int t = tokens[i];
        if (t < 0 || t >= T) { rc = -1; break; }
        for (int d = 0; d < D; ++d) xt[d] = orc_load(x, xdt, (size_t)t * D + d);
        orc_router_logits(1, D, E, xt, ORC_F64, wr, wdt, lg);
        orc_topk_gates(1, E, K, lg, idx, g);
        double *o = out + (size_t)i * D;
        for (int d = 0; d < D; ++d)
            o[d] = residual ? residual[(size_t)t * D + d] : 0.0;
        for (int k = 0; k < K; ++k) {
            int e = idx[k];
            orc_expert_ffn(D, F, xt, orc_expert_ptr(w1, wdt, (size_t)F * D, e),
                           orc_expert_ptr(v1, wdt, (size_t)F * D, e),
                           orc_expert_ptr(w2, wdt, (size_t)D * F, e), wdt, h, y);
            for (int d = 0; d < D; ++d) o[d] += g[k] * y[d];
        }
        if (idx_out)
            for (int k = 0; k < K; ++k) idx_out[(size_t)i * K + k] = idx[k];
        if (gate_out)
            for (int k = 0; k < K; ++k) gate_out[(size_t)i * K + k] = g[k];
    }
    free(xt); free(lg); free(h); free(y); free(idx); free(g);
    return rc;
}

/* Busy full loading (Sec. 4.2): every expert computes every token and the
 * unselected experts' outputs are zeroed in the weighted sum.  The result is
 * the same layer; it is kept as an independent route to the output. */
int orc_layer_dense_masked(int T, int D, int F, int E, int K, const void *x,
                           int xdt, const void *wr, const void *w1,
                           const void *v1, const void *w2, int wdt,
                           double *out)
{
    double *xt = (double *)malloc(sizeof(double) * (size_t)D);
    double *lg = (double *)malloc(sizeof(double) * (size_t)E);
    double *mask = (double *)malloc(sizeof(double) * (size_t)E);
    double *h = (double *)malloc(sizeof(double) * (size_t)F);
    double *y = (double *)malloc(sizeof(double) * (size_t)D);
    int32_t *idx = (int32_t *)malloc(sizeof(int32_t) * (size_t)K);
    double *g = (double *)malloc(sizeof(double) * (size_t)K);
    for (int t = 0; t < T; ++t) {
        for (int d = 0; d < D; ++d) xt[d] = orc_load(x, xdt, (size_t)t * D + d);
        orc_router_logits(1, D, E, xt, ORC_F64, wr, wdt, lg);
        orc_topk_gates(1, E, K, lg, idx, g);
        for (int e = 0; e < E; ++e) mask[e] = 0.0;
        for (int k = 0; k < K; ++k) mask[idx[k]] = g[k];
        double *o = out + (size_t)t * D;
        for (int d = 0; d < D; ++d) o[d] = 0.0;
        for (int e = 0; e < E; ++e) {
            orc_expert_ffn(D, F, xt, orc_expert_ptr(w1, wdt, (size_t)F * D, e),
                           orc_expert_ptr(v1, wdt, (size_t)F * D, e),
                           orc_expert_ptr(w2, wdt, (size_t)D * F, e), wdt, h, y);
            for (int d = 0; d < D; ++d) o[d] += mask[e] * y[d];
        }
    }
    free(xt); free(lg); free(mask); free(h); free(y); free(idx); free(g);
    return 0;
}

/* Parameter-free RMS pre-norm between stacked layers (reading C9; the paper
 * does not print the glue between MoE blocks):
 * out[t,:] = x[t,:] / sqrt(mean_d x[t,d]^2 + eps). */
void orc_rmsnorm0(int T, int D, const double *x, double eps, double *out)
{
    for (int t = 0; t < T; ++t) {
        const double *r = x + (size_t)t * D;
        double ss = 0.0;
        for (int d = 0; d < D; ++d) ss += r[d] * r[d];
        const double s = 1.0 / sqrt(ss / D + eps);
        for (int d = 0; d < D; ++d) out[(size_t)t * D + d] = r[d] * s;
    }
}

/* Storage rounding of an activation to bfloat16 (8 significant bits): the
 * representable value nearest to v, ties to the one with an even last
 * significant bit.  Used for the stacked layers' normalised input, which the
 * layer stores in bf16 (the paper's inference keeps activations in bf16,
 * Sec. 5.1).  Finite normal range only. */
void orc_round_bf16(size_t n, const double *in, double *out)
{
    for (size_t i = 0; i < n; ++i) {
        const double v = in[i];
        if (v == 0.0 || !isfinite(v)) { out[i] = v; continue; }
        int e;
        frexp(v, &e);                      /* |v| = m 2^e, m in [0.5, 1) */
        const double ulp = ldexp(1.0, e - 8);
        out[i] = nearbyint(v / ulp) * ulp; /* default mode: ties to even */
    }
}

/* Number of OpenMP threads the parallel loops above use (1 without OpenMP). */
int orc_num_threads(void)
{
    int n = 1;
    #pragma omp parallel
    {
        #pragma omp single
        {
#ifdef _OPENMP
            n = omp_get_num_threads();
#endif
        }
    }
    return n;
}
