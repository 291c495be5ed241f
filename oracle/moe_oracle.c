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

/* One node's share of the decentralised expert-parallel layer (Sec. 4.3,
 * Fig. 7): the node routes the token over all E experts like every other
 * node, runs only the selected experts it holds, e_begin <= e < e_end, and
 * contributes their gated outputs; the all-reduce of the nodes' [T,D]
 * shares forms the weighted sum.  out[i,:] = residual (if given) + sum over
 * k with e_begin <= idx[k] < e_end of g[k] * y^(k).  w1, v1, w2 hold all E
 * experts.  Returns 0, or -1 on an out-of-range token or expert range. */
int orc_layer_experts_tokens(int T, int D, int F, int E, int K, int e_begin,
                             int e_end, int n_tok, const int32_t *tokens,
                             const void *x, int xdt, const void *wr,
                             const void *w1, const void *v1, const void *w2,
                             int wdt, const double *residual, double *out)
{
    if (e_begin < 0 || e_end > E || e_begin >= e_end) return -1;
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
            if (e < e_begin || e >= e_end) continue; /* another node's expert */
            orc_expert_ffn(D, F, xt, orc_expert_ptr(w1, wdt, (size_t)F * D, e),
                           orc_expert_ptr(v1, wdt, (size_t)F * D, e),
                           orc_expert_ptr(w2, wdt, (size_t)D * F, e), wdt, h, y);
            for (int d = 0; d < D; ++d) o[d] += g[k] * y[d];
        }
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

/* ---- self-attention block of a decoder layer ----------------------------
 * Table 1 (note (b)) sizes the self-attention of a DBRX layer only by its
 * parameters, D_qkv_hidden x D_embed + D_embed^2 (D_qkv_hidden = 8,192,
 * D_embed = 6,144), and its FLOPs as twice that; Table 2 books it under
 * "Misc." with the router and the weighted sum.  Everything else is a
 * reading (the paper is silent):
 *
 *   Wqkv [(Hq + 2 Hkv) dh, D]: rows [0, Hq dh) project the queries, the next
 *     Hkv dh rows the keys, the last Hkv dh rows the values; Wo [D, Hq dh];
 *     no biases.  Grouped queries: head h reads key/value head h / (Hq/Hkv).
 *     (48 query heads and 8 key/value heads of 128 give D_qkv_hidden = 8,192.)
 *   Rotary position embedding of queries and keys: in every head, dims i and
 *     i + dh/2 (i < dh/2) turn by the angle pos * base^(-2i/dh).
 *   Causal softmax attention scaled by 1/sqrt(dh): a token at position p of
 *     sequence s attends to cache positions 0..p of s; the keys and values of
 *     all tokens of a call are written to the cache before any token attends.
 *   Block: resid += Wo . ctx, with ctx the attention of RMSNorm0(resid).
 *     With bf16 storage the normalised input, the rotated queries, the
 *     cached keys and values and ctx are rounded to bf16: each is an
 *     activation the paper's bf16 inference stores and the next step reads.
 *
 * Cache layout: [n_seq, Hkv, L, dh] (keys and values alike), as doubles
 * holding exactly the stored values. */

/* u [T, H, dh]: row (t, h) turned by position pos[t]. */
void orc_rope(int T, int H, int dh, double base, const int32_t *pos, double *u)
{
    const int half = dh / 2;
    for (int t = 0; t < T; ++t)
        for (int h = 0; h < H; ++h) {
            double *r = u + ((size_t)t * H + h) * dh;
            for (int i = 0; i < half; ++i) {
                const double ang = (double)pos[t] * pow(base, -2.0 * i / dh);
                const double c = cos(ang), s = sin(ang);
                const double a = r[i], b = r[i + half];
                r[i] = a * c - b * s;
                r[i + half] = b * c + a * s;
            }
        }
}

/* ctx[t, h, :] = sum_j softmax_j(q[t,h,:] . K[s,g,j,:] / sqrt(dh)) V[s,g,j,:]
 * over j = 0..pos[t], s = seq[t], g = h / (Hq/Hkv).  Returns -1 (nothing
 * written) if a sequence or position is out of range. */
int orc_attention(int T, int Hq, int Hkv, int dh, int n_seq, int L, const int32_t *seq,
                  const int32_t *pos, const double *q, const double *kc, const double *vc,
                  double *ctx)
{
    for (int t = 0; t < T; ++t)
        if (seq[t] < 0 || seq[t] >= n_seq || pos[t] < 0 || pos[t] >= L) return -1;
    const int group = Hq / Hkv;
    const double scale = 1.0 / sqrt((double)dh);
    #pragma omp parallel for schedule(dynamic)
    for (int th = 0; th < T * Hq; ++th) {
        const int t = th / Hq, h = th % Hq, g = h / group, n = pos[t] + 1;
        const double *qr = q + (size_t)th * dh;
        const double *kb = kc + ((size_t)seq[t] * Hkv + g) * L * dh;
        const double *vb = vc + ((size_t)seq[t] * Hkv + g) * L * dh;
        double *sc = malloc(sizeof(double) * (size_t)n);
        double m = -INFINITY;
        for (int j = 0; j < n; ++j) {
            double dot = 0.0;
            for (int i = 0; i < dh; ++i) dot += qr[i] * kb[(size_t)j * dh + i];
            sc[j] = dot * scale;
            if (sc[j] > m) m = sc[j];
        }
        double z = 0.0;
        for (int j = 0; j < n; ++j) {
            sc[j] = exp(sc[j] - m);
            z += sc[j];
        }
        double *o = ctx + (size_t)th * dh;
        for (int i = 0; i < dh; ++i) o[i] = 0.0;
        for (int j = 0; j < n; ++j)
            for (int i = 0; i < dh; ++i) o[i] += sc[j] / z * vb[(size_t)j * dh + i];
        free(sc);
    }
    return 0;
}

/* The whole block for T tokens: x [T, D] is the residual stream (in/out),
 * caches as above (updated), round = 1 for bf16 storage.  Returns -1 on a
 * bad sequence or position (nothing written). */
int orc_sa_forward(int T, int D, int Hq, int Hkv, int dh, double base, double eps, int n_seq,
                   int L, const int32_t *seq, const int32_t *pos, double *x, const void *wqkv,
                   const void *wo, int wdt, int round, double *kc, double *vc)
{
    for (int t = 0; t < T; ++t)
        if (seq[t] < 0 || seq[t] >= n_seq || pos[t] < 0 || pos[t] >= L) return -1;
    const int nq = Hq * dh, nkv = Hkv * dh, nr = nq + 2 * nkv;
    double *xn = malloc(sizeof(double) * (size_t)T * D);
    double *qkv = malloc(sizeof(double) * (size_t)T * nr);
    double *q = malloc(sizeof(double) * (size_t)T * nq);
    double *k = malloc(sizeof(double) * (size_t)T * nkv);
    double *v = malloc(sizeof(double) * (size_t)T * nkv);
    double *ctx = malloc(sizeof(double) * (size_t)T * nq);
    orc_rmsnorm0(T, D, x, eps, xn);
    if (round) orc_round_bf16((size_t)T * D, xn, xn);
    #pragma omp parallel for schedule(static)
    for (int r = 0; r < nr; ++r)
        for (int t = 0; t < T; ++t) {
            double acc = 0.0;
            for (int d = 0; d < D; ++d)
                acc += xn[(size_t)t * D + d] * orc_load(wqkv, wdt, (size_t)r * D + d);
            qkv[(size_t)t * nr + r] = acc;
        }
    for (int t = 0; t < T; ++t) {
        memcpy(q + (size_t)t * nq, qkv + (size_t)t * nr, sizeof(double) * nq);
        memcpy(k + (size_t)t * nkv, qkv + (size_t)t * nr + nq, sizeof(double) * nkv);
        memcpy(v + (size_t)t * nkv, qkv + (size_t)t * nr + nq + nkv, sizeof(double) * nkv);
    }
    orc_rope(T, Hq, dh, base, pos, q);
    orc_rope(T, Hkv, dh, base, pos, k);
    if (round) {
        orc_round_bf16((size_t)T * nq, q, q);
        orc_round_bf16((size_t)T * nkv, k, k);
        orc_round_bf16((size_t)T * nkv, v, v);
    }
    for (int t = 0; t < T; ++t)
        for (int g = 0; g < Hkv; ++g) {
            const size_t at = (((size_t)seq[t] * Hkv + g) * L + pos[t]) * dh;
            memcpy(kc + at, k + ((size_t)t * Hkv + g) * dh, sizeof(double) * dh);
            memcpy(vc + at, v + ((size_t)t * Hkv + g) * dh, sizeof(double) * dh);
        }
    orc_attention(T, Hq, Hkv, dh, n_seq, L, seq, pos, q, kc, vc, ctx);
    if (round) orc_round_bf16((size_t)T * nq, ctx, ctx);
    #pragma omp parallel for schedule(static)
    for (int d = 0; d < D; ++d)
        for (int t = 0; t < T; ++t) {
            double acc = 0.0;
            for (int c = 0; c < nq; ++c)
                acc += ctx[(size_t)t * nq + c] * orc_load(wo, wdt, (size_t)d * nq + c);
            x[(size_t)t * D + d] += acc;
        }
    free(xn); free(qkv); free(q); free(k); free(v); free(ctx);
    return 0;
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
