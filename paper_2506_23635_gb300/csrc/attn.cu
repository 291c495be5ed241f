// Self-attention block of a DBRX-style decoder layer and whole decoder
// layers (self-attention, then the MoE block).
//
// Table 1 (note (b)) of arxiv 2506.23635 sizes the self-attention of a layer
// only by its parameters (D_qkv_hidden x D_embed + D_embed^2) and FLOPs (twice
// that); Table 2 books it under "Misc.".  The block built here is the reading
// stated in include/moe.h: grouped-query attention with head_dim 128, rotary
// embedding of queries and keys, causal softmax attention over a bf16 KV
// cache, no biases, resid += W_o . Attn(RMSNorm0(resid)).
//
// Kernels, in launch order:
//   k_sa_prenorm   RMSNorm0 of the fp32 residual -> bf16 rows; block 0 also
//                  writes the trivial dispatch of a one-"expert" projection
//                  (offsets {0, T}, identity permutation, unit gates), so the
//                  two projections run on the MoE layer's own projection
//                  kernels with E = K = 1;
//   projection     W_qkv . x: the row-streaming kernel for one token, the
//                  tcgen05 kernel with the weights as the M operand for up to
//                  64 tokens, the grouped tcgen05 GEMM beyond (fp32 out);
//   k_rope_cache   rotary embedding of q and k (angles formed and reduced in
//                  fp64, evaluated in fp32), k and v written to the cache in
//                  bf16;
//   k_attn_partial one CTA per (token, key/value head, position split): the
//                  group's query heads against its positions, online softmax,
//                  partial (max, sum, weighted values) per split;
//   k_attn_merge   merges the splits, ctx in bf16;
//   projection     W_o . ctx added to the residual (fused into the streaming
//                  kernel for one token; a tcgen05 kernel + k_residual_add
//                  otherwise).
#include <math.h>

#include <algorithm>

#include "ptx.cuh"

namespace moe {
namespace {

constexpr int kHeadDim = 128;
constexpr int kMaxGroup = 8;       // query heads per key/value head
constexpr int kAttnThreads = 128;  // 4 warps
constexpr int kAttnWarps = kAttnThreads / 32;
constexpr int kPosInFlight = 8;    // positions a warp loads before using them
constexpr int kSplitTarget = 304;     // CTAs a decode step's attention aims for at least
constexpr int kSplitPositions = 128;  // cache positions per split it aims for at most
constexpr int kMaxSplit = 64;
constexpr int kMaxSplitCtas = 4096;   // bound on T * Hkv * splits (sizes the workspace)
constexpr int kMaxSaTokens = 65536;

// Most position splits a call of T tokens may use (the workspace holds this many).
int split_cap(int T, int Hkv) {
    const int tg = std::max(1, T * Hkv);
    return std::max(1, std::min(kMaxSplit, kMaxSplitCtas / tg));
}

// Splits per (token, key/value head): enough CTAs to cover the SMs and at
// most kSplitPositions cache positions per split, within split_cap.
int n_split_for(int T, int Hkv, int max_len) {
    const int tg = std::max(1, T * Hkv);
    const int by_ctas = (kSplitTarget + tg - 1) / tg;
    const int by_len = (max_len + kSplitPositions - 1) / kSplitPositions;
    return std::max(1, std::min(split_cap(T, Hkv), std::max(by_ctas, by_len)));
}

// Rotary angular rates base^(-2i/dh), i < dh/2, computed on the host in
// double precision and passed by value.
struct RopeRates {
    double w[kHeadDim / 2];
};

// ---- kernels --------------------------------------------------------------------

// The trivial dispatch of the one-"expert" projections (offsets {0, T},
// identity permutation, unit gates).
__device__ __forceinline__ void write_trivial_dispatch(int T, int32_t *offsets, int32_t *ident,
                                                       float *ones) {
    for (int i = threadIdx.x; i < T; i += blockDim.x) {
        ident[i] = i;
        ones[i] = 1.f;
    }
    if (threadIdx.x == 0) {
        offsets[0] = 0;
        offsets[1] = T;
    }
}

// One 1024-thread block per token: every thread's loads of the row are in
// flight together.
constexpr int kNormThreads = 1024;

__global__ void __launch_bounds__(kNormThreads)
k_sa_prenorm(int T, int D, const float *__restrict__ resid, bf16 *__restrict__ xn, float eps,
             int32_t *offsets, int32_t *ident, float *ones) {
    ptx::grid_dependency_wait();
    __shared__ float red[kNormThreads / 32];
    const int t = blockIdx.x;
    if (t == 0) write_trivial_dispatch(T, offsets, ident, ones);
    const float4 *r = reinterpret_cast<const float4 *>(resid + (size_t)t * D);
    const int nv = D >> 2;
    float ss = 0.f;
#pragma unroll 4
    for (int i = threadIdx.x; i < nv; i += blockDim.x) {
        const float4 v = r[i];
        ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < kNormThreads / 32; ++w) tot += red[w];
    const float s = 1.0f / sqrtf(tot / (float)D + eps);
    __nv_bfloat162 *o = reinterpret_cast<__nv_bfloat162 *>(xn + (size_t)t * D);
#pragma unroll 4
    for (int i = threadIdx.x; i < nv; i += blockDim.x) {
        const float4 v = r[i];
        o[2 * i] = __floats2bfloat162_rn(v.x * s, v.y * s);
        o[2 * i + 1] = __floats2bfloat162_rn(v.z * s, v.w * s);
    }
}

__global__ void __launch_bounds__(256)
k_sa_setup(int T, int32_t *offsets, int32_t *ident, float *ones) {
    ptx::grid_dependency_wait();
    write_trivial_dispatch(T, offsets, ident, ones);
}

// qkv [T, (Hq + 2 Hkv) 128] fp32 -> q [T, Hq, 128] fp32 (rotated); rotated
// keys and the values to the caches [n_seq, Hkv, L, 128] in bf16.  One
// 64-thread block per (head row of qkv, token): thread i turns the pair
// (i, i + 64) of a query or key head, or copies two value elements.
__global__ void __launch_bounds__(kHeadDim / 2)
k_rope_cache(int Hq, int Hkv, int n_seq, int L, RopeRates rates, const int32_t *__restrict__ seq,
             const int32_t *__restrict__ pos, const float *__restrict__ qkv, float *__restrict__ q,
             bf16 *__restrict__ kc, bf16 *__restrict__ vc, unsigned *err) {
    ptx::grid_dependency_wait();
    constexpr int H2 = kHeadDim / 2;
    const int hr = blockIdx.x, t = blockIdx.y, i = threadIdx.x;
    const int sq = seq[t], p = pos[t];
    const bool ok = sq >= 0 && sq < n_seq && p >= 0 && p < L;
    if (!ok && hr == 0 && i == 0) set_error(err, kErrIndex);
    const int nq = Hq * kHeadDim, nkv = Hkv * kHeadDim;
    const float *row = qkv + (size_t)t * (nq + 2 * nkv) + (size_t)hr * kHeadDim;
    const float a = row[i], b = row[i + H2];
    if (hr >= Hq + Hkv) {  // a value head: stored as it is
        if (!ok) return;
        bf16 *vd = vc + (((size_t)sq * Hkv + (hr - Hq - Hkv)) * L + p) * kHeadDim;
        vd[i] = __float2bfloat16_rn(a);
        vd[i + H2] = __float2bfloat16_rn(b);
        return;
    }
    // the angle of pair i is pos * rate_i, formed and reduced to [-pi, pi]
    // in fp64 (exact to far below fp32 resolution at any cache position),
    // then evaluated in fp32
    constexpr double kTwoPi = 6.283185307179586;
    const double ang = (double)(ok ? p : 0) * rates.w[i];
    const double red = fma(-rint(ang * (1.0 / kTwoPi)), kTwoPi, ang);
    float sn, cs;
    sincosf((float)red, &sn, &cs);
    const float x0 = a * cs - b * sn, x1 = b * cs + a * sn;
    if (hr < Hq) {
        float *qo = q + (size_t)t * nq + (size_t)hr * kHeadDim;
        qo[i] = x0;
        qo[i + H2] = x1;
    } else if (ok) {
        bf16 *kd = kc + (((size_t)sq * Hkv + (hr - Hq)) * L + p) * kHeadDim;
        kd[i] = __float2bfloat16_rn(x0);
        kd[i + H2] = __float2bfloat16_rn(x1);
    }
}

__device__ __forceinline__ void unpack4(uint2 u, float (&o)[4]) {
    unpack_bf16x2(u.x, o[0], o[1]);
    unpack_bf16x2(u.y, o[2], o[3]);
}

// One CTA per (split s, token t, key/value head g).  Lane l owns dims
// [4l, 4l+4) of the G query heads of the group; warp w takes positions
// j0 + w*P + i*(4P) + u (P = kPosInFlight) of the split's range [j0, j1).
// Partial results per (t, query head, s): max score, sum of exp, and the
// exp-weighted sum of values, all relative to that max.
template <int G>
__global__ void __launch_bounds__(kAttnThreads)
k_attn_partial(int Hq, int Hkv, int n_seq, int L, int n_split, const int32_t *__restrict__ seq,
               const int32_t *__restrict__ pos, const float *__restrict__ q,
               const bf16 *__restrict__ kc, const bf16 *__restrict__ vc,
               float *__restrict__ part_ml, float *__restrict__ part_acc) {
    ptx::grid_dependency_wait();
    __shared__ float sm_m[kAttnWarps][G], sm_l[kAttnWarps][G];
    __shared__ float sm_acc[kAttnWarps][G][kHeadDim];
    const int s = blockIdx.x, tg = blockIdx.y;
    const int t = tg / Hkv, g = tg - t * Hkv;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int sq = seq[t], p = pos[t];
    const bool ok = sq >= 0 && sq < n_seq && p >= 0 && p < L;
    const int n = ok ? p + 1 : 0;
    const int chunk = (n + n_split - 1) / n_split;
    const int j0 = min(n, s * chunk), j1 = min(n, j0 + chunk);
    const float scale = 1.0f / sqrtf((float)kHeadDim);

    float qv[G][4], m[G], l[G], acc[G][4];
#pragma unroll
    for (int h = 0; h < G; ++h) {
        const float4 v = *reinterpret_cast<const float4 *>(
            q + ((size_t)t * Hq + g * G + h) * kHeadDim + lane * 4);
        qv[h][0] = v.x * scale;
        qv[h][1] = v.y * scale;
        qv[h][2] = v.z * scale;
        qv[h][3] = v.w * scale;
        m[h] = -INFINITY;
        l[h] = 0.f;
#pragma unroll
        for (int i = 0; i < 4; ++i) acc[h][i] = 0.f;
    }
    const size_t base = ok ? ((size_t)sq * Hkv + g) * L * kHeadDim : 0;
    const bf16 *kb = kc + base + lane * 4;
    const bf16 *vb = vc + base + lane * 4;
    constexpr int P = kPosInFlight;
    for (int j = j0 + warp * P; j < j1; j += kAttnWarps * P) {
        uint2 kr[P], vr[P];
#pragma unroll
        for (int u = 0; u < P; ++u) {
            if (j + u < j1) {
                kr[u] = __ldg(reinterpret_cast<const uint2 *>(kb + (size_t)(j + u) * kHeadDim));
                vr[u] = __ldg(reinterpret_cast<const uint2 *>(vb + (size_t)(j + u) * kHeadDim));
            }
        }
#pragma unroll
        for (int u = 0; u < P; ++u) {
            if (j + u >= j1) break;
            float k4[4], v4[4];
            unpack4(kr[u], k4);
            unpack4(vr[u], v4);
            float sc[G];
#pragma unroll
            for (int h = 0; h < G; ++h)
                sc[h] = qv[h][0] * k4[0] + qv[h][1] * k4[1] + qv[h][2] * k4[2] + qv[h][3] * k4[3];
#pragma unroll
            for (int h = 0; h < G; ++h) sc[h] = warp_sum(sc[h]);
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float mn = fmaxf(m[h], sc[h]);
                const float corr = expf(m[h] - mn);  // 0 while m is -inf
                const float w = expf(sc[h] - mn);
                l[h] = l[h] * corr + w;
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[h][i] = fmaf(w, v4[i], acc[h][i] * corr);
                m[h] = mn;
            }
        }
    }
#pragma unroll
    for (int h = 0; h < G; ++h) {
        if (lane == 0) {
            sm_m[warp][h] = m[h];
            sm_l[warp][h] = l[h];
        }
#pragma unroll
        for (int i = 0; i < 4; ++i) sm_acc[warp][h][lane * 4 + i] = acc[h][i];
    }
    __syncthreads();
    const int d = threadIdx.x;
#pragma unroll 1
    for (int h = 0; h < G; ++h) {
        float M = -INFINITY;
#pragma unroll
        for (int w = 0; w < kAttnWarps; ++w) M = fmaxf(M, sm_m[w][h]);
        float Ls = 0.f, A = 0.f;
        if (M != -INFINITY) {
#pragma unroll
            for (int w = 0; w < kAttnWarps; ++w) {
                const float c = expf(sm_m[w][h] - M);
                Ls = fmaf(sm_l[w][h], c, Ls);
                A = fmaf(sm_acc[w][h][d], c, A);
            }
        }
        const size_t o = ((size_t)t * Hq + g * G + h) * n_split + s;
        if (d == 0) {
            part_ml[2 * o] = M;
            part_ml[2 * o + 1] = Ls;
        }
        part_acc[o * kHeadDim + d] = A;
    }
}

// ctx[t, h*128 + d] = merged weighted values / merged sum, over the splits:
// ctx = sum_s e^(M_s - M) A_s[d] / sum_s e^(M_s - M) L_s.  The splits'
// (max, sum) pairs are read once into shared memory; kMergeGroups groups of
// 128 threads each sum every kMergeGroups-th split of their dimension with
// independent loads, and the groups' sums are added in group order.
constexpr int kMergeGroups = 4;

__global__ void __launch_bounds__(kHeadDim * kMergeGroups)
k_attn_merge(int n_split, const float *__restrict__ part_ml, const float *__restrict__ part_acc,
             bf16 *__restrict__ ctx) {
    static_assert(kMaxSplit <= kHeadDim * kMergeGroups, "one thread per split");
    ptx::grid_dependency_wait();
    __shared__ float sm[kMaxSplit], sl[kMaxSplit], sc[kMaxSplit];
    __shared__ float sa[kMergeGroups][kHeadDim], sls[kMergeGroups][kHeadDim];
    const int th = blockIdx.x, tid = threadIdx.x;
    const int d = tid % kHeadDim, grp = tid / kHeadDim;
    const float *ml = part_ml + (size_t)th * n_split * 2;
    if (tid < n_split) {
        sm[tid] = ml[2 * tid];
        sl[tid] = ml[2 * tid + 1];
    }
    __syncthreads();
    float M = -INFINITY;
    for (int k = 0; k < n_split; ++k) M = fmaxf(M, sm[k]);
    if (tid < n_split) sc[tid] = M != -INFINITY ? expf(sm[tid] - M) : 0.f;
    __syncthreads();
    float Ls = 0.f, A = 0.f;
    const float *pa = part_acc + (size_t)th * n_split * kHeadDim + d;
#pragma unroll 4
    for (int k = grp; k < n_split; k += kMergeGroups) {
        Ls = fmaf(sl[k], sc[k], Ls);
        A = fmaf(pa[(size_t)k * kHeadDim], sc[k], A);
    }
    sa[grp][d] = A;
    sls[grp][d] = Ls;
    __syncthreads();
    if (grp != 0) return;
    for (int g = 1; g < kMergeGroups; ++g) {
        A += sa[g][d];
        Ls += sls[g][d];
    }
    ctx[(size_t)th * kHeadDim + d] = __float2bfloat16_rn(Ls > 0.f ? A / Ls : 0.f);
}

__global__ void __launch_bounds__(256)
k_residual_add(long long n4, float *__restrict__ resid, const float *__restrict__ y) {
    ptx::grid_dependency_wait();
    float4 *r = reinterpret_cast<float4 *>(resid);
    const float4 *a = reinterpret_cast<const float4 *>(y);
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (long long)gridDim.x * blockDim.x) {
        float4 v = r[i];
        const float4 w = a[i];
        v.x += w.x;
        v.y += w.y;
        v.z += w.z;
        v.w += w.w;
        r[i] = v;
    }
}

// ---- host ------------------------------------------------------------------------

struct SaWs {
    size_t offsets, ident, ones, xn, qkv, q, part_ml, part_acc, ctx, total;
};

SaWs sa_ws(const moe_sa_dims &d, int64_t T) {
    auto up = [](size_t v) { return (v + 255) & ~size_t(255); };
    const size_t nq = (size_t)d.n_heads * kHeadDim;
    const size_t nr = nq + 2 * (size_t)d.n_kv_heads * kHeadDim;
    const size_t parts = (size_t)T * d.n_heads * split_cap((int)T, d.n_kv_heads);
    SaWs L{};
    size_t o = 0;
    L.offsets = o; o += up(2 * 4);
    L.ident = o; o += up((size_t)T * 4);
    L.ones = o; o += up((size_t)T * 4);
    L.xn = o; o += up((size_t)T * d.d_model * 2);
    // projection outputs: qkv first, later the output projection's rows
    L.qkv = o; o += up((size_t)T * std::max(nr, (size_t)d.d_model) * 4);
    L.q = o; o += up((size_t)T * nq * 4);
    L.part_ml = o; o += up(parts * 2 * 4);
    L.part_acc = o; o += up(parts * kHeadDim * 4);
    L.ctx = o; o += up((size_t)T * nq * 2);
    L.total = o;
    return L;
}

template <typename P>
P *at(void *ws, size_t off) {
    return reinterpret_cast<P *>(static_cast<char *>(ws) + off);
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool ok_ptr(const void *p) { return p != nullptr && aligned16(p); }
moe_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MOE_OK : MOE_ERR_CUDA; }

moe_status check_sa(const moe_sa_dims *d) {
    if (!d) return MOE_ERR_INVALID_ARG;
    if (d->d_model < 8 || d->d_model > 49152 || d->d_model % 8) return MOE_ERR_INVALID_ARG;
    if (d->head_dim != kHeadDim) return MOE_ERR_UNSUPPORTED;
    if (d->n_kv_heads < 1 || d->n_heads < d->n_kv_heads || d->n_heads % d->n_kv_heads)
        return MOE_ERR_INVALID_ARG;
    if (d->n_heads / d->n_kv_heads > kMaxGroup) return MOE_ERR_UNSUPPORTED;
    if ((int64_t)(d->n_heads + 2 * d->n_kv_heads) * kHeadDim > 49152) return MOE_ERR_INVALID_ARG;
    if (!(d->rope_base > 1.f) || !isfinite(d->rope_base)) return MOE_ERR_INVALID_ARG;
    return MOE_OK;
}

moe_status check_sa_call(const moe_sa_dims *d, int32_t T, const int32_t *seq, const int32_t *pos,
                         int32_t n_seq, int32_t max_len) {
    moe_status s = check_sa(d);
    if (s != MOE_OK) return s;
    if (T < 0 || T > kMaxSaTokens || n_seq < 1 || max_len < 1) return MOE_ERR_INVALID_ARG;
    if (T > 0 && (!ok_ptr(seq) || !ok_ptr(pos))) return MOE_ERR_INVALID_ARG;
    return MOE_OK;
}

// The one-"expert" projection dims: Nw output rows, Kdim inputs.
moe_dims proj_dims(int Nw, int Kdim) {
    moe_dims p{};
    p.d_model = Nw;
    p.ffn_hidden = Kdim;
    p.n_experts = 1;
    p.top_k = 1;
    p.w_dtype = MOE_BF16;
    p.x_dtype = MOE_BF16;
    p.out_dtype = MOE_F32;
    return p;
}

struct SaCall {
    const moe_sa_dims &d;
    int T;
    cudaStream_t st;
    void *ws;
    SaWs L;
    int nq() const { return d.n_heads * kHeadDim; }
    int nr() const { return (d.n_heads + 2 * d.n_kv_heads) * kHeadDim; }
    bool streamed() const {
        return T == 1 && stream_path_ok(proj_dims(nr(), d.d_model), 1) &&
               stream_path_ok(proj_dims(d.d_model, nq()), 1);
    }
};

// W_qkv . xn -> qkv (fp32), then the rotary embedding and the cache writes.
cudaError_t qkv_rope(const SaCall &c, const void *xn, const void *w_qkv, const int32_t *seq,
                     const int32_t *pos, int n_seq, int L, float *q, void *kc, void *vc) {
    const moe_dims pd = proj_dims(c.nr(), c.d.d_model);
    const int32_t *offsets = at<int32_t>(c.ws, c.L.offsets);
    float *qkv = at<float>(c.ws, c.L.qkv);
    cudaError_t e;
    if (c.streamed())
        e = launch_down_stream(pd, 1, xn, offsets, at<int32_t>(c.ws, c.L.ident), w_qkv,
                               at<float>(c.ws, c.L.ones), nullptr, nullptr, qkv, false, c.st,
                               "qkv_stream");
    else if (c.T <= kRowsMaxTokens)
        e = launch_gemm_rows_tc(c.T, c.d.d_model, c.nr(), xn, w_qkv, qkv, c.st, "qkv_rows_tc");
    else
        e = launch_gemm_down_tc(pd, c.T, xn, offsets, w_qkv, qkv, c.st, "qkv_gemm_tc");
    if (e != cudaSuccess) return e;
    int Hq = c.d.n_heads, Hkv = c.d.n_kv_heads, ns = n_seq, Lv = L;
    RopeRates rates;
    for (int i = 0; i < kHeadDim / 2; ++i)
        rates.w[i] = pow((double)c.d.rope_base, -2.0 * i / (double)kHeadDim);
    const float *qkvc = qkv;
    bf16 *kcp = static_cast<bf16 *>(kc), *vcp = static_cast<bf16 *>(vc);
    unsigned *err = device_info().err;
    void *args[] = {&Hq, &Hkv, &ns, &Lv, &rates, &seq, &pos, &qkvc, &q, &kcp, &vcp, &err};
    LaunchScope ls("rope_cache", c.st);
    return launch_pdl((const void *)k_rope_cache, dim3(Hq + 2 * Hkv, c.T), dim3(kHeadDim / 2), 0,
                      c.st, args);
}

// Attention over the caches: per-split partials, then their merge.
cudaError_t attend(const SaCall &c, const float *q, const int32_t *seq, const int32_t *pos,
                   int n_seq, int L, const void *kc, const void *vc, void *ctx) {
    const int Hq = c.d.n_heads, Hkv = c.d.n_kv_heads, G = Hq / Hkv;
    int ns = n_split_for(c.T, Hkv, L);
    float *ml = at<float>(c.ws, c.L.part_ml), *acc = at<float>(c.ws, c.L.part_acc);
    const void *kern = nullptr;
    switch (G) {
        case 1: kern = (const void *)k_attn_partial<1>; break;
        case 2: kern = (const void *)k_attn_partial<2>; break;
        case 3: kern = (const void *)k_attn_partial<3>; break;
        case 4: kern = (const void *)k_attn_partial<4>; break;
        case 5: kern = (const void *)k_attn_partial<5>; break;
        case 6: kern = (const void *)k_attn_partial<6>; break;
        case 7: kern = (const void *)k_attn_partial<7>; break;
        default: kern = (const void *)k_attn_partial<8>; break;
    }
    int Hqv = Hq, Hkvv = Hkv, nsq = n_seq, Lv = L;
    const bf16 *kcp = static_cast<const bf16 *>(kc), *vcp = static_cast<const bf16 *>(vc);
    {
        void *args[] = {&Hqv, &Hkvv, &nsq, &Lv, &ns, &seq, &pos, &q, &kcp, &vcp, &ml, &acc};
        LaunchScope ls("attention", c.st);
        cudaError_t e = launch_pdl(kern, dim3(ns, c.T * Hkv), dim3(kAttnThreads), 0, c.st, args);
        if (e != cudaSuccess) return e;
    }
    const float *mlc = ml, *accc = acc;
    bf16 *cp = static_cast<bf16 *>(ctx);
    void *args[] = {&ns, &mlc, &accc, &cp};
    LaunchScope ls("attn_merge", c.st);
    return launch_pdl((const void *)k_attn_merge, dim3(c.T * Hq), dim3(kHeadDim * kMergeGroups), 0,
                      c.st, args);
}

// resid += W_o . ctx
cudaError_t out_proj(const SaCall &c, const void *ctx, const void *w_o, float *resid) {
    const moe_dims pd = proj_dims(c.d.d_model, c.nq());
    const int32_t *offsets = at<int32_t>(c.ws, c.L.offsets);
    const int32_t *ident = at<int32_t>(c.ws, c.L.ident);
    const float *ones = at<float>(c.ws, c.L.ones);
    if (c.streamed())  // the residual element is read before the same thread writes it
        return launch_down_stream(pd, 1, ctx, offsets, ident, w_o, ones, resid, resid, nullptr,
                                  true, c.st, "o_stream");
    float *y = at<float>(c.ws, c.L.qkv);
    cudaError_t e = c.T <= kRowsMaxTokens
                        ? launch_gemm_rows_tc(c.T, c.nq(), c.d.d_model, ctx, w_o, y, c.st,
                                              "o_rows_tc")
                        : launch_gemm_down_tc(pd, c.T, ctx, offsets, w_o, y, c.st, "o_gemm_tc");
    if (e != cudaSuccess) return e;
    long long n4 = (long long)c.T * c.d.d_model / 4;
    const long long cap = (long long)device_info().sm_count * 8;
    const int grid = (int)std::max(1LL, std::min((n4 + 255) / 256, cap));
    const float *yc = y;
    void *args[] = {&n4, &resid, &yc};
    LaunchScope ls("residual_add", c.st);
    return launch_pdl((const void *)k_residual_add, dim3(grid), dim3(256), 0, c.st, args);
}

moe_status check_ws(const moe_sa_dims *d, int T, void *ws, size_t ws_bytes) {
    size_t need = sa_ws(*d, T).total;
    if (!ws || !aligned16(ws) || ws_bytes < need) return MOE_ERR_WORKSPACE;
    return MOE_OK;
}

moe_status setup_dispatch(const SaCall &c) {
    int Tv = c.T;
    int32_t *off = at<int32_t>(c.ws, c.L.offsets), *id = at<int32_t>(c.ws, c.L.ident);
    float *ones = at<float>(c.ws, c.L.ones);
    void *args[] = {&Tv, &off, &id, &ones};
    LaunchScope ls("sa_setup", c.st);
    return cuda_status(launch_pdl((const void *)k_sa_setup, dim3(1), dim3(256), 0, c.st, args));
}

}  // namespace
}  // namespace moe

using namespace moe;

extern "C" {

moe_status moe_sa_workspace_size(const moe_sa_dims *dims, int32_t max_tokens, size_t *bytes) {
    moe_status s = check_sa(dims);
    if (s != MOE_OK) return s;
    if (!bytes || max_tokens < 0 || max_tokens > kMaxSaTokens) return MOE_ERR_INVALID_ARG;
    *bytes = sa_ws(*dims, max_tokens).total;
    return MOE_OK;
}

moe_status moe_sa_qkv(const moe_sa_dims *dims, int32_t T, const void *x_norm, const void *w_qkv,
                      const int32_t *seq, const int32_t *pos, int32_t n_seq, int32_t max_len,
                      float *q, void *k_cache, void *v_cache, void *ws, size_t ws_bytes,
                      moe_stream_t stream) {
    MOE_INJECT("moe_sa_qkv");
    moe_status s = check_sa_call(dims, T, seq, pos, n_seq, max_len);
    if (s != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(x_norm) || !ok_ptr(w_qkv) || !ok_ptr(q) || !ok_ptr(k_cache) || !ok_ptr(v_cache))
        return MOE_ERR_INVALID_ARG;
    if ((s = check_ws(dims, T, ws, ws_bytes)) != MOE_OK) return s;
    SaCall c{*dims, T, (cudaStream_t)stream, ws, sa_ws(*dims, T)};
    if (!c.streamed() && !tc_path_ok(proj_dims(c.nr(), dims->d_model))) return MOE_ERR_UNSUPPORTED;
    if ((s = setup_dispatch(c)) != MOE_OK) return s;
    return cuda_status(qkv_rope(c, x_norm, w_qkv, seq, pos, n_seq, max_len, q, k_cache, v_cache));
}

moe_status moe_sa_attend(const moe_sa_dims *dims, int32_t T, const float *q, const int32_t *seq,
                         const int32_t *pos, int32_t n_seq, int32_t max_len, const void *k_cache,
                         const void *v_cache, void *ctx, void *ws, size_t ws_bytes,
                         moe_stream_t stream) {
    MOE_INJECT("moe_sa_attend");
    moe_status s = check_sa_call(dims, T, seq, pos, n_seq, max_len);
    if (s != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(q) || !ok_ptr(k_cache) || !ok_ptr(v_cache) || !ok_ptr(ctx))
        return MOE_ERR_INVALID_ARG;
    if ((s = check_ws(dims, T, ws, ws_bytes)) != MOE_OK) return s;
    SaCall c{*dims, T, (cudaStream_t)stream, ws, sa_ws(*dims, T)};
    return cuda_status(attend(c, q, seq, pos, n_seq, max_len, k_cache, v_cache, ctx));
}

moe_status moe_sa_forward(const moe_sa_dims *dims, int32_t T, const int32_t *seq,
                          const int32_t *pos, int32_t n_seq, int32_t max_len, float *resid,
                          const void *w_qkv, const void *w_o, void *k_cache, void *v_cache,
                          float eps, void *ws, size_t ws_bytes, moe_stream_t stream) {
    MOE_INJECT("moe_sa_forward");
    moe_status s = check_sa_call(dims, T, seq, pos, n_seq, max_len);
    if (s != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(resid) || !ok_ptr(w_qkv) || !ok_ptr(w_o) || !ok_ptr(k_cache) ||
        !ok_ptr(v_cache) || !(eps > 0.f))
        return MOE_ERR_INVALID_ARG;
    if ((s = check_ws(dims, T, ws, ws_bytes)) != MOE_OK) return s;
    SaCall c{*dims, T, (cudaStream_t)stream, ws, sa_ws(*dims, T)};
    if (!c.streamed() && (!tc_path_ok(proj_dims(c.nr(), dims->d_model)) ||
                          !tc_path_ok(proj_dims(dims->d_model, c.nq()))))
        return MOE_ERR_UNSUPPORTED;
    bf16 *xn = at<bf16>(ws, c.L.xn);
    float *q = at<float>(ws, c.L.q);
    bf16 *ctx = at<bf16>(ws, c.L.ctx);
    {
        int Tv = T, D = dims->d_model;
        const float *rc = resid;
        int32_t *off = at<int32_t>(ws, c.L.offsets), *id = at<int32_t>(ws, c.L.ident);
        float *ones = at<float>(ws, c.L.ones);
        void *args[] = {&Tv, &D, &rc, &xn, &eps, &off, &id, &ones};
        LaunchScope ls("sa_prenorm", c.st);
        if (launch_pdl((const void *)k_sa_prenorm, dim3(T), dim3(kNormThreads), 0, c.st, args) !=
            cudaSuccess)
            return MOE_ERR_CUDA;
    }
    cudaError_t e = qkv_rope(c, xn, w_qkv, seq, pos, n_seq, max_len, q, k_cache, v_cache);
    if (e == cudaSuccess) e = attend(c, q, seq, pos, n_seq, max_len, k_cache, v_cache, ctx);
    if (e == cudaSuccess) e = out_proj(c, ctx, w_o, resid);
    return cuda_status(e);
}

moe_status moe_decoder_workspace_size(const moe_sa_dims *attn, const moe_dims *moe_d,
                                      int32_t max_tokens, size_t *bytes) {
    if (!bytes) return MOE_ERR_INVALID_ARG;
    size_t a = 0, b = 0;
    moe_status s = moe_sa_workspace_size(attn, max_tokens, &a);
    if (s != MOE_OK) return s;
    if ((s = moe_stack_workspace_size(moe_d, max_tokens, &b)) != MOE_OK) return s;
    *bytes = std::max(a, b);
    return MOE_OK;
}

moe_status moe_decoder_forward(const moe_sa_dims *attn, const moe_dims *moe_d, int32_t n_layers,
                               int32_t T, const int32_t *seq, const int32_t *pos, int32_t n_seq,
                               int32_t max_len, float *resid, const void *const *w_qkv,
                               const void *const *w_o, const void *const *w_router,
                               const void *const *w1, const void *const *v1,
                               const void *const *w2, void *const *k_cache,
                               void *const *v_cache, float eps, void *ws, size_t ws_bytes,
                               moe_stream_t stream) {
    MOE_INJECT("moe_decoder_forward");
    moe_status s = check_sa_call(attn, T, seq, pos, n_seq, max_len);
    if (s != MOE_OK) return s;
    if (!moe_d || moe_d->d_model != attn->d_model || moe_d->w_dtype != MOE_BF16 ||
        moe_d->x_dtype != MOE_BF16 || moe_d->out_dtype != MOE_F32 || n_layers < 0)
        return MOE_ERR_INVALID_ARG;
    if (T == 0 || n_layers == 0) return MOE_OK;
    if (!w_qkv || !w_o || !w_router || !w1 || !v1 || !w2 || !k_cache || !v_cache)
        return MOE_ERR_INVALID_ARG;
    size_t need = 0;
    if ((s = moe_decoder_workspace_size(attn, moe_d, T, &need)) != MOE_OK) return s;
    if (!ws || !aligned16(ws) || ws_bytes < need) return MOE_ERR_WORKSPACE;
    for (int l = 0; l < n_layers; ++l) {
        s = moe_sa_forward(attn, T, seq, pos, n_seq, max_len, resid, w_qkv[l], w_o[l],
                           k_cache[l], v_cache[l], eps, ws, ws_bytes, stream);
        if (s != MOE_OK) return s;
        s = moe_stack_forward(moe_d, 1, T, &w_router[l], &w1[l], &v1[l], &w2[l], resid, eps, ws,
                              ws_bytes, stream);
        if (s != MOE_OK) return s;
    }
    return MOE_OK;
}

}  // extern "C"
