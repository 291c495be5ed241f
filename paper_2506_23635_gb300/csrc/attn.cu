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
//                  (offsets {0, T}), for the grouped GEMM of prefill batches;
//                  it lets the projection launch at once (the projection's
//                  weight loads do not depend on it);
//   projection     W_qkv . x: the tcgen05 kernel with the weights as the M
//                  operand (split reduction) for up to 64 tokens, the grouped
//                  tcgen05 GEMM with E = 1 beyond (fp32 out);
//   k_rope_cache   rotary embedding of q and k (angles formed and reduced in
//                  fp64, evaluated in fp32), k and v written to the cache in
//                  bf16;
//   k_attn_partial one CTA per (token, key/value head, position split): the
//                  group's query heads against its positions, online softmax,
//                  partial (max, sum, weighted values) per split;
//   k_attn_merge   merges the splits, ctx in bf16 (a single split writes ctx
//                  itself); in moe_sa_forward, calls of 128 tokens or more
//                  first run the tensor-core prefill attention (attn_tc.cu)
//                  on every full 128-token tile of consecutive positions of
//                  one sequence, and the kernels above only on the rest;
//   projection     W_o . ctx (the same two kernels), its partial sums added to
//                  the residual by k_residual_add.
#include <math.h>
#include <stdlib.h>

#include <algorithm>

#include "ptx.cuh"

namespace moe {
namespace {

constexpr int kHeadDim = 128;
constexpr int kMaxGroup = 8;       // query heads per key/value head
constexpr int kAttnThreads = 128;  // 4 warps
constexpr int kAttnWarps = kAttnThreads / 32;
constexpr int kSplitTarget = 152;     // CTAs a decode step's attention aims for at least
constexpr int kSplitPositions = 128;  // cache positions per split (a 32-position tile per warp)
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

// The trivial dispatch of a one-"expert" projection: offsets {0, T}.
__device__ __forceinline__ void write_trivial_dispatch(int T, int32_t *offsets) {
    if (threadIdx.x == 0) {
        offsets[0] = 0;
        offsets[1] = T;
    }
}

// One block per token: 1024 threads for decode batches (every thread's
// loads of the row in flight together), 256 threads with 16 float4 of the
// row each for larger batches (the 1024-thread form ran at 1.9 TB/s over
// 2048 tokens: too little work per thread between block barriers).  The row
// stays in registers between the sum of squares and the scaling.
constexpr int kNormThreads = 1024;
constexpr int kNormThreadsWide = 256;
constexpr int kNormWideMinTokens = 64;
constexpr int kNormMaxVec = 16;  // float4 per thread: D <= 4 * 16 * 256

template <int NT, int VEC>
__global__ void __launch_bounds__(NT)
k_sa_prenorm(int T, int D, const float *__restrict__ resid, bf16 *__restrict__ xn, float eps,
             int32_t *offsets) {
    // the projection after this kernel may start now: its weight loads do
    // not depend on anything here
    ptx::launch_dependents();
    ptx::grid_dependency_wait();
    __shared__ float red[NT / 32];
    const int t = blockIdx.x;
    if (t == 0) write_trivial_dispatch(T, offsets);
    const float4 *r = reinterpret_cast<const float4 *>(resid + (size_t)t * D);
    const int nv = D >> 2;
    float4 keep[VEC];
    float ss = 0.f;
#pragma unroll
    for (int u = 0; u < VEC; ++u) {
        const int i = threadIdx.x + u * NT;
        keep[u] = i < nv ? r[i] : make_float4(0.f, 0.f, 0.f, 0.f);
        ss += keep[u].x * keep[u].x + keep[u].y * keep[u].y + keep[u].z * keep[u].z +
              keep[u].w * keep[u].w;
    }
    for (int i = threadIdx.x + VEC * NT; i < nv; i += NT) {  // rows wider than the registers
        const float4 v = r[i];
        ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
    }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < NT / 32; ++w) tot += red[w];
    const float s = 1.0f / sqrtf(tot / (float)D + eps);
    __nv_bfloat162 *o = reinterpret_cast<__nv_bfloat162 *>(xn + (size_t)t * D);
#pragma unroll
    for (int u = 0; u < VEC; ++u) {
        const int i = threadIdx.x + u * NT;
        if (i < nv) {
            o[2 * i] = __floats2bfloat162_rn(keep[u].x * s, keep[u].y * s);
            o[2 * i + 1] = __floats2bfloat162_rn(keep[u].z * s, keep[u].w * s);
        }
    }
    for (int i = threadIdx.x + VEC * NT; i < nv; i += NT) {
        const float4 v = r[i];
        o[2 * i] = __floats2bfloat162_rn(v.x * s, v.y * s);
        o[2 * i + 1] = __floats2bfloat162_rn(v.z * s, v.w * s);
    }
}

__global__ void __launch_bounds__(256)
k_sa_setup(int T, int32_t *offsets) {
    ptx::grid_dependency_wait();
    write_trivial_dispatch(T, offsets);
}

// qkv [T, (Hq + 2 Hkv) 128] fp32 (the sum of n_part partial projections
// part_stride floats apart) -> q [T, Hq, 128] fp32 (rotated); rotated keys
// and the values to the caches [n_seq, Hkv, L, 128] in bf16.  A block holds
// kRopeRows head rows of one token, 64 threads each: thread i turns the pair
// (i, i + 64) of a query or key head, or copies two value elements.
constexpr int kRopeRows = 8;  // head rows per block
constexpr int kRopeTokens = 4;  // tokens per block, one after the other

__global__ void __launch_bounds__(kRopeRows * kHeadDim / 2)
k_rope_cache(int T, int Hq, int Hkv, int n_seq, int L, RopeRates rates,
             const int32_t *__restrict__ seq, const int32_t *__restrict__ pos,
             const float *__restrict__ qkv, int n_part, long long part_stride,
             float *__restrict__ q, bf16 *__restrict__ q16, bf16 *__restrict__ kc,
             bf16 *__restrict__ vc, unsigned *err) {
    // a decode-type call (no 128-token prefill tile): the tensor-core decode
    // attention, one CTA per SM on the SMs this small grid leaves free, may
    // launch now and set itself up while this kernel runs
    if (T < kAttnTcTile) ptx::launch_dependents();
    ptx::grid_dependency_wait();
    constexpr int H2 = kHeadDim / 2;
    static_assert(kRopeTokens * H2 <= kRopeRows * H2, "one thread per (token, pair)");
    __shared__ float cs_s[kRopeTokens][H2], sn_s[kRopeTokens][H2];
    __shared__ int seq_s[kRopeTokens], pos_s[kRopeTokens];
    const int hr = blockIdx.x * kRopeRows + threadIdx.x / H2;
    const int i = threadIdx.x % H2;
    const int nq = Hq * kHeadDim, nkv = Hkv * kHeadDim;
    const int tb = blockIdx.y * kRopeTokens;
    const int nt = min(kRopeTokens, T - tb);
    // every token's pair first (independent loads in flight together, and
    // in flight while the angles are formed), the projection's partial sums
    // added in order
    const bool row_ok = hr < Hq + 2 * Hkv;
    float av[kRopeTokens], bv[kRopeTokens];
#pragma unroll
    for (int u = 0; u < kRopeTokens; ++u) {
        av[u] = 0.f;
        bv[u] = 0.f;
        if (row_ok && u < nt) {
            const float *row = qkv + (size_t)(tb + u) * (nq + 2 * nkv) + (size_t)hr * kHeadDim;
            for (int k = 0; k < n_part; ++k) {
                av[u] += row[k * part_stride + i];
                bv[u] += row[k * part_stride + i + H2];
            }
        }
    }
    // the angles of every token of the block: pair i of token tb+u turns by
    // pos * rate_i, formed and reduced to [-pi, pi] in fp64 (exact to far
    // below fp32 resolution at any cache position), evaluated in fp32
    if (threadIdx.x < nt * H2) {
        const int u = threadIdx.x / H2, k = threadIdx.x % H2;
        const int sq = seq[tb + u], p = pos[tb + u];
        const bool ok = sq >= 0 && sq < n_seq && p >= 0 && p < L;
        if (k == 0) {
            seq_s[u] = ok ? sq : -1;
            pos_s[u] = p;
            if (!ok && blockIdx.x == 0) set_error(err, kErrIndex);
        }
        constexpr double kTwoPi = 6.283185307179586;
        const double ang = (double)(ok ? p : 0) * rates.w[k];
        const double red = fma(-rint(ang * (1.0 / kTwoPi)), kTwoPi, ang);
        sincosf((float)red, &sn_s[u][k], &cs_s[u][k]);
    }
    __syncthreads();
    if (!row_ok) return;
#pragma unroll
    for (int u = 0; u < kRopeTokens; ++u) {
        if (u >= nt) break;
        const int t = tb + u, sq = seq_s[u], p = pos_s[u];
        const float a = av[u], b = bv[u];
        if (hr >= Hq + Hkv) {  // a value head: stored as it is
            if (sq < 0) continue;
            bf16 *vd = vc + (((size_t)sq * Hkv + (hr - Hq - Hkv)) * L + p) * kHeadDim;
            vd[i] = __float2bfloat16_rn(a);
            vd[i + H2] = __float2bfloat16_rn(b);
            continue;
        }
        const float cs = cs_s[u][i], sn = sn_s[u][i];
        const float x0 = a * cs - b * sn, x1 = b * cs + a * sn;
        if (hr < Hq) {
            float *qo = q + (size_t)t * nq + (size_t)hr * kHeadDim;
            qo[i] = x0;
            qo[i + H2] = x1;
            if (q16) {  // the tensor-core attention's copy
                bf16 *qh = q16 + (size_t)t * nq + (size_t)hr * kHeadDim;
                qh[i] = __float2bfloat16_rn(x0);
                qh[i + H2] = __float2bfloat16_rn(x1);
            }
        } else if (sq >= 0) {
            bf16 *kd = kc + (((size_t)sq * Hkv + (hr - Hq)) * L + p) * kHeadDim;
            kd[i] = __float2bfloat16_rn(x0);
            kd[i + H2] = __float2bfloat16_rn(x1);
        }
    }
}

// 8-byte asynchronous global -> shared copy (per thread) and its group wait.
__device__ __forceinline__ void cp_async8(void *dst_smem, const void *src) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8;" ::"r"(ptx::smem_u32(dst_smem)),
                 "l"(src)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
    asm volatile("cp.async.wait_group 0;" ::: "memory");
}

__device__ __forceinline__ void unpack4(uint2 u, float (&o)[4]) {
    unpack_bf16x2(u.x, o[0], o[1]);
    unpack_bf16x2(u.y, o[2], o[3]);
}

// One CTA per (split s, token t, key/value head g); the split covers cache
// positions [j0, j1) of token t's sequence.  Each warp takes tiles of 32
// positions (tile i of warp w starts at j0 + 32*(w + kAttnWarps*i)):
//   scores: lane l owns position l of the tile and computes the full dot
//     products with the G query heads (queries pre-scaled in shared memory),
//     so no cross-lane reduction per position;
//   softmax: per head, one warp max and one warp sum per tile update the
//     running (max m, sum l) and rescale the accumulator;
//   values: lane l owns dims [4l, 4l+4); for each position of the tile the
//     head weights are broadcast from the owning lane and the value row is
//     read coalesced.
// Partial results per (t, query head, s): m, l, and the weighted value sum
// (relative to m).
template <int G>
__global__ void __launch_bounds__(kAttnThreads)
k_attn_partial(int Hq, int Hkv, int n_seq, int L, int n_split, int n_tg,
               const int32_t *__restrict__ seq, const int32_t *__restrict__ pos,
               const float *__restrict__ q, const bf16 *__restrict__ kc,
               const bf16 *__restrict__ vc, float *__restrict__ part_ml,
               float *__restrict__ part_acc, bf16 *__restrict__ ctx,
               const int *__restrict__ tile_ok) {
    ptx::grid_dependency_wait();
    __shared__ __align__(16) float qs[G][kHeadDim];
    __shared__ float sm_m[kAttnWarps][G], sm_l[kAttnWarps][G];
    __shared__ float sm_acc[kAttnWarps][G][kHeadDim];
    __shared__ __align__(16) bf16 vtile[kAttnWarps][32][kHeadDim];  // each warp's value tile
    __shared__ unsigned char s_ok[kMaxSaTokens / kAttnTcTile];
    const int s = blockIdx.x;
    // (token, key/value head) items blockIdx.y, + gridDim.y, ...: a call
    // whose prefill tiles went to the tensor cores launches a bounded grid
    // that skips them (their flags read once into shared memory), instead
    // of a block per item
    if (tile_ok) {
        const int n_tiles = (n_tg / Hkv + kAttnTcTile - 1) / kAttnTcTile;
        for (int i = threadIdx.x; i < n_tiles; i += blockDim.x) s_ok[i] = tile_ok[i] ? 1 : 0;
        __syncthreads();
    }
    for (int tg = blockIdx.y; tg < n_tg; tg += gridDim.y) {
        const int t = tg / Hkv, g = tg - t * Hkv;
        if (tile_ok && s_ok[t / kAttnTcTile]) continue;  // the tensor-core kernel has it
        const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
        const int sq = seq[t], p = pos[t];
        const bool ok = sq >= 0 && sq < n_seq && p >= 0 && p < L;
        const int n = ok ? p + 1 : 0;
        const int chunk = (n + n_split - 1) / n_split;
        const int j0 = min(n, s * chunk), j1 = min(n, j0 + chunk);
        const float scale = 1.0f / sqrtf((float)kHeadDim);
        // the queries as stored activations: rounded to bf16, as the
        // tensor-core kernels read them
        for (int i = threadIdx.x; i < G * kHeadDim; i += blockDim.x)
            qs[i / kHeadDim][i % kHeadDim] =
                __bfloat162float(
                    __float2bfloat16_rn(q[((size_t)t * Hq + g * G) * kHeadDim + i])) *
                scale;
        __syncthreads();

        float m[G], l[G], acc[G][4];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            m[h] = -INFINITY;
            l[h] = 0.f;
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[h][i] = 0.f;
        }
        const size_t base = ok ? ((size_t)sq * Hkv + g) * L * kHeadDim : 0;
        const bf16 *kb = kc + base;
        const bf16 *vb = vc + base;
        for (int jt = j0 + warp * 32; jt < j1; jt += kAttnWarps * 32) {
            const int jl = jt + lane;  // this lane's position
            const bool live = jl < j1;
            const int nt = min(32, j1 - jt);
            // the tile's value rows land in shared memory while the scores are
            // computed: lane l copies bytes [8l, 8l+8) of every row
            __syncwarp();
            for (int u = 0; u < nt; ++u)
                cp_async8(&vtile[warp][u][lane * 4], vb + (size_t)(jt + u) * kHeadDim + lane * 4);
            cp_async_commit();
            float sc[G];
#pragma unroll
            for (int h = 0; h < G; ++h) sc[h] = 0.f;
            if (live) {
                const uint4 *kr = reinterpret_cast<const uint4 *>(kb + (size_t)jl * kHeadDim);
#pragma unroll
                for (int c = 0; c < kHeadDim / 32; ++c) {  // 32 dims per step
                    uint4 u[4];
#pragma unroll
                    for (int v = 0; v < 4; ++v) u[v] = __ldg(kr + c * 4 + v);
#pragma unroll
                    for (int v = 0; v < 4; ++v) {
                        float k8[8];
                        unpack_bf16x2(u[v].x, k8[0], k8[1]);
                        unpack_bf16x2(u[v].y, k8[2], k8[3]);
                        unpack_bf16x2(u[v].z, k8[4], k8[5]);
                        unpack_bf16x2(u[v].w, k8[6], k8[7]);
                        const int d0 = c * 32 + v * 8;
#pragma unroll
                        for (int h = 0; h < G; ++h) {
                            const float4 qa = *reinterpret_cast<const float4 *>(&qs[h][d0]);
                            const float4 qb = *reinterpret_cast<const float4 *>(&qs[h][d0 + 4]);
                            sc[h] = fmaf(qa.x, k8[0], sc[h]);
                            sc[h] = fmaf(qa.y, k8[1], sc[h]);
                            sc[h] = fmaf(qa.z, k8[2], sc[h]);
                            sc[h] = fmaf(qa.w, k8[3], sc[h]);
                            sc[h] = fmaf(qb.x, k8[4], sc[h]);
                            sc[h] = fmaf(qb.y, k8[5], sc[h]);
                            sc[h] = fmaf(qb.z, k8[6], sc[h]);
                            sc[h] = fmaf(qb.w, k8[7], sc[h]);
                        }
                    }
                }
            }
            float w[G];
#pragma unroll
            for (int h = 0; h < G; ++h) {
                float tm = live ? sc[h] : -INFINITY;
#pragma unroll
                for (int o = 16; o > 0; o >>= 1)
                    tm = fmaxf(tm, __shfl_xor_sync(0xffffffffu, tm, o));
                const float mn = fmaxf(m[h], tm);  // finite: the tile has a live lane
                const float corr = expf(m[h] - mn);  // 0 while m is -inf
                w[h] = live ? expf(sc[h] - mn) : 0.f;
                l[h] = l[h] * corr + warp_sum(w[h]);
#pragma unroll
                for (int i = 0; i < 4; ++i) acc[h][i] *= corr;
                m[h] = mn;
            }
            cp_async_wait_all();
            __syncwarp();
#pragma unroll 4
            for (int u = 0; u < nt; ++u) {
                float v4[4];
                unpack4(*reinterpret_cast<const uint2 *>(&vtile[warp][u][lane * 4]), v4);
#pragma unroll
                for (int h = 0; h < G; ++h) {
                    const float wu = __shfl_sync(0xffffffffu, w[h], u);
#pragma unroll
                    for (int i = 0; i < 4; ++i) acc[h][i] = fmaf(wu, v4[i], acc[h][i]);
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
            if (n_split == 1) {  // the only split: this is the result
                ctx[((size_t)t * Hq + g * G + h) * kHeadDim + d] =
                    __float2bfloat16_rn(Ls > 0.f ? A / Ls : 0.f);
                continue;
            }
            const size_t o = ((size_t)t * Hq + g * G + h) * n_split + s;
            if (d == 0) {
                part_ml[2 * o] = M;
                part_ml[2 * o + 1] = Ls;
            }
            part_acc[o * kHeadDim + d] = A;
        }
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
    ptx::launch_dependents();  // the output projection may start streaming its weights
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

// The tensor-core attention's bf16 copy of fp32 queries, for a call that
// brings its own queries (moe_sa_attend); in the whole block the rotary
// kernel writes it.  n4 groups of four elements.
__global__ void __launch_bounds__(256)
k_q_bf16(long long n4, const float *__restrict__ q, bf16 *__restrict__ q16) {
    ptx::grid_dependency_wait();
    const float4 *a = reinterpret_cast<const float4 *>(q);
    __nv_bfloat162 *o = reinterpret_cast<__nv_bfloat162 *>(q16);
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (long long)gridDim.x * blockDim.x) {
        const float4 v = a[i];
        o[2 * i] = __floats2bfloat162_rn(v.x, v.y);
        o[2 * i + 1] = __floats2bfloat162_rn(v.z, v.w);
    }
}

// resid += y_0 + ... + y_{n_part-1} (partial projections n4 float4 apart,
// added in order before the residual).
__global__ void __launch_bounds__(256)
k_residual_add(long long n4, int n_part, float *__restrict__ resid, const float *__restrict__ y) {
    ptx::grid_dependency_wait();
    float4 *r = reinterpret_cast<float4 *>(resid);
    const float4 *a = reinterpret_cast<const float4 *>(y);
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < n4;
         i += (long long)gridDim.x * blockDim.x) {
        float4 w = a[i];
        for (int k = 1; k < n_part; ++k) {
            const float4 u = a[k * n4 + i];
            w.x += u.x;
            w.y += u.y;
            w.z += u.z;
            w.w += u.w;
        }
        float4 v = r[i];
        v.x += w.x;
        v.y += w.y;
        v.z += w.z;
        v.w += w.w;
        r[i] = v;
    }
}

// Decoder layers: resid[t] += sum of the partial projections, then the MoE
// block's input xn[t] = bf16(RMSNorm0(resid[t])) -- the residual add of the
// attention block and the pre-norm of the MoE block in one pass, one block
// per token with the row in registers (NT threads x VEC float4: 1024 x 4 for
// decode batches, 256 x 16 for larger ones, as k_sa_prenorm; D <= 16384).
constexpr int kResNormCap = 4 * 4 * kNormThreads;  // row length the fused form holds

template <int NT, int VEC>
__global__ void __launch_bounds__(NT)
k_residual_prenorm(int T, int D, int n_part, float *__restrict__ resid, const float *__restrict__ y,
                   bf16 *__restrict__ xn, float eps) {
    static_assert(4 * NT * VEC == kResNormCap, "both forms hold a row of kResNormCap");
    ptx::grid_dependency_wait();
    __shared__ float red[NT / 32];
    const int t = blockIdx.x;
    const int nv = D >> 2;
    const long long stride4 = (long long)T * nv;  // between partial projections, in float4
    float4 *r = reinterpret_cast<float4 *>(resid + (size_t)t * D);
    const float4 *a = reinterpret_cast<const float4 *>(y + (size_t)t * D);
    float4 keep[VEC];
    float ss = 0.f;
#pragma unroll
    for (int u = 0; u < VEC; ++u) {
        const int i = threadIdx.x + u * NT;
        keep[u] = make_float4(0.f, 0.f, 0.f, 0.f);
        if (i < nv) {
            float4 w = a[i];
            for (int k = 1; k < n_part; ++k) {
                const float4 v = a[k * stride4 + i];
                w.x += v.x;
                w.y += v.y;
                w.z += v.z;
                w.w += v.w;
            }
            float4 v = r[i];
            v.x += w.x;
            v.y += w.y;
            v.z += w.z;
            v.w += w.w;
            r[i] = v;
            keep[u] = v;
            ss += v.x * v.x + v.y * v.y + v.z * v.z + v.w * v.w;
        }
    }
    ss = warp_sum(ss);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
    __syncthreads();
    float tot = 0.f;
#pragma unroll
    for (int w = 0; w < NT / 32; ++w) tot += red[w];
    const float sc = 1.0f / sqrtf(tot / (float)D + eps);
    __nv_bfloat162 *o = reinterpret_cast<__nv_bfloat162 *>(xn + (size_t)t * D);
#pragma unroll
    for (int u = 0; u < VEC; ++u) {
        const int i = threadIdx.x + u * NT;
        if (i < nv) {
            o[2 * i] = __floats2bfloat162_rn(keep[u].x * sc, keep[u].y * sc);
            o[2 * i + 1] = __floats2bfloat162_rn(keep[u].z * sc, keep[u].w * sc);
        }
    }
}

// ---- host ------------------------------------------------------------------------

struct SaWs {
    size_t offsets, xn, qkv, q, q16, tile_ok, part_ml, part_acc, ctx, total;
};

SaWs sa_ws(const moe_sa_dims &d, int64_t T) {
    auto up = [](size_t v) { return (v + 255) & ~size_t(255); };
    const size_t nq = (size_t)d.n_heads * kHeadDim;
    const size_t nr = nq + 2 * (size_t)d.n_kv_heads * kHeadDim;
    const size_t splits = (size_t)T * d.n_heads * split_cap((int)T, d.n_kv_heads);
    SaWs L{};
    size_t o = 0;
    L.offsets = o; o += up(2 * 4);
    L.xn = o; o += up((size_t)T * d.d_model * 2);
    // projection outputs (partial sums of a split reduction for up to
    // kRowsMaxTokens tokens): qkv first, later the output projection's rows
    const size_t parts = T <= kRowsMaxTokens ? kRowsMaxParts : 1;
    L.qkv = o; o += up(parts * T * std::max(nr, (size_t)d.d_model) * 4);
    L.q = o; o += up((size_t)T * nq * 4);
    L.q16 = o; o += up((size_t)T * nq * 2);
    L.tile_ok = o; o += up((size_t)(T + kAttnTcTile - 1) / kAttnTcTile * 4);
    L.part_ml = o; o += up(splits * 2 * 4);
    L.part_acc = o; o += up(splits * kHeadDim * 4);
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
};

// W_qkv . xn -> qkv (fp32), then the rotary embedding and the cache writes.
// Whether the call's attention takes the tensor-core prefill kernel for its
// full 128-token tiles (the CUDA-core kernel keeps the others).
bool tc_attention(int T) { return T >= kAttnTcTile && attn_prefill_tc_ok(); }

cudaError_t qkv_rope(const SaCall &c, const void *xn, const void *w_qkv, const int32_t *seq,
                     const int32_t *pos, int n_seq, int L, float *q, void *kc, void *vc,
                     bf16 *q16 = nullptr) {
    const moe_dims pd = proj_dims(c.nr(), c.d.d_model);
    const int32_t *offsets = at<int32_t>(c.ws, c.L.offsets);
    float *qkv = at<float>(c.ws, c.L.qkv);
    cudaError_t e;
    int n_part = 1;
    if (c.T <= kRowsMaxTokens) {
        n_part = gemm_rows_parts(c.d.d_model, c.nr());
        e = launch_gemm_rows_tc(c.T, c.d.d_model, c.nr(), xn, w_qkv, n_part, qkv, c.st,
                                "qkv_rows_tc");
    } else {
        e = launch_gemm_down_tc(pd, c.T, xn, offsets, w_qkv, qkv, c.st, "qkv_gemm_tc");
    }
    if (e != cudaSuccess) return e;
    long long pstride = (long long)c.T * c.nr();
    int Hq = c.d.n_heads, Hkv = c.d.n_kv_heads, ns = n_seq, Lv = L;
    RopeRates rates;
    for (int i = 0; i < kHeadDim / 2; ++i)
        rates.w[i] = pow((double)c.d.rope_base, -2.0 * i / (double)kHeadDim);
    const float *qkvc = qkv;
    bf16 *kcp = static_cast<bf16 *>(kc), *vcp = static_cast<bf16 *>(vc);
    unsigned *err = device_info().err;
    int Tv = c.T;
    void *args[] = {&Tv,     &Hq,      &Hkv, &ns,  &Lv,  &rates, &seq, &pos,
                    &qkvc,   &n_part,  &pstride, &q, &q16, &kcp, &vcp, &err};
    LaunchScope ls("rope_cache", c.st);
    const int rows = Hq + 2 * Hkv;
    return launch_pdl((const void *)k_rope_cache,
                      dim3((rows + kRopeRows - 1) / kRopeRows, (c.T + kRopeTokens - 1) / kRopeTokens),
                      dim3(kRopeRows * kHeadDim / 2), 0, c.st, args);
}

// Whether decode-type calls (no full prefill tile) attend on the tensor
// cores; MOE_ATTN_CUDA_CORES=1 keeps them on the CUDA-core kernel.
bool decode_tc() {
    static const bool off = [] {
        const char *v = getenv("MOE_ATTN_CUDA_CORES");
        return v && v[0] == '1';
    }();
    return !off && attn_decode_tc_ok();
}

// Whether a call of T tokens wants the bf16 copy of its queries (one of the
// tensor-core attention kernels reads it).
bool wants_q16(int T) { return tc_attention(T) || decode_tc(); }

// Attention over the caches.  A call with 128 or more tokens: full prefill
// tiles on the tensor cores, the rest on the CUDA-core kernel (one split);
// a smaller call: the decode kernel on the tensor cores.  Per-split
// partials, when there are several splits, are merged last.
cudaError_t attend(const SaCall &c, const float *q, const int32_t *seq, const int32_t *pos,
                   int n_seq, int L, const void *kc, const void *vc, void *ctx,
                   const bf16 *q16 = nullptr) {
    const int Hq = c.d.n_heads, Hkv = c.d.n_kv_heads, G = Hq / Hkv;
    int ns = n_split_for(c.T, Hkv, L);
    int *tile_ok = nullptr;
    float *ml = at<float>(c.ws, c.L.part_ml), *acc = at<float>(c.ws, c.L.part_acc);
    bf16 *cp = static_cast<bf16 *>(ctx);
    if (q16 && tc_attention(c.T)) {  // full prefill tiles on the tensor cores, the rest below
        tile_ok = at<int>(c.ws, c.L.tile_ok);
        cudaError_t e = launch_attn_prefill_tc(c.T, Hq, Hkv, n_seq, L, seq, pos, q16, kc, vc, ctx,
                                               tile_ok, c.st);
        if (e != cudaSuccess) return e;
        ns = 1;
    } else if (q16 && decode_tc()) {
        // splits merged inside the kernel (a cluster per token and key/value head)
        return launch_attn_decode_tc(c.T, Hq, Hkv, n_seq, L, attn_decode_tc_splits(c.T, Hkv, L),
                                     seq, pos, q16, kc, vc, ctx, c.st);
    }
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
        const int *tok = tile_ok;
        int n_tg = c.T * Hkv;
        // (a prefill call usually leaves no token: one wave of CTAs that
        // read the tile flags and find nothing to do; otherwise a block per
        // item up to the grid's y limit, the kernel looping past it)
        const int gy = std::min(n_tg, tile_ok ? 2 * device_info().sm_count : 65535);
        void *args[] = {&Hqv, &Hkvv, &nsq, &Lv, &ns, &n_tg, &seq, &pos, &q, &kcp, &vcp, &ml,
                        &acc, &cp, &tok};
        LaunchScope ls("attention", c.st);
        cudaError_t e = launch_pdl(kern, dim3(ns, gy), dim3(kAttnThreads), 0, c.st, args);
        if (e != cudaSuccess || ns == 1) return e;
    }
    const float *mlc = ml, *accc = acc;
    void *args[] = {&ns, &mlc, &accc, &cp};
    LaunchScope ls("attn_merge", c.st);
    return launch_pdl((const void *)k_attn_merge, dim3(c.T * Hq), dim3(kHeadDim * kMergeGroups), 0,
                      c.st, args);
}

// resid += W_o . ctx
// resid += W_o . ctx; with xn_next (decoder layers, D <= 4 * 4 * 1024) the
// MoE block's normalised input is written in the same pass.
cudaError_t out_proj(const SaCall &c, const void *ctx, const void *w_o, float *resid,
                     bf16 *xn_next = nullptr, float eps = 0.f) {
    const moe_dims pd = proj_dims(c.d.d_model, c.nq());
    const int32_t *offsets = at<int32_t>(c.ws, c.L.offsets);
    float *y = at<float>(c.ws, c.L.qkv);
    int n_part = 1;
    cudaError_t e;
    if (c.T <= kRowsMaxTokens) {
        n_part = gemm_rows_parts(c.nq(), c.d.d_model);
        e = launch_gemm_rows_tc(c.T, c.nq(), c.d.d_model, ctx, w_o, n_part, y, c.st, "o_rows_tc");
    } else {
        e = launch_gemm_down_tc(pd, c.T, ctx, offsets, w_o, y, c.st, "o_gemm_tc");
    }
    if (e != cudaSuccess) return e;
    if (xn_next) {
        int Tv = c.T, D = c.d.d_model;
        const float *yc = y;
        void *args[] = {&Tv, &D, &n_part, &resid, &yc, &xn_next, &eps};
        LaunchScope ls("residual_prenorm", c.st);
        if (c.T >= kNormWideMinTokens)
            return launch_pdl((const void *)k_residual_prenorm<kNormThreadsWide, kNormMaxVec>,
                              dim3(c.T), dim3(kNormThreadsWide), 0, c.st, args);
        return launch_pdl((const void *)k_residual_prenorm<kNormThreads, 4>, dim3(c.T),
                          dim3(kNormThreads), 0, c.st, args);
    }
    long long n4 = (long long)c.T * c.d.d_model / 4;
    const long long cap = (long long)device_info().sm_count * 8;
    const int grid = (int)std::max(1LL, std::min((n4 + 255) / 256, cap));
    const float *yc = y;
    void *args[] = {&n4, &n_part, &resid, &yc};
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
    int32_t *off = at<int32_t>(c.ws, c.L.offsets);
    void *args[] = {&Tv, &off};
    LaunchScope ls("sa_setup", c.st);
    return cuda_status(launch_pdl((const void *)k_sa_setup, dim3(1), dim3(256), 0, c.st, args));
}

}  // namespace
}  // namespace moe

using namespace moe;

namespace {

moe_status sa_forward_impl(const moe_sa_dims *dims, int32_t T, const int32_t *seq,
                           const int32_t *pos, int32_t n_seq, int32_t max_len, float *resid,
                           const void *w_qkv, const void *w_o, void *k_cache, void *v_cache,
                           float eps, void *ws, size_t ws_bytes, moe_stream_t stream,
                           bf16 *xn_next) {
    moe_status s = check_sa_call(dims, T, seq, pos, n_seq, max_len);
    if (s != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(resid) || !ok_ptr(w_qkv) || !ok_ptr(w_o) || !ok_ptr(k_cache) ||
        !ok_ptr(v_cache) || !(eps > 0.f))
        return MOE_ERR_INVALID_ARG;
    if ((s = check_ws(dims, T, ws, ws_bytes)) != MOE_OK) return s;
    SaCall c{*dims, T, (cudaStream_t)stream, ws, sa_ws(*dims, T)};
    if (!tc_path_ok(proj_dims(c.nr(), dims->d_model)) ||
        !tc_path_ok(proj_dims(dims->d_model, c.nq())))
        return MOE_ERR_UNSUPPORTED;
    bf16 *xn = at<bf16>(ws, c.L.xn);
    float *q = at<float>(ws, c.L.q);
    bf16 *ctx = at<bf16>(ws, c.L.ctx);
    {
        int Tv = T, D = dims->d_model;
        const float *rc = resid;
        int32_t *off = at<int32_t>(ws, c.L.offsets);
        void *args[] = {&Tv, &D, &rc, &xn, &eps, &off};
        LaunchScope ls("sa_prenorm", c.st);
        const cudaError_t e =
            T >= kNormWideMinTokens
                ? launch_pdl((const void *)k_sa_prenorm<kNormThreadsWide, kNormMaxVec>, dim3(T),
                             dim3(kNormThreadsWide), 0, c.st, args)
                : launch_pdl((const void *)k_sa_prenorm<kNormThreads, 4>, dim3(T),
                             dim3(kNormThreads), 0, c.st, args);
        if (e != cudaSuccess) return MOE_ERR_CUDA;
    }
    bf16 *q16 = wants_q16(T) ? at<bf16>(ws, c.L.q16) : nullptr;
    cudaError_t e = qkv_rope(c, xn, w_qkv, seq, pos, n_seq, max_len, q, k_cache, v_cache, q16);
    if (e == cudaSuccess) e = attend(c, q, seq, pos, n_seq, max_len, k_cache, v_cache, ctx, q16);
    if (e == cudaSuccess) e = out_proj(c, ctx, w_o, resid, xn_next, eps);
    return cuda_status(e);
}

}  // namespace

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
    if (!tc_path_ok(proj_dims(c.nr(), dims->d_model))) return MOE_ERR_UNSUPPORTED;
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
    // the same kernels as the whole block: the tensor-core attention
    // kernels, from a bf16 copy of the queries
    bf16 *q16 = nullptr;
    if (wants_q16(T)) {
        q16 = at<bf16>(ws, c.L.q16);
        long long n4 = (long long)T * dims->n_heads * dims->head_dim / 4;
        const float *qc = q;
        void *args[] = {&n4, &qc, &q16};
        const int blocks = (int)std::min<long long>((n4 + 255) / 256, 4LL * device_info().sm_count);
        LaunchScope ls("q_bf16", c.st);
        cudaError_t e = launch_pdl((const void *)k_q_bf16, dim3(std::max(blocks, 1)), dim3(256), 0,
                                   c.st, args);
        if (e != cudaSuccess) return cuda_status(e);
    }
    return cuda_status(attend(c, q, seq, pos, n_seq, max_len, k_cache, v_cache, ctx, q16));
}

moe_status moe_sa_forward(const moe_sa_dims *dims, int32_t T, const int32_t *seq,
                          const int32_t *pos, int32_t n_seq, int32_t max_len, float *resid,
                          const void *w_qkv, const void *w_o, void *k_cache, void *v_cache,
                          float eps, void *ws, size_t ws_bytes, moe_stream_t stream) {
    MOE_INJECT("moe_sa_forward");
    return sa_forward_impl(dims, T, seq, pos, n_seq, max_len, resid, w_qkv, w_o, k_cache, v_cache,
                           eps, ws, ws_bytes, stream, nullptr);
}


moe_status moe_decoder_workspace_size(const moe_sa_dims *attn, const moe_dims *moe_d,
                                      int32_t max_tokens, size_t *bytes) {
    if (!bytes) return MOE_ERR_INVALID_ARG;
    size_t a = 0, b = 0, c = 0;
    moe_status s = moe_sa_workspace_size(attn, max_tokens, &a);
    if (s != MOE_OK) return s;
    if ((s = moe_workspace_size(moe_d, max_tokens, &b)) != MOE_OK) return s;
    if ((s = moe_stack_workspace_size(moe_d, max_tokens, &c)) != MOE_OK) return s;
    // the MoE block's normalised input, then the attention block's or the
    // MoE layer's scratch (never live together)
    const size_t xn = ((size_t)max_tokens * attn->d_model * 2 + 255) & ~size_t(255);
    *bytes = std::max(xn + std::max(a, b), std::max(a, c));
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
    // the attention block's residual add and the MoE block's pre-norm run as
    // one kernel when a row fits its registers; otherwise as the stack does
    const bool fused = attn->d_model <= kResNormCap;
    const size_t xn_bytes = ((size_t)T * attn->d_model * 2 + 255) & ~size_t(255);
    bf16 *xn = static_cast<bf16 *>(ws);
    void *inner = static_cast<char *>(ws) + xn_bytes;
    for (int l = 0; l < n_layers; ++l) {
        if (fused) {
            s = sa_forward_impl(attn, T, seq, pos, n_seq, max_len, resid, w_qkv[l], w_o[l],
                                k_cache[l], v_cache[l], eps, inner, ws_bytes - xn_bytes, stream,
                                xn);
            if (s != MOE_OK) return s;
            // resid <- resid + MoE_l(xn): the combine reads each residual
            // element before it writes the same element
            s = moe_layer_forward(moe_d, T, xn, w_router[l], w1[l], v1[l], w2[l], resid, resid,
                                  inner, ws_bytes - xn_bytes, stream);
        } else {
            s = moe_sa_forward(attn, T, seq, pos, n_seq, max_len, resid, w_qkv[l], w_o[l],
                               k_cache[l], v_cache[l], eps, ws, ws_bytes, stream);
            if (s != MOE_OK) return s;
            s = moe_stack_forward(moe_d, 1, T, &w_router[l], &w1[l], &v1[l], &w2[l], resid, eps,
                                  ws, ws_bytes, stream);
        }
        if (s != MOE_OK) return s;
    }
    return MOE_OK;
}

}  // extern "C"
