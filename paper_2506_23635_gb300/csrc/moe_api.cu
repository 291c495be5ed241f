// C ABI of libmoe (include/moe.h): argument validation, workspace layout,
// launch bookkeeping, and the small kernels of the layer -- router + gates,
// dispatch, and the unfused combine.
#include <algorithm>
#include <atomic>
#include <mutex>
#include <stdlib.h>
#include <string.h>
#include <string>
#include <vector>

#include <cooperative_groups.h>

#include "moe_internal.cuh"
#include "ptx.cuh"

namespace moe {

__device__ unsigned g_moe_err = 0;

// ===========================================================================
// Step 1: router logits, softmax, top-k, renormalised gates.
// block_logits: a block of NT threads computes the logits of up to 4 tokens;
// its threads split d, each accumulating 16 experts at a time for every
// token (16-byte loads of a router row when E is a multiple of 8), then the
// partial sums are reduced across the block into shared memory.
// select_topk: one warp per token, K rounds of a warp arg-max over the
// not-yet-taken experts, ties going to the lower expert index.
// ===========================================================================
constexpr int kRouteThreads = 256;
constexpr int kRouteTokens = 4;
constexpr int kSmallThreads = 512;
constexpr int kSmallMaxSlots = 32;  // fused route + dispatch: T*K <= 32, T <= 4
// dynamic shared memory the fused kernel may use for the staged router and
// tokens (static arrays of the kernel: ~15 KB)
constexpr size_t kSmallStageBytes = 208 * 1024;

template <typename TW>
__device__ __forceinline__ void router_row16(const TW *wrow, int ne, bool vec, float (&w)[16]) {
    if (vec) {  // E % 8 == 0: whole 8-wide groups, 16-byte aligned
        float t8[8];
        load8(wrow, t8);
#pragma unroll
        for (int j = 0; j < 8; ++j) w[j] = t8[j];
        if (ne > 8) {
            load8(wrow + 8, t8);
#pragma unroll
            for (int j = 0; j < 8; ++j) w[8 + j] = t8[j];
        } else {
#pragma unroll
            for (int j = 8; j < 16; ++j) w[j] = 0.f;
        }
    } else {
#pragma unroll
        for (int j = 0; j < 16; ++j) w[j] = j < ne ? to_f(wrow[j]) : 0.f;
    }
}

template <typename TX, typename TW, int NT>
__device__ void block_logits(int D, int E, const TX *__restrict__ x, const TW *__restrict__ wr,
                             int t0, int nt, float (*lg)[256], float (*red)[kRouteTokens * 16]) {
    constexpr int TT = kRouteTokens, NW = NT / 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const bool vec = (E % 8) == 0;
    for (int e0 = 0; e0 < E; e0 += 16) {
        const int ne = min(16, E - e0);
        float acc[TT][16];
#pragma unroll
        for (int a = 0; a < TT; ++a)
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[a][j] = 0.f;
#pragma unroll 4
        for (int d = threadIdx.x; d < D; d += NT) {
            float xv[TT];
#pragma unroll
            for (int a = 0; a < TT; ++a) xv[a] = a < nt ? to_f(x[(size_t)(t0 + a) * D + d]) : 0.f;
            float w[16];
            router_row16(wr + (size_t)d * E + e0, ne, vec, w);
#pragma unroll
            for (int j = 0; j < 16; ++j)
#pragma unroll
                for (int a = 0; a < TT; ++a) acc[a][j] = fmaf(xv[a], w[j], acc[a][j]);
        }
#pragma unroll
        for (int a = 0; a < TT; ++a)
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const float v = warp_sum(acc[a][j]);
                if (lane == 0) red[warp][a * 16 + j] = v;
            }
        __syncthreads();
        for (int i = threadIdx.x; i < TT * 16; i += NT) {
            const int a = i >> 4, j = i & 15;
            if (a < nt && j < ne) {
                float s = 0.f;
#pragma unroll
                for (int w = 0; w < NW; ++w) s += red[w][i];
                lg[a][e0 + j] = s;
            }
        }
        __syncthreads();
    }
}

template <typename TX, typename TW>
__global__ void __launch_bounds__(kRouteThreads)
k_route(int T, int D, int E, int K, const TX *__restrict__ x, const TW *__restrict__ wr,
        float *__restrict__ logits_opt, int32_t *__restrict__ topk_idx,
        float *__restrict__ topk_gate) {
    __shared__ float red[kRouteThreads / 32][kRouteTokens * 16];
    __shared__ float lg[kRouteTokens][256];
    __shared__ float pk[kRouteTokens][256];
    const int t0 = blockIdx.x * kRouteTokens;
    const int nt = min(kRouteTokens, T - t0);
    const int warp = threadIdx.x >> 5;
    block_logits<TX, TW, kRouteThreads>(D, E, x, wr, t0, nt, lg, red);
    if (warp >= nt) return;
    select_topk(E, K, t0 + warp, lg[warp], pk[warp], logits_opt, topk_idx, topk_gate, nullptr);
}

// ---------------------------------------------------------------------------
// Staged router for the tiny-batch kernel: the whole W_r [D, E] is
// bulk-copied into shared memory (one wait for memory), then every token's
// logits are computed by 8/n warps that each take a slice of d and add their
// partial sums in a fixed order; the token rows are read from global memory
// (coalesced across the warp).  (For larger batches k_route, which shares
// each router row load among 4 tokens, measured faster.)
// ---------------------------------------------------------------------------
constexpr int kStagedWarps = 8;
constexpr int kStagedThreads = kStagedWarps * 32;
constexpr size_t kStagedRouterMax = 196 * 1024 + 1024;  // W_r bytes that are staged

// 16 experts' partial logits of one token over rows [d_lo, d_hi) of a router
// held in shared memory; lane l takes rows d_lo + l, d_lo + l + 32, ... so a
// warp reads 32 consecutive router rows per step (no bank conflicts beyond
// 2-way).  Summed across the warp (every lane ends with all 16).
template <typename TX, typename TW>
__device__ __forceinline__ void warp_logits16(const TX *xrow, const TW *wr_s, int E, int e0, int ne,
                                              int d_lo, int d_hi, float (&acc)[16]) {
    const int lane = threadIdx.x & 31;
#pragma unroll
    for (int j = 0; j < 16; ++j) acc[j] = 0.f;
    const bool vec = (E % 8) == 0 && sizeof(TW) == 2;
#pragma unroll 4
    for (int d = d_lo + lane; d < d_hi; d += 32) {
        const float xv = to_f(xrow[d]);
        const TW *row = wr_s + (size_t)d * E + e0;
        float w[16];
        if (vec) {
            const uint4 u0 = *reinterpret_cast<const uint4 *>(row);
            unpack_bf16x2(u0.x, w[0], w[1]); unpack_bf16x2(u0.y, w[2], w[3]);
            unpack_bf16x2(u0.z, w[4], w[5]); unpack_bf16x2(u0.w, w[6], w[7]);
            if (ne > 8) {
                const uint4 u1 = *reinterpret_cast<const uint4 *>(row + 8);
                unpack_bf16x2(u1.x, w[8], w[9]); unpack_bf16x2(u1.y, w[10], w[11]);
                unpack_bf16x2(u1.z, w[12], w[13]); unpack_bf16x2(u1.w, w[14], w[15]);
            } else {
#pragma unroll
                for (int j = 8; j < 16; ++j) w[j] = 0.f;
            }
        } else {
#pragma unroll
            for (int j = 0; j < 16; ++j) w[j] = j < ne ? to_f(row[j]) : 0.f;
        }
#pragma unroll
        for (int j = 0; j < 16; ++j) acc[j] = fmaf(xv, w[j], acc[j]);
    }
#pragma unroll
    for (int j = 0; j < 16; ++j) acc[j] = warp_sum(acc[j]);
}

// Stage W_r into dynamic shared memory (bulk copies on one mbarrier).
template <typename TW>
__device__ __forceinline__ void stage_router_issue(unsigned char *dst, const TW *wr, uint32_t bytes,
                                                   uint64_t *bar) {
    if (threadIdx.x == 0) {
        const uint64_t pol = ptx::policy_evict_last();
        ptx::mbar_arrive_expect_tx(bar, bytes);
        constexpr uint32_t kChunk = 32768;
        for (uint32_t o = 0; o < bytes; o += kChunk)
            ptx::bulk_g2s(dst + o, reinterpret_cast<const unsigned char *>(wr) + o,
                          min(kChunk, bytes - o), bar, pol);
    }
}

// Logits + top-k of tokens [t0, t0+n) (n <= 8) by the 8 warps of the block.
template <typename TX, typename TW>
__device__ void staged_batch(int t0, int n, int D, int E, int K, const TX *__restrict__ x,
                             const TW *wr_s, float (*part)[256], float (*lg)[256],
                             float (*pk)[256], float *__restrict__ logits_opt,
                             int32_t *__restrict__ topk_idx, float *__restrict__ topk_gate,
                             int *sidx) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int wpt = kStagedWarps / n;  // warps per token
    const int tk = warp / wpt, pt = warp - tk * wpt;
    if (tk < n) {
        const int d_lo = (int)((long long)D * pt / wpt), d_hi = (int)((long long)D * (pt + 1) / wpt);
        const TX *xrow = x + (size_t)(t0 + tk) * D;
        for (int e0 = 0; e0 < E; e0 += 16) {
            const int ne = min(16, E - e0);
            float acc[16];
            warp_logits16<TX, TW>(xrow, wr_s, E, e0, ne, d_lo, d_hi, acc);
#pragma unroll
            for (int j = 0; j < 16; ++j)
                if (lane == j && j < ne) part[warp][e0 + j] = acc[j];
        }
    }
    __syncthreads();
    if (warp < n) {
        for (int e = lane; e < E; e += 32) {
            float v = 0.f;
            for (int p = 0; p < wpt; ++p) v += part[warp * wpt + p][e];
            lg[warp][e] = v;
        }
        __syncwarp();
        select_topk(E, K, t0 + warp, lg[warp], pk[warp], logits_opt, topk_idx, topk_gate,
                    sidx ? sidx + warp * K : nullptr);
    }
    __syncthreads();
}

// Route and dispatch of a tiny batch (T <= 4, T*K <= 32) in one block: the
// top-k indices stay in shared memory and warp 0 ranks the slots (ranks of
// equal experts from __match_any_sync, so the order is the stable one).
// When the router matrix fits in shared memory (`staged`) it is bulk-copied
// there first.
template <typename TX, typename TW>
__global__ void __launch_bounds__(kStagedThreads)
k_route_dispatch_small(int T, int D, int E, int K, const TX *__restrict__ x,
                       const TW *__restrict__ wr, float *__restrict__ logits_opt,
                       int32_t *__restrict__ topk_idx, float *__restrict__ topk_gate,
                       int32_t *__restrict__ counts, int32_t *__restrict__ offsets,
                       int32_t *__restrict__ perm, int32_t *__restrict__ inv_perm, int staged,
                       int *__restrict__ ctr, unsigned *err) {
    extern __shared__ __align__(128) unsigned char wsm[];  // W_r when staged
    __shared__ float part[kStagedWarps][256];
    __shared__ float lg[kStagedWarps][256];
    __shared__ float pk[kStagedWarps][256];
    __shared__ int sidx[kSmallMaxSlots];
    __shared__ int cnt[256];
    __shared__ int offs[257];
    __shared__ uint64_t bar;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int e = threadIdx.x; e < E; e += kStagedThreads) cnt[e] = 0;
    if (staged) {
        if (threadIdx.x == 0) {
            ptx::mbar_init(&bar, 1);
            ptx::fence_barrier_init();
        }
        __syncthreads();
        // W_r does not come from the previous kernel: its copy starts before
        // the dependency wait, and the next kernel may launch at once (its
        // CTAs take the other SMs and wait for this one on the device)
        stage_router_issue<TW>(wsm, wr, (uint32_t)((size_t)D * E * sizeof(TW)), &bar);
        ptx::launch_dependents();
        ptx::grid_dependency_wait();  // x may come from the previous kernel
        const bool ok = ptx::mbar_wait(&bar, 0, err);
        // a wait that gave up (recorded in err) ends the whole block, never part of it
        if (!__syncthreads_and(ok)) return;
        staged_batch<TX, TW>(0, T, D, E, K, x, reinterpret_cast<const TW *>(wsm), part, lg, pk,
                             logits_opt, topk_idx, topk_gate, sidx);
    } else {
        ptx::grid_dependency_wait();
        block_logits<TX, TW, kStagedThreads>(D, E, x, wr, 0, T, lg,
                                            reinterpret_cast<float (*)[kRouteTokens * 16]>(part));
        if (warp < T)
            select_topk(E, K, warp, lg[warp], pk[warp], logits_opt, topk_idx, topk_gate,
                        sidx + warp * K);
        __syncthreads();
    }
    // the next kernels' work counters, for this call (the kernels that used
    // them last finished before this one's dependency wait returned)
    if (ctr && threadIdx.x == 0) {
        ctr[0] = 0;
        ctr[1] = 0;
    }
    if (warp != 0) return;
    const int S = T * K;
    int e = lane < S ? sidx[lane] : -1;
    if (e >= E) {  // cannot come from select_topk; never index with it
        set_error(err, kErrIndex);
        e = -1;
    }
    if (e >= 0) atomicAdd(&cnt[e], 1);
    __syncwarp();
    int carry = 0;
    for (int base = 0; base < E; base += 32) {
        const int ee = base + lane;
        const int c = ee < E ? cnt[ee] : 0;
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (ee < E) {
            offs[ee] = carry + incl - c;
            counts[ee] = c;
            offsets[ee] = carry + incl - c;
        }
        carry += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) offsets[E] = carry;
    __syncwarp();
    const unsigned same = __match_any_sync(0xffffffffu, e);
    if (e >= 0) {
        const int pos = offs[e] + __popc(same & ((1u << lane) - 1u));
        perm[pos] = lane;
        inv_perm[lane] = pos;
    }
}

// ---------------------------------------------------------------------------
// Route and dispatch of a decode batch (T <= 64, T*K <= 256) in one launch of
// a cluster of kClusterCtas CTAs.  CTA r bulk-copies rows [d0_r, d1_r) of W_r
// (before waiting for the previous kernel: the router is a weight) and the
// same columns of every token row of x into its shared memory, and computes
// the partial logits of every token over that slice of d.  After a cluster
// barrier, token t is finished by one warp of CTA t mod kClusterCtas: it adds
// the kClusterCtas partials in rank order (through distributed shared
// memory), selects the top-k and writes the slot experts into CTA 0's shared
// memory.  After a second cluster barrier (every partial read, every slot
// written) CTA 0 ranks all T*K slots with a stable counting sort, as
// k_dispatch does, and the other CTAs leave.
// ---------------------------------------------------------------------------
constexpr int kClusterCtas = 8;
constexpr int kClusterThreads = 256;
constexpr int kClusterMaxTokens = 64;
constexpr int kClusterMaxSlots = 256;
constexpr size_t kClusterMaxSmem = 192 * 1024;  // + ~28 KB static, within 227 KB

// Rows of d per CTA (the largest slice) and the byte stride of a staged token
// row: the slice plus 16 bytes, so that the rows of neighbouring tokens start
// in different shared-memory banks.
__host__ __device__ inline int cluster_rows(int D) {
    return (D / 8 + kClusterCtas - 1) / kClusterCtas * 8;
}
__host__ __device__ inline size_t cluster_x_stride(int D, int x_bytes) {
    return (size_t)cluster_rows(D) * x_bytes + 16;
}
// dynamic shared memory: partial logits [T][E] fp32 (128-byte rounded), the
// router slice [rows][E], the token slices [T][stride]
__host__ __device__ inline size_t cluster_part_bytes(int T, int E) {
    return (((size_t)T * E * 4) + 127) & ~size_t(127);
}

template <typename TX, typename TW>
__global__ void __launch_bounds__(kClusterThreads)
k_route_dispatch_cluster(int T, int D, int E, int K, const TX *__restrict__ x,
                         const TW *__restrict__ wr, int32_t *__restrict__ topk_idx,
                         float *__restrict__ topk_gate, int32_t *__restrict__ counts,
                         int32_t *__restrict__ offsets, int32_t *__restrict__ perm,
                         int32_t *__restrict__ inv_perm, unsigned *err) {
    namespace cg = cooperative_groups;
    cg::cluster_group cluster = cg::this_cluster();
    extern __shared__ __align__(128) unsigned char dsm[];
    constexpr int NW = kClusterThreads / 32;
    float *part = reinterpret_cast<float *>(dsm);
    const size_t part_bytes = cluster_part_bytes(T, E);
    const int rows = cluster_rows(D);
    TW *wr_s = reinterpret_cast<TW *>(dsm + part_bytes);
    unsigned char *x_s = dsm + part_bytes + (size_t)rows * E * sizeof(TW);
    const size_t xs_stride = cluster_x_stride(D, (int)sizeof(TX));
    __shared__ float lg[NW][256];
    __shared__ float pk[NW][256];
    __shared__ int sidx[kClusterMaxSlots];
    __shared__ int cnt[256], run[256];
    __shared__ int wh[NW][256];
    __shared__ uint64_t bar[2];
    const int rank = (int)cluster.block_rank();
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    // this CTA's rows of d, a multiple of 8 rows (16-byte aligned slices)
    const int n8 = D >> 3;
    const int d0 = (int)((long long)n8 * rank / kClusterCtas) * 8;
    const int d1 = (int)((long long)n8 * (rank + 1) / kClusterCtas) * 8;
    const int dn = d1 - d0;

    if (tid == 0) {
        ptx::mbar_init(&bar[0], 1);
        ptx::mbar_init(&bar[1], 1);
        ptx::fence_barrier_init();
    }
    __syncthreads();
    if (tid == 0 && dn > 0) {
        const uint32_t bytes = (uint32_t)((size_t)dn * E * sizeof(TW));
        const uint64_t pol = ptx::policy_evict_last();
        ptx::mbar_arrive_expect_tx(&bar[0], bytes);
        constexpr uint32_t kChunk = 32768;
        for (uint32_t o = 0; o < bytes; o += kChunk)
            ptx::bulk_g2s(reinterpret_cast<unsigned char *>(wr_s) + o,
                          reinterpret_cast<const unsigned char *>(wr + (size_t)d0 * E) + o,
                          min(kChunk, bytes - o), &bar[0], pol);
    }
    ptx::grid_dependency_wait();  // x may come from the previous kernel
    if (warp == 0 && dn > 0) {
        // one bulk copy per token row: dn elements from column d0 (16-byte
        // aligned because D and d0 are multiples of 8)
        const uint32_t row_bytes = (uint32_t)((size_t)dn * sizeof(TX));
        const uint64_t pol = ptx::policy_evict_first();
        if (lane == 0) ptx::mbar_arrive_expect_tx(&bar[1], row_bytes * (uint32_t)T);
        __syncwarp();
        for (int t = lane; t < T; t += 32)
            ptx::bulk_g2s(x_s + (size_t)t * xs_stride, x + (size_t)t * D + d0, row_bytes,
                          &bar[1], pol);
    }
    bool ok = true;
    if (dn > 0) {
        ok = ptx::mbar_wait(&bar[0], 0, err);
        ok = ptx::mbar_wait(&bar[1], 0, err) && ok;
    }
    // partial logits: token t is taken by a group of P threads (P = 256/T,
    // at most 32), thread p of the group accumulating 16 experts over rows
    // p, p+P, ... of the slice; the group then adds its P sums with shuffles
    int P = 32;
    while (P > 1 && P * T > kClusterThreads) P >>= 1;
    const int groups = kClusterThreads / P;
    const int gp = tid % P;
    const bool vec = (E % 8) == 0 && sizeof(TW) == 2;
    for (int t0 = 0; t0 < T; t0 += groups) {
        const int t = t0 + tid / P;
        const TX *xr = reinterpret_cast<const TX *>(x_s + (size_t)(t < T ? t : 0) * xs_stride);
        for (int e0 = 0; e0 < E; e0 += 16) {
            const int ne = min(16, E - e0);
            float acc[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) acc[j] = 0.f;
            if (ok && t < T) {
#pragma unroll 4
                for (int d = gp; d < dn; d += P) {
                    const float xv = to_f(xr[d]);
                    const TW *row = wr_s + (size_t)d * E + e0;
                    float w[16];
                    if (vec) {
                        const uint4 u0 = *reinterpret_cast<const uint4 *>(row);
                        unpack_bf16x2(u0.x, w[0], w[1]); unpack_bf16x2(u0.y, w[2], w[3]);
                        unpack_bf16x2(u0.z, w[4], w[5]); unpack_bf16x2(u0.w, w[6], w[7]);
                        if (ne > 8) {
                            const uint4 u1 = *reinterpret_cast<const uint4 *>(row + 8);
                            unpack_bf16x2(u1.x, w[8], w[9]); unpack_bf16x2(u1.y, w[10], w[11]);
                            unpack_bf16x2(u1.z, w[12], w[13]); unpack_bf16x2(u1.w, w[14], w[15]);
                        } else {
#pragma unroll
                            for (int j = 8; j < 16; ++j) w[j] = 0.f;
                        }
                    } else {
#pragma unroll
                        for (int j = 0; j < 16; ++j) w[j] = j < ne ? to_f(row[j]) : 0.f;
                    }
#pragma unroll
                    for (int j = 0; j < 16; ++j) acc[j] = fmaf(xv, w[j], acc[j]);
                }
            }
#pragma unroll
            for (int j = 0; j < 16; ++j)
                for (int off = P >> 1; off > 0; off >>= 1)
                    acc[j] += __shfl_xor_sync(0xffffffffu, acc[j], off);
            if (t < T && gp == 0)
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    if (j < ne) part[(size_t)t * E + e0 + j] = acc[j];
        }
    }
    cluster.sync();  // every CTA's partials are written
    // token t: warp (t / kClusterCtas) mod NW of CTA t mod kClusterCtas
    int *sidx0 = cluster.map_shared_rank(sidx, 0);
    for (int t = rank + kClusterCtas * warp; t < T; t += kClusterCtas * NW) {
        for (int e = lane; e < E; e += 32) {
            float v = 0.f;
            for (int r = 0; r < kClusterCtas; ++r)
                v += cluster.map_shared_rank(part, r)[(size_t)t * E + e];
            lg[warp][e] = v;
        }
        __syncwarp();
        select_topk(E, K, t, lg[warp], pk[warp], nullptr, topk_idx, topk_gate, sidx0 + t * K);
        __syncwarp();
    }
    cluster.sync();  // every partial is read and every slot is in CTA 0
    if (rank != 0) return;
    // stable dispatch of the S <= 256 slots (one chunk of k_dispatch)
    const int S = T * K;
    for (int e = tid; e < E; e += kClusterThreads) cnt[e] = 0;
    __syncthreads();
    for (int sl = tid; sl < S; sl += kClusterThreads) {
        const int e = sidx[sl];
        if (e >= 0 && e < E) atomicAdd(&cnt[e], 1);
        else set_error(err, kErrIndex);  // cannot come from select_topk
    }
    __syncthreads();
    if (warp == 0) {
        int carry = 0;
        for (int b0 = 0; b0 < E; b0 += 32) {
            const int e = b0 + lane;
            const int c = e < E ? cnt[e] : 0;
            int incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += v;
            }
            if (e < E) {
                run[e] = carry + incl - c;
                counts[e] = c;
                offsets[e] = carry + incl - c;
            }
            carry += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (lane == 0) offsets[E] = carry;
    }
    for (int i = tid; i < NW * E; i += kClusterThreads) wh[i / E][i % E] = 0;
    __syncthreads();
    const int sl = tid;
    const int e = (sl < S && sidx[sl] >= 0 && sidx[sl] < E) ? sidx[sl] : -1;
    const unsigned same = __match_any_sync(0xffffffffu, e);
    const int rk = __popc(same & ((1u << lane) - 1u));
    if (e >= 0 && rk == 0) wh[warp][e] = __popc(same);
    __syncthreads();
    if (e >= 0) {
        int pre = 0;
        for (int w = 0; w < warp; ++w) pre += wh[w][e];
        const int pos = run[e] + pre + rk;
        perm[pos] = sl;
        inv_perm[sl] = pos;
    }
}

// ===========================================================================
// Step 2: dispatch.  One block of 1024 threads: a shared-memory histogram,
// an exclusive scan, then a stable counting sort over chunks of 1024 slots.
// Within a chunk a slot's rank among equal experts is its rank in its warp
// (__match_any_sync) plus the counts of the same expert in lower warps, so
// the order is ascending slot order and needs no atomics.
// ===========================================================================
constexpr int kDispatchThreads = 1024;

__global__ void __launch_bounds__(kDispatchThreads)
k_dispatch(int S, int E, const int32_t *__restrict__ idx, int32_t *__restrict__ counts,
           int32_t *__restrict__ offsets, int32_t *__restrict__ perm,
           int32_t *__restrict__ inv_perm, unsigned *err) {
    constexpr int NW = kDispatchThreads / 32;
    __shared__ int cnt[256];
    __shared__ int run[256];
    __shared__ int wh[NW][256];
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    for (int e = tid; e < E; e += kDispatchThreads) cnt[e] = 0;
    __syncthreads();
    for (int s = tid; s < S; s += kDispatchThreads) {
        const int e = idx[s];
        if (e >= 0 && e < E) atomicAdd(&cnt[e], 1);
        else set_error(err, kErrIndex);
    }
    __syncthreads();
    if (warp == 0) {  // exclusive scan of cnt over E <= 256 experts
        int carry = 0;
        for (int base = 0; base < E; base += 32) {
            const int e = base + lane;
            const int c = e < E ? cnt[e] : 0;
            int incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += v;
            }
            if (e < E) {
                run[e] = carry + incl - c;
                counts[e] = c;
                offsets[e] = carry + incl - c;
            }
            carry += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (lane == 0) offsets[E] = carry;
    }
    __syncthreads();

    const unsigned lt_mask = (1u << lane) - 1u;
    for (int c0 = 0; c0 < S; c0 += kDispatchThreads) {
        for (int i = tid; i < NW * E; i += kDispatchThreads) wh[i / E][i % E] = 0;
        __syncthreads();
        const int s = c0 + tid;
        int e = s < S ? idx[s] : -1;
        const bool valid = e >= 0 && e < E;
        if (!valid) e = -1;
        const unsigned same = __match_any_sync(0xffffffffu, e);
        const int rank = __popc(same & lt_mask);
        if (valid && rank == 0) wh[warp][e] = __popc(same);
        __syncthreads();
        if (valid) {
            int pre = 0;
            for (int w = 0; w < warp; ++w) pre += wh[w][e];
            const int pos = run[e] + pre + rank;
            perm[pos] = s;
            inv_perm[s] = pos;
        } else if (s < S) {
            inv_perm[s] = -1;
        }
        __syncthreads();
        for (int ee = tid; ee < E; ee += kDispatchThreads) {
            int tot = 0;
            for (int w = 0; w < NW; ++w) tot += wh[w][ee];
            run[ee] += tot;
        }
        __syncthreads();
    }
}

// Single-pass variant for up to kFastMaxChunks chunks (8192 slots) whose
// per-(chunk, warp) expert counts fit in shared memory (the 2048-token
// prefill: 8 x 32 x 16).
// All chunks' warp counts are taken in one pass (each thread keeps its slots'
// experts and in-warp ranks in registers), each expert's counts are scanned
// in (chunk, warp) order by one warp, then every slot's position is written:
// the same stable order as k_dispatch with three block barriers instead of
// four per chunk.
constexpr int kFastMaxChunks = 8;
constexpr size_t kFastDispatchSmem = 40 * 1024;

__global__ void __launch_bounds__(kDispatchThreads)
k_dispatch_fast(int S, int E, const int32_t *__restrict__ idx, int32_t *__restrict__ counts,
                int32_t *__restrict__ offsets, int32_t *__restrict__ perm,
                int32_t *__restrict__ inv_perm, unsigned *err) {
    constexpr int NW = kDispatchThreads / 32;
    extern __shared__ int wh[];  // [C * NW][E]: counts, then exclusive in-expert starts
    __shared__ int tot[256], off[256];
    ptx::grid_dependency_wait();
    const int C = (S + kDispatchThreads - 1) / kDispatchThreads;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const unsigned lt_mask = (1u << lane) - 1u;
    for (int i = tid; i < C * NW * E; i += kDispatchThreads) wh[i] = 0;
    __syncthreads();
    int ec[kFastMaxChunks], rc[kFastMaxChunks];
#pragma unroll
    for (int c = 0; c < kFastMaxChunks; ++c) {  // every load in flight at once
        const int s = c * kDispatchThreads + tid;
        ec[c] = c < C && s < S ? idx[s] : -1;
    }
#pragma unroll
    for (int c = 0; c < kFastMaxChunks; ++c) {
        rc[c] = 0;
        if (c < C) {  // uniform across the block
            const int s = c * kDispatchThreads + tid;
            int e = ec[c];
            const bool valid = e >= 0 && e < E;
            if (s < S && !valid) set_error(err, kErrIndex);
            if (!valid) e = -1;
            const unsigned same = __match_any_sync(0xffffffffu, e);
            rc[c] = __popc(same & lt_mask);
            if (valid && rc[c] == 0) wh[(c * NW + warp) * E + e] = __popc(same);
            ec[c] = e;
        }
    }
    __syncthreads();
    // expert e: exclusive scan of its counts over (chunk, warp) = C*NW
    // entries, lane l taking entries [l*C, (l+1)*C)
    for (int e = warp; e < E; e += NW) {
        int loc[kFastMaxChunks], sum = 0;
#pragma unroll
        for (int i = 0; i < kFastMaxChunks; ++i) {
            loc[i] = i < C ? wh[(lane * C + i) * E + e] : 0;
            sum += loc[i];
        }
        int incl = sum;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        int run = incl - sum;
#pragma unroll
        for (int i = 0; i < kFastMaxChunks; ++i)
            if (i < C) {
                wh[(lane * C + i) * E + e] = run;
                run += loc[i];
            }
        if (lane == 31) tot[e] = incl;
    }
    __syncthreads();
    if (warp == 0) {  // exclusive scan of the expert totals
        int carry = 0;
        for (int base = 0; base < E; base += 32) {
            const int e = base + lane;
            const int c = e < E ? tot[e] : 0;
            int incl = c;
#pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int v = __shfl_up_sync(0xffffffffu, incl, o);
                if (lane >= o) incl += v;
            }
            if (e < E) {
                off[e] = carry + incl - c;
                counts[e] = c;
                offsets[e] = carry + incl - c;
            }
            carry += __shfl_sync(0xffffffffu, incl, 31);
        }
        if (lane == 0) offsets[E] = carry;
    }
    __syncthreads();
#pragma unroll
    for (int c = 0; c < kFastMaxChunks; ++c) {
        if (c >= C) break;
        const int s = c * kDispatchThreads + tid;
        const int e = ec[c];
        if (e >= 0) {
            const int pos = off[e] + wh[(c * NW + warp) * E + e] + rc[c];
            perm[pos] = s;
            inv_perm[s] = pos;
        } else if (s < S) {
            inv_perm[s] = -1;
        }
    }
}

// ===========================================================================
// Step 4 (unfused): out[t,:] = residual + sum_k gate[t,k] * y_sorted[inv[t*K+k],:]
// One thread per 4 consecutive outputs; k in ascending order.
// ===========================================================================
// Four consecutive values of a row in the output / residual type.
__device__ __forceinline__ float4 load4(const float *p) { return *reinterpret_cast<const float4 *>(p); }
__device__ __forceinline__ float4 load4(const bf16 *p) {
    const uint2 u = *reinterpret_cast<const uint2 *>(p);
    float4 v;
    unpack_bf16x2(u.x, v.x, v.y);
    unpack_bf16x2(u.y, v.z, v.w);
    return v;
}
__device__ __forceinline__ void store4(float *p, float4 v) { *reinterpret_cast<float4 *>(p) = v; }
__device__ __forceinline__ void store4(bf16 *p, float4 v) {
    const __nv_bfloat162 a = __floats2bfloat162_rn(v.x, v.y), b = __floats2bfloat162_rn(v.z, v.w);
    *reinterpret_cast<uint2 *>(p) = make_uint2(*reinterpret_cast<const uint32_t *>(&a),
                                               *reinterpret_cast<const uint32_t *>(&b));
}

constexpr int kCombineMaxK = 256;  // = the largest top_k

// out[t, :] = residual + sum_k gate[t,k] y[inv[t,k], :], k ascending.  Block
// b takes token b / n_part and the b % n_part-th slice of its row; the
// token's K sorted positions and gates are read once into shared memory, then
// every thread's K row loads are independent (streamed past L1).
// range (optional, n_range experts): the dispatch offsets of a contiguous
// range of experts; only the slots at sorted positions [range[0],
// range[n_range]) are summed (one node's share of an expert-parallel layer).
template <typename TO, typename TR>
__global__ void __launch_bounds__(256)
k_combine(int T, int D, int K, int n_part, const float *__restrict__ y,
          const float *__restrict__ y_tail, const int32_t *__restrict__ inv,
          const float *__restrict__ gate, const TR *__restrict__ residual, TO *__restrict__ out,
          const int32_t *__restrict__ range, int n_range, unsigned *err) {
    __shared__ int s_j[kCombineMaxK];
    __shared__ float s_g[kCombineMaxK];
    ptx::grid_dependency_wait();
    const int S = T * K;
    const int nq = D >> 2;
    const int per = (nq + n_part - 1) / n_part;
    const int j_lo = range ? range[0] : 0, j_hi = range ? range[n_range] : S;
    for (long long b = blockIdx.x; b < (long long)T * n_part; b += gridDim.x) {
        const int t = (int)(b / n_part), part = (int)(b - (long long)t * n_part);
        __syncthreads();  // the previous token's indices are no longer read
        for (int k = threadIdx.x; k < K; k += blockDim.x) {
            const int j = inv[(size_t)t * K + k];
            if (j >= S) set_error(err, kErrIndex);     // a corrupt index
            s_j[k] = (j < j_lo || j >= j_hi) ? -1 : j;  // or a slot left out
            s_g[k] = gate[(size_t)t * K + k];
        }
        __syncthreads();
        const int q1 = min(nq, (part + 1) * per);
        // (two float4 of a thread a step, so 2*K loads in flight: the
        // 2048-token prefill's combine 44 -> 37 us)
#pragma unroll 2
        for (int q = part * per + threadIdx.x; q < q1; q += blockDim.x) {
            float4 a = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 4
            for (int k = 0; k < K; ++k) {
                const int j = s_j[k];
                if (j < 0) continue;
                const float g = s_g[k];
                const uint4 u = ld_stream16(y + (size_t)j * D + 4 * q);
                float4 v = make_float4(__uint_as_float(u.x), __uint_as_float(u.y),
                                       __uint_as_float(u.z), __uint_as_float(u.w));
                if (y_tail) {  // head + tail of a split down projection, in that order
                    const uint4 w = ld_stream16(y_tail + (size_t)j * D + 4 * q);
                    v.x += __uint_as_float(w.x);
                    v.y += __uint_as_float(w.y);
                    v.z += __uint_as_float(w.z);
                    v.w += __uint_as_float(w.w);
                }
                a.x = fmaf(g, v.x, a.x);
                a.y = fmaf(g, v.y, a.y);
                a.z = fmaf(g, v.z, a.z);
                a.w = fmaf(g, v.w, a.w);
            }
            if (residual) {
                const float4 r = load4(residual + (size_t)t * D + 4 * q);
                a.x += r.x;
                a.y += r.y;
                a.z += r.z;
                a.w += r.w;
            }
            store4(out + (size_t)t * D + 4 * q, a);
        }
    }
}

// ===========================================================================
// Stack glue (reading C9): x_norm[t,:] = bf16( r[t,:] / sqrt(mean(r[t,:]^2) + eps) )
// One block per token; fp32 sum of squares reduced in a fixed order.
// ===========================================================================
template <typename TR, typename TX>
__global__ void __launch_bounds__(256)
k_prenorm(int T, int D, const TR *__restrict__ r, TX *__restrict__ xn, float eps) {
    __shared__ float red[8];
    ptx::grid_dependency_wait();
    for (int t = blockIdx.x; t < T; t += gridDim.x) {
        const TR *row = r + (size_t)t * D;
        float ss = 0.f;
        for (int d = threadIdx.x; d < D; d += 256) {
            const float v = to_f(row[d]);
            ss = fmaf(v, v, ss);
        }
        ss = warp_sum(ss);
        if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = ss;
        __syncthreads();
        float tot = 0.f;
#pragma unroll
        for (int w = 0; w < 8; ++w) tot += red[w];
        const float scale = rsqrtf(tot / (float)D + eps);
        for (int d = threadIdx.x; d < D; d += 256)
            xn[(size_t)t * D + d] = from_f<TX>(to_f(row[d]) * scale);
        __syncthreads();
    }
}

// ===========================================================================
// Busy full loading (Sec. 4.2): every expert takes every token, and the
// experts the router did not select get gate 0 in the weighted sum.
// k_densify turns the top-k routing into that dense form: slot (t, e) of
// the dense layout has expert e and gate g[t,k] if e = idx[t,k], else 0.
// ===========================================================================
__global__ void __launch_bounds__(256)
k_densify(int T, int E, int K, const int32_t *__restrict__ idx, const float *__restrict__ gate,
          int32_t *__restrict__ didx, float *__restrict__ dgate) {
    ptx::grid_dependency_wait();
    const long long total = (long long)T * E;
    for (long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (long long)gridDim.x * blockDim.x) {
        const int t = (int)(i / E), e = (int)(i - (long long)t * E);
        float g = 0.f;
        for (int k = 0; k < K; ++k)
            if (idx[(size_t)t * K + k] == e) g = gate[(size_t)t * K + k];
        didx[i] = e;
        dgate[i] = g;
    }
}

// ===========================================================================
// Self-test of the bounded waits: one thread waits on an mbarrier that
// nothing will complete.  The wait gives up after limit_ns, records
// kErrTimeout and the kernel returns normally.
// ===========================================================================
__global__ void k_wait_timeout_selftest(uint64_t limit_ns, unsigned *err, int *gave_up) {
    __shared__ uint64_t bar;
    ptx::mbar_init(&bar, 1);
    ptx::fence_barrier_init();
    *gave_up = ptx::mbar_wait_limit(&bar, 0, err, limit_ns) ? 0 : 1;
}

// ===========================================================================
// host side
// ===========================================================================

const DeviceInfo &device_info() {
    static DeviceInfo info[64];
    static bool ready[64];
    static std::mutex mu;
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev < 0 || dev >= 64) dev = 0;
    std::lock_guard<std::mutex> g(mu);
    if (!ready[dev]) {
        int sms = 0;
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        void *p = nullptr;
        cudaGetSymbolAddress(&p, g_moe_err);
        info[dev].sm_count = sms > 0 ? sms : 1;
        info[dev].err = static_cast<unsigned *>(p);
        ready[dev] = true;
    }
    return info[dev];
}

namespace {

struct ProfState {
    std::mutex mu;
    bool on = false;
    std::vector<std::string> names;
    std::vector<int64_t> launches;
    std::vector<double> ms;
    struct Pending { int kind; cudaEvent_t a, b; };
    std::vector<Pending> pending;
    std::vector<cudaEvent_t> pool;
    std::vector<cudaEvent_t> begin_of_slot;  // begin event of each open launch
};

ProfState &prof() {
    static ProfState *p = new ProfState();  // never destroyed: used at exit
    return *p;
}

std::atomic<int64_t> g_launches{0};

cudaEvent_t take_event(ProfState &P) {
    if (!P.pool.empty()) {
        cudaEvent_t e = P.pool.back();
        P.pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    cudaEventCreate(&e);
    return e;
}

int kind_of(ProfState &P, const char *name) {
    for (size_t i = 0; i < P.names.size(); ++i)
        if (P.names[i] == name) return (int)i;
    P.names.push_back(name);
    P.launches.push_back(0);
    P.ms.push_back(0.0);
    return (int)P.names.size() - 1;
}

}  // namespace

LaunchScope::LaunchScope(const char *n, cudaStream_t s) : name(n), stream(s), slot(-1) {
    g_launches.fetch_add(1, std::memory_order_relaxed);
    ProfState &P = prof();
    std::lock_guard<std::mutex> g(P.mu);
    if (!P.on) return;
    cudaEvent_t a = take_event(P);
    cudaEventRecord(a, stream);
    P.begin_of_slot.push_back(a);
    slot = (int)P.begin_of_slot.size() - 1;
}

LaunchScope::~LaunchScope() {
    if (slot < 0) return;
    ProfState &P = prof();
    std::lock_guard<std::mutex> g(P.mu);
    cudaEvent_t b = take_event(P);
    cudaEventRecord(b, stream);
    P.pending.push_back({kind_of(P, name), P.begin_of_slot[slot], b});
}

moe_status injected_failure(const char *entry) {
    const char *v = getenv("MOE_INJECT_FAILURE");
    if (!v) return MOE_OK;
    const size_t n = strlen(entry);
    if (strncmp(v, entry, n) != 0 || v[n] != ':') return MOE_OK;
    const int code = atoi(v + n + 1);
    return (code > 0 && code <= MOE_ERR_DEVICE_INDEX) ? (moe_status)code : MOE_OK;
}

WsLayout ws_layout(const moe_dims &d, int64_t T) {
    auto up = [](size_t v) { return (v + 255) & ~size_t(255); };
    const size_t S = (size_t)T * d.top_k;
    WsLayout L{};
    size_t o = 0;
    L.idx = o; o += up(S * 4);
    L.gate = o; o += up(S * 4);
    L.counts = o; o += up((size_t)d.n_experts * 4);
    L.offsets = o; o += up(((size_t)d.n_experts + 1) * 4);
    L.perm = o; o += up(S * 4);
    L.inv_perm = o; o += up(S * 4);
    const bool bf = d.w_dtype == MOE_BF16;
    // GLU hidden vectors: bf16 on the bf16 paths, fp32 on the fp32 path
    L.h = o; o += up(S * d.ffn_hidden * (bf ? 2 : 4));
    // gathered token rows (tensor-core path, bf16 only)
    L.xs = o; o += bf ? up(S * d.d_model * 2) : 0;
    // ungated expert outputs: the tensor-core path, and the fp32 path above
    // the fused-combine limit
    L.y = o; o += (bf || T > kFusedCombineMaxTokens) ? up(S * d.d_model * 4) : 0;
    // the stream-K down projection's tails (bf16 decode batches)
    L.y_tail = o; o += (bf && T <= kStreamKMaxTokens) ? up(S * d.d_model * 4) : 0;
    // work counters of the one-token streaming kernels (zeroed by the
    // routing kernel of the same call)
    L.ctr = o; o += up(4 * sizeof(int));
    L.total = o;
    return L;
}

}  // namespace moe

using namespace moe;

namespace {

bool dt_ok(int32_t v) { return v == MOE_F32 || v == MOE_BF16; }


moe_status check_dims(const moe_dims *d) {
    if (!d) return MOE_ERR_INVALID_ARG;
    if (d->d_model < 8 || d->d_model > 49152 || d->d_model % 8) return MOE_ERR_INVALID_ARG;
    if (d->ffn_hidden < 8 || d->ffn_hidden > 65536 || d->ffn_hidden % 8) return MOE_ERR_INVALID_ARG;
    if (d->n_experts < 1 || d->n_experts > 256) return MOE_ERR_INVALID_ARG;
    if (d->top_k < 1 || d->top_k > d->n_experts) return MOE_ERR_INVALID_ARG;
    if (!dt_ok(d->w_dtype) || !dt_ok(d->x_dtype) || !dt_ok(d->out_dtype)) return MOE_ERR_INVALID_ARG;
    if (d->w_dtype != d->x_dtype) return MOE_ERR_UNSUPPORTED;
    return MOE_OK;
}

moe_status check_T(const moe_dims *d, int32_t T) {
    if (T < 0 || T > (1 << 20)) return MOE_ERR_INVALID_ARG;
    if ((int64_t)T * d->top_k > (1 << 24)) return MOE_ERR_INVALID_ARG;
    return MOE_OK;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
bool ok_ptr(const void *p) { return p != nullptr && aligned16(p); }
bool ok_opt(const void *p) { return p == nullptr || aligned16(p); }

moe_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MOE_OK : MOE_ERR_CUDA; }

size_t router_bytes(const moe_dims &d) {
    return (size_t)d.d_model * d.n_experts * (d.w_dtype == MOE_BF16 ? 2 : 4);
}

template <typename TX, typename TW>
cudaError_t launch_route(const moe_dims &d, int T, const void *x, const void *wr, float *logits,
                         int32_t *idx, float *gate, cudaStream_t st) {
    const int grid = (T + kRouteTokens - 1) / kRouteTokens;
    LaunchScope ls("route", st);
    k_route<TX, TW><<<grid, kRouteThreads, 0, st>>>(T, d.d_model, d.n_experts, d.top_k,
                                                   static_cast<const TX *>(x),
                                                   static_cast<const TW *>(wr), logits, idx, gate);
    return cudaGetLastError();
}

template <typename TX, typename TW>
cudaError_t launch_route_dispatch_small(const moe_dims &d, int T, const void *x, const void *wr,
                                        int32_t *idx, float *gate, int32_t *counts,
                                        int32_t *offsets, int32_t *perm, int32_t *inv,
                                        cudaStream_t st, int *ctr) {
    int Tv = T, D = d.d_model, E = d.n_experts, K = d.top_k;
    const TX *xp = static_cast<const TX *>(x);
    const TW *wp = static_cast<const TW *>(wr);
    float *logits = nullptr;
    unsigned *err = device_info().err;
    const size_t wrb = router_bytes(d);
    int staged = wrb <= kStagedRouterMax ? 1 : 0;
    const void *kern = (const void *)k_route_dispatch_small<TX, TW>;
    if (staged) {
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kStagedRouterMax);
        if (e != cudaSuccess) return e;
    }
    void *args[] = {&Tv, &D, &E, &K, &xp, &wp, &logits, &idx, &gate, &counts, &offsets, &perm, &inv,
                    &staged, &ctr, &err};
    LaunchScope ls("route_dispatch_small", st);
    return launch_pdl(kern, dim3(1), dim3(kStagedThreads), staged ? wrb : 0, st, args);
}

// Dynamic shared memory of the cluster kernel: the partial logits, one CTA's
// slice of the router and the same slice of every token row.
size_t cluster_smem_bytes(const moe_dims &d, int T) {
    const int wb = d.w_dtype == MOE_BF16 ? 2 : 4, xb = d.x_dtype == MOE_BF16 ? 2 : 4;
    return cluster_part_bytes(T, d.n_experts) +
           (size_t)cluster_rows(d.d_model) * d.n_experts * wb +
           (size_t)T * cluster_x_stride(d.d_model, xb);
}

template <typename TX, typename TW>
cudaError_t launch_route_dispatch_cluster(const moe_dims &d, int T, const void *x,
                                          const void *wr, int32_t *idx, float *gate,
                                          int32_t *counts, int32_t *offsets, int32_t *perm,
                                          int32_t *inv, cudaStream_t st) {
    int Tv = T, D = d.d_model, E = d.n_experts, K = d.top_k;
    const TX *xp = static_cast<const TX *>(x);
    const TW *wp = static_cast<const TW *>(wr);
    unsigned *err = device_info().err;
    const size_t smem = cluster_smem_bytes(d, T);
    const void *kern = (const void *)k_route_dispatch_cluster<TX, TW>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    void *args[] = {&Tv, &D, &E, &K, &xp, &wp, &idx, &gate, &counts, &offsets, &perm, &inv, &err};
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(kClusterCtas);
    cfg.blockDim = dim3(kClusterThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = kClusterCtas;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    LaunchScope ls("route_dispatch_cluster", st);
    return cudaLaunchKernelExC(&cfg, kern, args);
}

bool cluster_route_ok(const moe_dims &d, int T) {
    if (T < 1 || T > kClusterMaxTokens || T * d.top_k > kClusterMaxSlots) return false;
    return cluster_smem_bytes(d, T) <= kClusterMaxSmem;
}

cudaError_t route_dispatch_cluster_any(const moe_dims &d, int T, const void *x, const void *wr,
                                       int32_t *idx, float *gate, int32_t *counts,
                                       int32_t *offsets, int32_t *perm, int32_t *inv,
                                       cudaStream_t st) {
    if (d.w_dtype == MOE_BF16)
        return launch_route_dispatch_cluster<bf16, bf16>(d, T, x, wr, idx, gate, counts, offsets,
                                                         perm, inv, st);
    return launch_route_dispatch_cluster<float, float>(d, T, x, wr, idx, gate, counts, offsets,
                                                       perm, inv, st);
}

bool small_route_ok(const moe_dims &d, int T) {
    return T <= kRouteTokens && T * d.top_k <= kSmallMaxSlots;
}

cudaError_t route_dispatch_small_any(const moe_dims &d, int T, const void *x, const void *wr,
                                     int32_t *idx, float *gate, int32_t *counts, int32_t *offsets,
                                     int32_t *perm, int32_t *inv, cudaStream_t st,
                                     int *ctr = nullptr) {
    if (d.w_dtype == MOE_BF16)
        return launch_route_dispatch_small<bf16, bf16>(d, T, x, wr, idx, gate, counts, offsets,
                                                       perm, inv, st, ctr);
    return launch_route_dispatch_small<float, float>(d, T, x, wr, idx, gate, counts, offsets, perm,
                                                     inv, st, ctr);
}

// scratch (optional, scratch_bytes): room for the tensor-core router's
// partial logits; without it (moe_route) the CUDA-core kernel routes.
cudaError_t route_any(const moe_dims &d, int T, const void *x, const void *wr, float *logits,
                      int32_t *idx, float *gate, cudaStream_t st, void *scratch = nullptr,
                      size_t scratch_bytes = 0) {
    if (scratch && route_tc_ok(d, T) && aligned16(scratch) &&
        scratch_bytes >= route_tc_scratch_bytes(d, T))
        return launch_route_tc(d, T, x, wr, logits, idx, gate, static_cast<float *>(scratch), st);
    if (d.w_dtype == MOE_BF16) return launch_route<bf16, bf16>(d, T, x, wr, logits, idx, gate, st);
    return launch_route<float, float>(d, T, x, wr, logits, idx, gate, st);
}

cudaError_t dispatch_any(const moe_dims &d, int T, const int32_t *idx, int32_t *counts,
                         int32_t *offsets, int32_t *perm, int32_t *inv, cudaStream_t st) {
    const long long S = (long long)T * d.top_k;
    const long long C = (S + kDispatchThreads - 1) / kDispatchThreads;
    const size_t wh_bytes = (size_t)C * (kDispatchThreads / 32) * d.n_experts * sizeof(int);
    if (C >= 1 && C <= kFastMaxChunks && wh_bytes <= kFastDispatchSmem) {
        cudaError_t e = cudaFuncSetAttribute((const void *)k_dispatch_fast,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kFastDispatchSmem);
        if (e != cudaSuccess) return e;
        int Sv = (int)S, E = d.n_experts;
        unsigned *err = device_info().err;
        void *args[] = {&Sv, &E, &idx, &counts, &offsets, &perm, &inv, &err};
        LaunchScope ls("dispatch", st);
        return launch_pdl((const void *)k_dispatch_fast, dim3(1), dim3(kDispatchThreads), wh_bytes,
                          st, args);
    }
    LaunchScope ls("dispatch", st);
    k_dispatch<<<1, kDispatchThreads, 0, st>>>(T * d.top_k, d.n_experts, idx, counts, offsets,
                                               perm, inv, device_info().err);
    return cudaGetLastError();
}

template <typename TO, typename TR>
cudaError_t launch_combine(const moe_dims &d, int T, const float *y, const float *y_tail,
                           const int32_t *inv, const float *gate, const void *res, void *out,
                           cudaStream_t st, const int32_t *range, int n_range) {
    // enough blocks for 8 per SM: a token's row is split into n_part slices
    // of at least 256 float4 when there are few tokens
    const int nq = d.d_model / 4;
    const long long cap = (long long)device_info().sm_count * 8;
    int n_part = (int)std::max(1LL, std::min<long long>((cap + T - 1) / T, (nq + 255) / 256));
    const int grid = (int)std::max(1LL, std::min((long long)T * n_part, cap));
    int Tv = T, D = d.d_model, K = d.top_k;
    const TR *rp = static_cast<const TR *>(res);
    TO *op = static_cast<TO *>(out);
    unsigned *err = device_info().err;
    void *args[] = {&Tv, &D, &K, &n_part, &y, &y_tail, &inv, &gate, &rp, &op, &range, &n_range,
                    &err};
    LaunchScope ls("combine", st);
    return launch_pdl((const void *)k_combine<TO, TR>, dim3(grid), dim3(256), 0, st, args);
}

cudaError_t combine_any(const moe_dims &d, int T, const float *y, const int32_t *inv,
                        const float *gate, const void *res, void *out, cudaStream_t st,
                        const float *y_tail = nullptr, const int32_t *range = nullptr,
                        int n_range = 0) {
    // the residual has the output's dtype
    if (d.out_dtype == MOE_BF16)
        return launch_combine<bf16, bf16>(d, T, y, y_tail, inv, gate, res, out, st, range,
                                          n_range);
    return launch_combine<float, float>(d, T, y, y_tail, inv, gate, res, out, st, range,
                                        n_range);
}

bool use_stream_path(const moe_dims &d, int T) {
    return T <= kStreamMaxTokens && stream_path_ok(d, T);
}

cudaError_t prenorm_any(const moe_dims &d, int T, const void *r, void *xn, float eps,
                        cudaStream_t st) {
    const int grid = std::max(1, std::min(T, device_info().sm_count * 8));
    int Tv = T, D = d.d_model;
    void *args[] = {&Tv, &D, const_cast<void **>(&r), &xn, &eps};
    const void *kern;
    if (d.out_dtype == MOE_F32)
        kern = d.x_dtype == MOE_BF16 ? (const void *)k_prenorm<float, bf16>
                                     : (const void *)k_prenorm<float, float>;
    else
        kern = d.x_dtype == MOE_BF16 ? (const void *)k_prenorm<bf16, bf16>
                                     : (const void *)k_prenorm<bf16, float>;
    LaunchScope ls("prenorm", st);
    return launch_pdl(kern, dim3(grid), dim3(256), 0, st, args);
}

template <typename P> P *at(void *ws, size_t off) {
    return reinterpret_cast<P *>(static_cast<char *>(ws) + off);
}

// The one-token streaming kernels' work counters, when the routing of the
// same call zeroes them (route_dispatch_ws on its one-token path), else null
// (equal static shares).
int *stream_ctr(const moe_dims &d, int T, const WsLayout &L, void *ws) {
    return T == 1 && small_route_ok(d, T) ? at<int>(ws, L.ctr) : nullptr;
}

// Routing and dispatch of the whole layer into the workspace regions of L:
// the fused one-CTA or one-cluster kernels for decode batches, else the
// router (on the tensor cores for large batches, with the GLU hidden
// vectors' region, free until the up projection, as its scratch) and the
// dispatch kernel.
cudaError_t route_dispatch_ws(const moe_dims &d, int T, const void *x, const void *w_router,
                              const WsLayout &L, void *ws, cudaStream_t st) {
    int32_t *idx = at<int32_t>(ws, L.idx);
    float *gate = at<float>(ws, L.gate);
    int32_t *counts = at<int32_t>(ws, L.counts);
    int32_t *offsets = at<int32_t>(ws, L.offsets);
    int32_t *perm = at<int32_t>(ws, L.perm);
    int32_t *inv = at<int32_t>(ws, L.inv_perm);
    if (T == 1 && small_route_ok(d, T))
        return route_dispatch_small_any(d, T, x, w_router, idx, gate, counts, offsets, perm, inv,
                                        st, stream_ctr(d, T, L, ws));
    if (cluster_route_ok(d, T))
        return route_dispatch_cluster_any(d, T, x, w_router, idx, gate, counts, offsets, perm,
                                          inv, st);
    if (small_route_ok(d, T))
        return route_dispatch_small_any(d, T, x, w_router, idx, gate, counts, offsets, perm, inv,
                                        st);
    cudaError_t e = route_any(d, T, x, w_router, nullptr, idx, gate, st, at<float>(ws, L.h),
                              L.xs > L.h ? L.xs - L.h : 0);
    if (e == cudaSuccess) e = dispatch_any(d, T, idx, counts, offsets, perm, inv, st);
    return e;
}

}  // namespace

extern "C" {

moe_status moe_workspace_size(const moe_dims *dims, int32_t max_tokens, size_t *bytes) {
    moe_status s = check_dims(dims);
    if (s == MOE_ERR_UNSUPPORTED) s = MOE_OK;  // sizing does not depend on dtypes
    if (s != MOE_OK) return s;
    if (!bytes || max_tokens < 0) return MOE_ERR_INVALID_ARG;
    if ((s = check_T(dims, max_tokens)) != MOE_OK) return s;
    *bytes = ws_layout(*dims, max_tokens).total;
    return MOE_OK;
}

moe_status moe_route(const moe_dims *dims, int32_t T, const void *x, const void *w_router,
                     float *logits_opt, int32_t *topk_idx, float *topk_gate, moe_stream_t stream) {
    MOE_INJECT("moe_route");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(x) || !ok_ptr(w_router) || !ok_opt(logits_opt) || !topk_idx || !topk_gate)
        return MOE_ERR_INVALID_ARG;
    return cuda_status(route_any(*dims, T, x, w_router, logits_opt, topk_idx, topk_gate,
                                 (cudaStream_t)stream));
}

moe_status moe_dispatch(const moe_dims *dims, int32_t T, const int32_t *topk_idx,
                        int32_t *counts, int32_t *offsets, int32_t *perm, int32_t *inv_perm,
                        moe_stream_t stream) {
    MOE_INJECT("moe_dispatch");
    moe_status s = check_dims(dims);
    if (s == MOE_ERR_UNSUPPORTED) s = MOE_OK;  // dispatch does not read floating point data
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (!counts || !offsets) return MOE_ERR_INVALID_ARG;
    if (T > 0 && (!topk_idx || !perm || !inv_perm)) return MOE_ERR_INVALID_ARG;
    return cuda_status(dispatch_any(*dims, T, topk_idx, counts, offsets, perm, inv_perm,
                                    (cudaStream_t)stream));
}

moe_status moe_expert_ffn(const moe_dims *dims, int32_t T, const void *x, const int32_t *perm,
                          const int32_t *offsets, const void *w1, const void *v1, const void *w2,
                          float *y_sorted, void *ws, size_t ws_bytes, moe_stream_t stream) {
    MOE_INJECT("moe_expert_ffn");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(x) || !perm || !offsets || !ok_ptr(w1) || !ok_ptr(v1) || !ok_ptr(w2) ||
        !ok_ptr(y_sorted))
        return MOE_ERR_INVALID_ARG;
    const WsLayout L = ws_layout(*dims, T);
    if (!ws || !aligned16(ws) || ws_bytes < L.total) return MOE_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    float *h = at<float>(ws, L.h);
    cudaError_t e;
    if (use_stream_path(*dims, T)) {
        // bf16 weights, few slots: bulk-copy pipelined kernels, bf16 h
        e = launch_up_glu_stream(*dims, T, x, perm, offsets, w1, v1, h, st);
        if (e == cudaSuccess)
            e = launch_down_stream(*dims, T, h, offsets, nullptr, w2, nullptr, nullptr, nullptr,
                                   y_sorted, false, st);
        return cuda_status(e);
    }
    if (tc_path_ok(*dims)) {
        // bf16 weights: gather the token rows, then the two tcgen05 GEMMs
        void *xs = at<void>(ws, L.xs);
        e = launch_gather_rows(*dims, T, x, perm, xs, st);
        if (e == cudaSuccess) e = launch_gemm_up_tc(*dims, T, xs, offsets, w1, v1, h, st);
        if (e == cudaSuccess) e = launch_gemm_down_tc(*dims, T, h, offsets, w2, y_sorted, st);
        return cuda_status(e);
    }
    e = launch_up_glu_gemv(*dims, T, x, perm, offsets, w1, v1, h, st);
    if (e == cudaSuccess)
        e = launch_down_gemv(*dims, T, h, perm, offsets, w2, nullptr, y_sorted, nullptr, nullptr,
                             false, st);
    return cuda_status(e);
}

moe_status moe_combine(const moe_dims *dims, int32_t T, const float *y_sorted,
                       const int32_t *inv_perm, const float *topk_gate, const void *residual_opt,
                       void *out, moe_stream_t stream) {
    MOE_INJECT("moe_combine");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(y_sorted) || !inv_perm || !topk_gate || !ok_opt(residual_opt) || !ok_ptr(out))
        return MOE_ERR_INVALID_ARG;
    return cuda_status(combine_any(*dims, T, y_sorted, inv_perm, topk_gate, residual_opt, out,
                                   (cudaStream_t)stream));
}

moe_status moe_layer_forward(const moe_dims *dims, int32_t T, const void *x, const void *w_router,
                             const void *w1, const void *v1, const void *w2,
                             const void *residual_opt, void *out, void *ws, size_t ws_bytes,
                             moe_stream_t stream) {
    MOE_INJECT("moe_layer_forward");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(x) || !ok_ptr(w_router) || !ok_ptr(w1) || !ok_ptr(v1) || !ok_ptr(w2) ||
        !ok_opt(residual_opt) || !ok_ptr(out))
        return MOE_ERR_INVALID_ARG;
    const WsLayout L = ws_layout(*dims, T);
    if (!ws || !aligned16(ws) || ws_bytes < L.total) return MOE_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    const moe_dims &d = *dims;
    float *gate = at<float>(ws, L.gate);
    int32_t *offsets = at<int32_t>(ws, L.offsets);
    int32_t *perm = at<int32_t>(ws, L.perm);
    int32_t *inv = at<int32_t>(ws, L.inv_perm);
    float *h = at<float>(ws, L.h);

    cudaError_t e = route_dispatch_ws(d, T, x, w_router, L, ws, st);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    if (use_stream_path(d, T)) {
        // decode, bf16: bulk-copy pipelined kernels, combine fused into the
        // down projection
        e = launch_up_glu_stream(d, T, x, perm, offsets, w1, v1, h, st, stream_ctr(d, T, L, ws));
        if (e == cudaSuccess)
            e = launch_down_stream(d, T, h, offsets, inv, w2, gate, residual_opt, out, nullptr,
                                   true, st);
        return cuda_status(e);
    }
    if (tc_path_ok(d)) {
        // bf16: gathered token rows, tcgen05 GEMMs (GLU fused into the up
        // projection's epilogue), then the gated combine
        void *xs = at<void>(ws, L.xs);
        float *y = at<float>(ws, L.y);
        e = launch_gather_rows(d, T, x, perm, xs, st);
        if (e == cudaSuccess) e = launch_gemm_up_tc(d, T, xs, offsets, w1, v1, h, st);
        // decode batches: the stream-K down projection keeps every SM busy
        // when the selected experts give few weight tiles
        float *y_tail = T <= kStreamKMaxTokens ? at<float>(ws, L.y_tail) : nullptr;
        if (e == cudaSuccess) e = launch_gemm_down_tc(d, T, h, offsets, w2, y, st, nullptr, y_tail);
        if (e == cudaSuccess) e = combine_any(d, T, y, inv, gate, residual_opt, out, st, y_tail);
        return cuda_status(e);
    }
    e = launch_up_glu_gemv(d, T, x, perm, offsets, w1, v1, h, st);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    if (T <= kFusedCombineMaxTokens) {
        e = launch_down_gemv(d, T, h, perm, offsets, w2, gate, nullptr, residual_opt, out, true, st);
    } else {
        float *y = at<float>(ws, L.y);
        e = launch_down_gemv(d, T, h, perm, offsets, w2, nullptr, y, nullptr, nullptr, false, st);
        if (e == cudaSuccess) e = combine_any(d, T, y, inv, gate, residual_opt, out, st);
    }
    return cuda_status(e);
}

moe_status moe_layer_forward_experts(const moe_dims *dims, int32_t T, const void *x,
                                     const void *w_router, int32_t e_begin, int32_t e_end,
                                     const void *w1_local, const void *v1_local,
                                     const void *w2_local, const float *residual_opt,
                                     float *partial_out, void *ws, size_t ws_bytes,
                                     moe_stream_t stream) {
    MOE_INJECT("moe_layer_forward_experts");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (e_begin < 0 || e_end > dims->n_experts || e_begin >= e_end) return MOE_ERR_INVALID_ARG;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(x) || !ok_ptr(w_router) || !ok_ptr(w1_local) || !ok_ptr(v1_local) ||
        !ok_ptr(w2_local) || !ok_opt(residual_opt) || !ok_ptr(partial_out))
        return MOE_ERR_INVALID_ARG;
    const WsLayout L = ws_layout(*dims, T);
    if (!ws || !aligned16(ws) || ws_bytes < L.total) return MOE_ERR_WORKSPACE;
    cudaStream_t st = (cudaStream_t)stream;
    const moe_dims &d = *dims;
    float *gate = at<float>(ws, L.gate);
    int32_t *offsets = at<int32_t>(ws, L.offsets);
    int32_t *perm = at<int32_t>(ws, L.perm);
    int32_t *inv = at<int32_t>(ws, L.inv_perm);
    float *h = at<float>(ws, L.h);

    // every node routes and dispatches over all E experts (the replicated
    // router of Sec. 4.3) ...
    cudaError_t e = route_dispatch_ws(d, T, x, w_router, L, ws, st);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    // ... and runs the expert kernels over its own experts only: their
    // dispatch offsets start at offsets[e_begin] and address the same sorted
    // slot arrays, and the weights hold experts e_begin..e_end-1
    moe_dims dl = d;
    dl.n_experts = e_end - e_begin;
    dl.out_dtype = MOE_F32;
    const int32_t *loff = offsets + e_begin;
    if (use_stream_path(d, T)) {
        e = launch_up_glu_stream(dl, T, x, perm, loff, w1_local, v1_local, h, st,
                                 stream_ctr(d, T, L, ws));
        if (e == cudaSuccess)
            e = launch_down_stream(dl, T, h, loff, inv, w2_local, gate, residual_opt, partial_out,
                                   nullptr, true, st);
        return cuda_status(e);
    }
    if (tc_path_ok(d)) {
        void *xs = at<void>(ws, L.xs);
        float *y = at<float>(ws, L.y);
        float *y_tail = T <= kStreamKMaxTokens ? at<float>(ws, L.y_tail) : nullptr;
        e = launch_gather_rows(d, T, x, perm, xs, st, loff, dl.n_experts);
        if (e == cudaSuccess) e = launch_gemm_up_tc(dl, T, xs, loff, w1_local, v1_local, h, st);
        if (e == cudaSuccess)
            e = launch_gemm_down_tc(dl, T, h, loff, w2_local, y, st, nullptr, y_tail);
        if (e == cudaSuccess)
            e = combine_any(dl, T, y, inv, gate, residual_opt, partial_out, st, y_tail, loff,
                            dl.n_experts);
        return cuda_status(e);
    }
    e = launch_up_glu_gemv(dl, T, x, perm, loff, w1_local, v1_local, h, st);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    if (T <= kFusedCombineMaxTokens) {
        // the fused down projection sums over the experts it is given
        e = launch_down_gemv(dl, T, h, perm, loff, w2_local, gate, nullptr, residual_opt,
                             partial_out, true, st);
    } else {
        float *y = at<float>(ws, L.y);
        e = launch_down_gemv(dl, T, h, perm, loff, w2_local, nullptr, y, nullptr, nullptr, false,
                             st);
        if (e == cudaSuccess)
            e = combine_any(dl, T, y, inv, gate, residual_opt, partial_out, st, nullptr, loff,
                            dl.n_experts);
    }
    return cuda_status(e);
}

moe_status moe_prenorm(const moe_dims *dims, int32_t T, const void *resid, void *x_norm,
                       float eps, moe_stream_t stream) {
    MOE_INJECT("moe_prenorm");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(resid) || !ok_ptr(x_norm) || !(eps > 0.f)) return MOE_ERR_INVALID_ARG;
    return cuda_status(prenorm_any(*dims, T, resid, x_norm, eps, (cudaStream_t)stream));
}

moe_status moe_stack_workspace_size(const moe_dims *dims, int32_t max_tokens, size_t *bytes) {
    size_t layer = 0;
    moe_status s = moe_workspace_size(dims, max_tokens, &layer);
    if (s != MOE_OK) return s;
    const size_t xn = ((size_t)max_tokens * dims->d_model * (dims->x_dtype == MOE_BF16 ? 2 : 4) +
                       255) & ~size_t(255);
    *bytes = xn + layer;
    return MOE_OK;
}

moe_status moe_stack_forward(const moe_dims *dims, int32_t n_layers, int32_t T,
                             const void *const *w_router, const void *const *w1,
                             const void *const *v1, const void *const *w2, void *resid, float eps,
                             void *ws, size_t ws_bytes, moe_stream_t stream) {
    MOE_INJECT("moe_stack_forward");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    if ((s = check_T(dims, T)) != MOE_OK) return s;
    if (n_layers < 0) return MOE_ERR_INVALID_ARG;
    if (T == 0 || n_layers == 0) return MOE_OK;
    if (!w_router || !w1 || !v1 || !w2 || !ok_ptr(resid) || !(eps > 0.f))
        return MOE_ERR_INVALID_ARG;
    for (int l = 0; l < n_layers; ++l)
        if (!ok_ptr(w_router[l]) || !ok_ptr(w1[l]) || !ok_ptr(v1[l]) || !ok_ptr(w2[l]))
            return MOE_ERR_INVALID_ARG;
    size_t need = 0;
    if ((s = moe_stack_workspace_size(dims, T, &need)) != MOE_OK) return s;
    if (!ws || !aligned16(ws) || ws_bytes < need) return MOE_ERR_WORKSPACE;
    const size_t xn_bytes = need - ws_layout(*dims, T).total;
    void *xn = ws;
    void *lws = static_cast<char *>(ws) + xn_bytes;
    for (int l = 0; l < n_layers; ++l) {
        if (prenorm_any(*dims, T, resid, xn, eps, (cudaStream_t)stream) != cudaSuccess)
            return MOE_ERR_CUDA;
        // resid <- resid + MoE_l(x_norm): the combine reads each residual
        // element before it writes the same element
        s = moe_layer_forward(dims, T, xn, w_router[l], w1[l], v1[l], w2[l], resid, resid, lws,
                              ws_bytes - xn_bytes, stream);
        if (s != MOE_OK) return s;
    }
    return MOE_OK;
}

// Dense (busy-full-loading) layout: the layer's own workspace for top_k = E,
// followed by the sparse routing [T, K] (indices and gates).
moe_status moe_dense_workspace_size(const moe_dims *dims, int32_t max_tokens, size_t *bytes) {
    moe_status s = check_dims(dims);
    if (s == MOE_ERR_UNSUPPORTED) s = MOE_OK;
    if (s != MOE_OK) return s;
    if (!bytes || max_tokens < 0) return MOE_ERR_INVALID_ARG;
    moe_dims dd = *dims;
    dd.top_k = dims->n_experts;
    if ((s = check_T(&dd, max_tokens)) != MOE_OK) return s;
    const size_t sparse = (((size_t)max_tokens * dims->top_k * 8) + 255) & ~size_t(255);
    *bytes = ws_layout(dd, max_tokens).total + sparse;
    return MOE_OK;
}

moe_status moe_layer_forward_dense(const moe_dims *dims, int32_t T, const void *x,
                                   const void *w_router, const void *w1, const void *v1,
                                   const void *w2, const void *residual_opt, void *out, void *ws,
                                   size_t ws_bytes, moe_stream_t stream) {
    MOE_INJECT("moe_layer_forward_dense");
    moe_status s = check_dims(dims);
    if (s != MOE_OK) return s;
    moe_dims dd = *dims;
    dd.top_k = dims->n_experts;  // every expert takes every token
    if ((s = check_T(&dd, T)) != MOE_OK) return s;
    if (T == 0) return MOE_OK;
    if (!ok_ptr(x) || !ok_ptr(w_router) || !ok_ptr(w1) || !ok_ptr(v1) || !ok_ptr(w2) ||
        !ok_opt(residual_opt) || !ok_ptr(out))
        return MOE_ERR_INVALID_ARG;
    if (!tc_path_ok(*dims)) return MOE_ERR_UNSUPPORTED;
    size_t need = 0;
    if ((s = moe_dense_workspace_size(dims, T, &need)) != MOE_OK) return s;
    if (!ws || !aligned16(ws) || ws_bytes < need) return MOE_ERR_WORKSPACE;
    const WsLayout L = ws_layout(dd, T);
    cudaStream_t st = (cudaStream_t)stream;
    int32_t *sidx = at<int32_t>(ws, L.total);
    float *sgate = at<float>(ws, L.total + (size_t)T * dims->top_k * 4);
    int32_t *didx = at<int32_t>(ws, L.idx);
    float *dgate = at<float>(ws, L.gate);
    int32_t *counts = at<int32_t>(ws, L.counts);
    int32_t *offsets = at<int32_t>(ws, L.offsets);
    int32_t *perm = at<int32_t>(ws, L.perm);
    int32_t *inv = at<int32_t>(ws, L.inv_perm);
    void *h = at<void>(ws, L.h);
    void *xs = at<void>(ws, L.xs);
    float *y = at<float>(ws, L.y);

    cudaError_t e = route_any(*dims, T, x, w_router, nullptr, sidx, sgate, st);
    if (e == cudaSuccess) {
        const long long total = (long long)T * dd.n_experts;
        const int grid = (int)std::max(1LL, std::min((total + 255) / 256,
                                                     (long long)device_info().sm_count * 8));
        int Tv = T, E = dd.n_experts, K = dims->top_k;
        void *args[] = {&Tv, &E, &K, &sidx, &sgate, &didx, &dgate};
        LaunchScope ls("densify", st);
        e = launch_pdl((const void *)k_densify, dim3(grid), dim3(256), 0, st, args);
    }
    if (e == cudaSuccess) e = dispatch_any(dd, T, didx, counts, offsets, perm, inv, st);
    if (e == cudaSuccess) e = launch_gather_rows(dd, T, x, perm, xs, st);
    if (e == cudaSuccess) e = launch_gemm_up_tc(dd, T, xs, offsets, w1, v1, h, st);
    if (e == cudaSuccess) e = launch_gemm_down_tc(dd, T, h, offsets, w2, y, st);
    if (e == cudaSuccess) e = combine_any(dd, T, y, inv, dgate, residual_opt, out, st);
    return cuda_status(e);
}

const char *moe_status_string(moe_status status) {
    switch (status) {
    case MOE_OK: return "MOE_OK";
    case MOE_ERR_INVALID_ARG: return "MOE_ERR_INVALID_ARG: invalid argument";
    case MOE_ERR_UNSUPPORTED: return "MOE_ERR_UNSUPPORTED: unsupported dtype combination";
    case MOE_ERR_WORKSPACE: return "MOE_ERR_WORKSPACE: workspace missing or too small";
    case MOE_ERR_CUDA: return "MOE_ERR_CUDA: CUDA launch or runtime error";
    case MOE_ERR_TIMEOUT: return "MOE_ERR_TIMEOUT: a bounded device wait gave up";
    case MOE_ERR_DEVICE_INDEX: return "MOE_ERR_DEVICE_INDEX: expert index out of range";
    }
    return "unknown moe_status";
}

moe_status moe_get_last_error(moe_stream_t stream) {
    cudaError_t e = cudaStreamSynchronize((cudaStream_t)stream);
    if (e != cudaSuccess) return MOE_ERR_CUDA;
    if (cudaGetLastError() != cudaSuccess) return MOE_ERR_CUDA;
    unsigned v = 0;
    if (cudaMemcpyFromSymbol(&v, g_moe_err, sizeof v) != cudaSuccess) return MOE_ERR_CUDA;
    if (v != kErrNone) {
        const unsigned zero = 0;
        if (cudaMemcpyToSymbol(g_moe_err, &zero, sizeof zero) != cudaSuccess) return MOE_ERR_CUDA;
    }
    if (v == kErrIndex) return MOE_ERR_DEVICE_INDEX;
    if (v == kErrTimeout) return MOE_ERR_TIMEOUT;
    return MOE_OK;
}

moe_status moe_selftest_wait_timeout(uint64_t limit_ns, int32_t *gave_up, moe_stream_t stream) {
    if (!gave_up || limit_ns == 0 || limit_ns > 10000000000ull) return MOE_ERR_INVALID_ARG;
    LaunchScope ls("selftest_wait_timeout", (cudaStream_t)stream);
    k_wait_timeout_selftest<<<1, 1, 0, (cudaStream_t)stream>>>(limit_ns, device_info().err,
                                                              gave_up);
    return cuda_status(cudaGetLastError());
}

int64_t moe_launch_count(void) { return g_launches.load(); }

void moe_profile_enable(int on) {
    ProfState &P = prof();
    std::lock_guard<std::mutex> g(P.mu);
    P.on = on != 0;
}

void moe_profile_reset(void) {
    ProfState &P = prof();
    std::lock_guard<std::mutex> g(P.mu);
    for (auto &p : P.pending) {
        cudaEventSynchronize(p.b);
        P.pool.push_back(p.a);
        P.pool.push_back(p.b);
    }
    P.pending.clear();
    P.begin_of_slot.clear();
    for (auto &v : P.launches) v = 0;
    for (auto &v : P.ms) v = 0.0;
}

int32_t moe_profile_read(moe_kernel_stat *stats, int32_t max_stats) {
    ProfState &P = prof();
    std::lock_guard<std::mutex> g(P.mu);
    for (auto &p : P.pending) {
        cudaEventSynchronize(p.b);
        float ms = 0.f;
        if (cudaEventElapsedTime(&ms, p.a, p.b) == cudaSuccess) P.ms[p.kind] += ms;
        P.launches[p.kind] += 1;
        P.pool.push_back(p.a);
        P.pool.push_back(p.b);
    }
    P.pending.clear();
    P.begin_of_slot.clear();
    const int n = (int)P.names.size();
    for (int i = 0; i < n && i < max_stats; ++i) {
        memset(stats[i].name, 0, sizeof stats[i].name);
        strncpy(stats[i].name, P.names[i].c_str(), sizeof stats[i].name - 1);
        stats[i].launches = P.launches[i];
        stats[i].total_ms = P.ms[i];
    }
    return n;
}

}  // extern "C"
