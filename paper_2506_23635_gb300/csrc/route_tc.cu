// Router of a large batch on the tensor cores (step a1 of the layer: Sec. 3.1
// of arxiv 2506.23635 feeds every token's router output to the expert
// selection): logits[t, e] = sum_d x[t, d] W_r[d, e] as a [T x D] . [D x E]
// product with E <= 16, then the softmax, top-K and renormalised gates.
//
// k_route_tc: CTA (m, s) takes the 128 tokens of tile m against the s-th of
//   `ksplit` equal shares of the 64-column blocks of d.  Its slice of W_r is
//   written by the threads, transposed, into shared memory in the 128-byte
//   swizzled K-major layout (16 expert rows per 64-column panel) -- before
//   the dependency wait, as W_r comes from no earlier kernel; the token rows
//   arrive by TMA in a 4-stage ring; one lane issues tcgen05.mma
//   (M = 128 tokens, N = 16 experts, K = 16) into a 128 x 16 fp32
//   accumulator in tensor memory; the four warps read their 32 tokens' rows
//   and write the partial logits part[s][t][0..16).
// k_route_topk: one warp per token adds the shares' partial logits in share
//   order and runs select_topk (ties to the lower index, NaN ranked as -inf);
//   one thread per token was slower (12.5 vs 10.6 us at 2048 tokens).
// At 2048 tokens the two take 16.6 + 10.6 us where the CUDA-core kernel
// (k_route, which re-reads W_r from L2 for every 4 tokens) took 65 us.
#include <cuda.h>
#include <cudaTypedefs.h>

#include "tc.cuh"

namespace moe {
namespace {

using namespace tc;

constexpr int kRtThreads = 128;
constexpr int kRtM = 128;                                 // tokens per tile
constexpr int kRtBK = 64;                                 // d per k-block (one 128 B row)
constexpr int kRtStages = 4;
constexpr uint32_t kRtStageBytes = kRtM * kRtBK * 2;      // 16 KB of token rows
constexpr int kRtMaxKb = 16;                              // k-blocks per share at most
constexpr uint32_t kRtPanelBytes = 16 * kRtBK * 2;        // 16 expert rows x 128 B
constexpr size_t kRtSmem = 1024 + kRtStages * kRtStageBytes + kRtMaxKb * kRtPanelBytes + 256;
// kind::f16: bf16 A and B, fp32 D, both K-major, N = 16, M = 128
constexpr uint32_t kRtIdesc =
    (1u << 4) | (1u << 7) | (1u << 10) | ((16u >> 3) << 17) | ((uint32_t)(kRtM >> 4) << 24);

struct RtHeader {
    uint64_t full[kRtStages];
    uint64_t empty[kRtStages];
    uint64_t done;
    uint32_t tmem;
};

__global__ void __launch_bounds__(kRtThreads, 1)
k_route_tc(const __grid_constant__ CUtensorMap tmX, int T, int D, int E, int nkb_total, int ksplit,
           const bf16 *__restrict__ wr, float *__restrict__ part, unsigned *err) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    unsigned char *wt = smem + kRtStages * kRtStageBytes;  // W_r^T slice, kRtMaxKb panels
    RtHeader *hd = reinterpret_cast<RtHeader *>(wt + kRtMaxKb * kRtPanelBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int m0 = blockIdx.x * kRtM, sh = blockIdx.y;
    const int kb0 = (int)((long long)nkb_total * sh / ksplit);
    const int nkb = (int)((long long)nkb_total * (sh + 1) / ksplit) - kb0;  // <= kRtMaxKb (host)

    if (threadIdx.x == 0) {
        for (int s = 0; s < kRtStages; ++s) {
            ptx::mbar_init(&hd->full[s], 1);
            ptx::mbar_init(&hd->empty[s], 1);
        }
        ptx::mbar_init(&hd->done, 1);
        ptx::fence_barrier_init();
        ptx::prefetch_tmap(&tmX);
    }
    if (warp == 1) tmem_alloc(&hd->tmem, 32);
    // W_r^T slice: panel i holds d = (kb0 + i) * 64 + c, c < 64; row e of the
    // panel is expert e (zero past E or past D)
    const bool vec = E == 16;  // a router row is 32 B: two 16-byte loads
#pragma unroll 4
    for (int idx = threadIdx.x; idx < nkb * kRtBK; idx += kRtThreads) {
        const int i = idx / kRtBK, c = idx - i * kRtBK;
        const int d = (kb0 + i) * kRtBK + c;
        unsigned char *panel = wt + i * kRtPanelBytes;
        uint32_t w[8];  // 16 bf16, expert e in half (e & 1) of w[e / 2]
        if (d < D && vec) {
            const uint4 a = __ldg(reinterpret_cast<const uint4 *>(wr + (size_t)d * 16));
            const uint4 b = __ldg(reinterpret_cast<const uint4 *>(wr + (size_t)d * 16 + 8));
            w[0] = a.x; w[1] = a.y; w[2] = a.z; w[3] = a.w;
            w[4] = b.x; w[5] = b.y; w[6] = b.z; w[7] = b.w;
        } else {
            const unsigned short *row = reinterpret_cast<const unsigned short *>(wr) + (size_t)d * E;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const uint32_t lo = (d < D && 2 * j < E) ? row[2 * j] : 0u;
                const uint32_t hi = (d < D && 2 * j + 1 < E) ? row[2 * j + 1] : 0u;
                w[j] = lo | (hi << 16);
            }
        }
#pragma unroll
        for (int e = 0; e < 16; ++e)
            *reinterpret_cast<unsigned short *>(panel + swizzle_offset((uint32_t)e, (uint32_t)c)) =
                (unsigned short)(w[e >> 1] >> ((e & 1) * 16));
    }
    fence_proxy_async_smem();  // the slice is read by the MMA (async proxy)
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = hd->tmem;
    ptx::grid_dependency_wait();  // the token rows may come from the previous kernel

    if (warp == 0) {
        if (lane == 0) {
            const uint64_t pol = ptx::policy_evict_first();
            int i = 0;
            for (; i < nkb; ++i) {
                const uint32_t s = i % kRtStages, ph = (i / kRtStages) & 1;
                if (!ptx::mbar_wait_hint(&hd->empty[s], ph ^ 1, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->full[s], kRtStageBytes);
                ptx::tma_load_2d(smem + s * kRtStageBytes, &tmX, (kb0 + i) * kRtBK, m0,
                                 &hd->full[s], pol);
            }
            // let copies still in flight land before the block can exit
            for (int k = (i > kRtStages ? i - kRtStages : 0); k < i; ++k)
                ptx::mbar_wait_hint(&hd->full[k % kRtStages], (k / kRtStages) & 1, err);
        }
        __syncwarp();
    } else if (warp == 1) {
        if (lane == 0) {
            for (int i = 0; i < nkb; ++i) {
                const uint32_t s = i % kRtStages, ph = (i / kRtStages) & 1;
                if (!ptx::mbar_wait_hint(&hd->full[s], ph, err)) break;
                tc_fence_after();
                const uint64_t adesc = smem_desc(ptx::smem_u32(smem + s * kRtStageBytes));
                const uint64_t bdesc = smem_desc(ptx::smem_u32(wt + i * kRtPanelBytes));
#pragma unroll
                for (int kk = 0; kk < kRtBK / 16; ++kk)
                    mma_bf16(tmem, adesc + 2 * kk, bdesc + 2 * kk, kRtIdesc, (i | kk) != 0 ? 1u : 0u);
                mma_commit(&hd->empty[s]);
            }
            // `done` flips once every MMA issued here has completed
            mma_commit(&hd->done);
        }
        __syncwarp();
    }
    // every warp: its 32 tokens' partial logits
    if (ptx::mbar_wait_hint(&hd->done, 0, err)) {
        tc_fence_after();
        float v[32];
        tmem_ld32(tmem + ((uint32_t)(warp * 32) << 16), v);
        tmem_ld_wait();
        const int t = m0 + warp * 32 + lane;
        if (t < T && nkb > 0) {
            float4 *dst = reinterpret_cast<float4 *>(part + ((size_t)sh * T + t) * 16);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                dst[q] = make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]);
        } else if (t < T) {  // an empty share: zero partials
            float4 *dst = reinterpret_cast<float4 *>(part + ((size_t)sh * T + t) * 16);
#pragma unroll
            for (int q = 0; q < 4; ++q) dst[q] = make_float4(0.f, 0.f, 0.f, 0.f);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, 32);
}

constexpr int kTopkWarps = 8;

__global__ void __launch_bounds__(kTopkWarps * 32)
k_route_topk(int T, int E, int K, int ksplit, const float *__restrict__ part,
             float *__restrict__ logits_opt, int32_t *__restrict__ topk_idx,
             float *__restrict__ topk_gate) {
    __shared__ float lg[kTopkWarps][16];
    __shared__ float pk[kTopkWarps][16];
    ptx::grid_dependency_wait();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int t = blockIdx.x * kTopkWarps + warp;
    if (t >= T) return;
    if (lane < 16) {
        float v = 0.f;
        for (int s = 0; s < ksplit; ++s) v += part[((size_t)s * T + t) * 16 + lane];
        lg[warp][lane] = v;
    }
    __syncwarp();
    select_topk(E, K, t, lg[warp], pk[warp], logits_opt, topk_idx, topk_gate, nullptr);
}

}  // namespace

bool route_tc_ok(const moe_dims &d, int T) {
    return T >= kRtM && d.n_experts <= 16 && d.x_dtype == MOE_BF16 && d.w_dtype == MOE_BF16 &&
           encode_fn() != nullptr;
}

size_t route_tc_scratch_bytes(const moe_dims &d, int T) {
    const int m_tiles = (T + kRtM - 1) / kRtM;
    const int nkb = (d.d_model + kRtBK - 1) / kRtBK;
    int ksplit = std::max((nkb + kRtMaxKb - 1) / kRtMaxKb,
                          (device_info().sm_count + m_tiles - 1) / m_tiles);
    ksplit = std::min(ksplit, nkb);
    return (size_t)ksplit * T * 16 * sizeof(float);
}

cudaError_t launch_route_tc(const moe_dims &d, int T, const void *x, const void *wr,
                            float *logits, int32_t *idx, float *gate, float *scratch,
                            cudaStream_t st) {
    const int D = d.d_model;
    const int m_tiles = (T + kRtM - 1) / kRtM;
    const int nkb = (D + kRtBK - 1) / kRtBK;
    int ksplit = std::max((nkb + kRtMaxKb - 1) / kRtMaxKb,
                          (device_info().sm_count + m_tiles - 1) / m_tiles);
    ksplit = std::min(ksplit, nkb);
    CUtensorMap tmx;
    if (!make_map(&tmx, x, (uint64_t)T, (uint64_t)D, kRtM)) return cudaErrorInvalidValue;
    const void *kern = (const void *)k_route_tc;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)kRtSmem);
    if (e != cudaSuccess) return e;
    int Tv = T, Dv = D, E = d.n_experts, K = d.top_k, nkbv = nkb, ks = ksplit;
    const bf16 *wp = static_cast<const bf16 *>(wr);
    unsigned *err = device_info().err;
    {
        void *args[] = {&tmx, &Tv, &Dv, &E, &nkbv, &ks, &wp, &scratch, &err};
        LaunchScope ls("route", st);
        e = launch_pdl(kern, dim3(m_tiles, ksplit), dim3(kRtThreads), kRtSmem, st, args);
        if (e != cudaSuccess) return e;
    }
    const float *pc = scratch;
    void *args[] = {&Tv, &E, &K, &ks, &pc, &logits, &idx, &gate};
    LaunchScope ls("route_topk", st);
    return launch_pdl((const void *)k_route_topk, dim3((T + kTopkWarps - 1) / kTopkWarps),
                      dim3(kTopkWarps * 32), 0, st, args);
}

}  // namespace moe
