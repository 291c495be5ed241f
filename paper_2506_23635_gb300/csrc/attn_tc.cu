// Causal attention of prefill tiles on the tcgen05 tensor cores.
//
// A tile is 128 consecutive tokens of one call that are consecutive positions
// p0 .. p0+127 of one sequence (a prefill chunk).  One CTA per (tile, query
// head h), key/value head g = h / (Hq/Hkv), over cache positions 0 .. p0+127
// in key/value tiles of 128 positions:
//
//   warp 0      TMA: the tile's bf16 queries once, then the key and value
//               tiles of positions [128j, 128j+128) into a two-stage ring;
//   warp 1      tensor memory (512 columns: two score buffers and one output
//               tile) and the MMAs: S_j = Q K_j^T (M = 128 queries, N = 128
//               positions, K = 128 dims) into score buffer j % 2, and once
//               the softmax warps have written P_j and V_j^T,
//               O_j = P_j V_j (M = 128 queries, N = 128 dims, K = 128
//               positions) into the output tile;
//   warps 2-5   one thread per query row: fold O_{j-1} into the row's fp32
//               accumulator (registers), transpose V_j into the K-major V^T
//               tile (positions past the tile's last query are written as
//               zero), then the online softmax of S_j (causal mask, base-2
//               exponent of the 1/sqrt(128)-scaled scores) and the bf16
//               probabilities P_j, both written in the 128-byte-swizzled
//               K-major layout the MMA reads.
//
// Every wait is bounded (ptx.cuh).  Tiles that do not satisfy the layout
// condition record tile_ok = 0 and are left to the CUDA-core kernel.
#include <math.h>

#include "tc.cuh"

namespace moe {
namespace {

using namespace tc;

constexpr int kFa = 128;                 // queries per tile, positions per key/value tile
constexpr int kHeadDimFa = 128;
constexpr int kFaThreads = 192;          // 6 warps
constexpr uint32_t kHalfBytes = kFa * 128;     // one 64-column half of a 128-row tile
constexpr uint32_t kTileBytes = 2 * kHalfBytes;  // 32 KB
// shared memory: Q, K[2], V[2], V^T, P (each a 32 KB tile), then the header
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kTileBytes;
constexpr uint32_t kOffV = 3 * kTileBytes;
constexpr uint32_t kOffVt = 5 * kTileBytes;
constexpr uint32_t kOffP = 6 * kTileBytes;
constexpr uint32_t kOffHdr = 7 * kTileBytes;
constexpr size_t kFaSmem = 1024 + kOffHdr + 256;
static_assert(kFaSmem <= 227 * 1024, "shared memory");
// kind::f16 instruction descriptor: bf16 A and B, fp32 D, K-major, N = M = 128
constexpr uint32_t kFaIdesc =
    (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kFa >> 3) << 17) | ((uint32_t)(kFa >> 4) << 24);
constexpr uint32_t kFaTmemCols = 512;  // S[0] 0..127, S[1] 128..255, O 256..383

struct FaHeader {
    uint64_t q_full;
    uint64_t kv_full[2];
    uint64_t kv_empty[2];
    uint64_t s_full[2];
    uint64_t s_free[2];  // the softmax warps have read score buffer b (4 arrivals)
    uint64_t p_ready;    // P_j and V_j^T written (4 arrivals)
    uint64_t o_full;
    uint64_t done;
    uint32_t tmem_base;
    int ok;
};
static_assert(sizeof(FaHeader) <= 256, "flash-attention header");

// 128 x 128 bf16 tile: two 64-column halves, K-major, 128-byte swizzle.
__device__ __forceinline__ uint32_t tile_offset(uint32_t r, uint32_t k) {
    return (k >> 6) * kHalfBytes + swizzle_offset(r, k & 63u);
}

__device__ __forceinline__ void issue_128x128x128(uint32_t d_tmem, uint32_t a_smem, uint32_t b_smem) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const uint64_t ad = smem_desc(a_smem + half * kHalfBytes);
        const uint64_t bd = smem_desc(b_smem + half * kHalfBytes);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
            mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, kFaIdesc, (half | kk) != 0 ? 1u : 0u);
    }
}

__global__ void __launch_bounds__(kFaThreads, 1)
k_attn_prefill_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                  const __grid_constant__ CUtensorMap tmV, int T, int Hq, int Hkv, int n_seq, int L,
                  const int32_t *__restrict__ seq, const int32_t *__restrict__ pos,
                  bf16 *__restrict__ ctx, int *__restrict__ tile_ok, unsigned *err) {
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    FaHeader *hd = reinterpret_cast<FaHeader *>(smem + kOffHdr);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int n_tiles = (T + kFa - 1) / kFa;
    const int tile = n_tiles - 1 - (int)blockIdx.x;  // the longest tiles first
    const int h = blockIdx.y, g = h / (Hq / Hkv);
    const int t0 = tile * kFa;

    if (threadIdx.x == 0) {
        ptx::mbar_init(&hd->q_full, 1);
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&hd->kv_full[b], 1);
            ptx::mbar_init(&hd->kv_empty[b], 1);
            ptx::mbar_init(&hd->s_full[b], 1);
            ptx::mbar_init(&hd->s_free[b], 4);
        }
        ptx::mbar_init(&hd->p_ready, 4);
        ptx::mbar_init(&hd->o_full, 1);
        ptx::mbar_init(&hd->done, 1);
        ptx::fence_barrier_init();
        ptx::prefetch_tmap(&tmQ);
        ptx::prefetch_tmap(&tmK);
        ptx::prefetch_tmap(&tmV);
        hd->ok = 1;
    }
    if (warp == 1) tmem_alloc(&hd->tmem_base, kFaTmemCols);
    ptx::grid_dependency_wait();  // queries and caches come from the previous kernel
    __syncthreads();
    // the tile qualifies if its 128 tokens exist and are positions p0..p0+127
    // of one sequence inside the cache
    const int sq = seq[min(t0, T - 1)], p0 = pos[min(t0, T - 1)];
    if (threadIdx.x < kFa) {
        const int t = t0 + threadIdx.x;
        const bool good = t < T && seq[t] == sq && pos[t] == p0 + (int)threadIdx.x && sq >= 0 &&
                          sq < n_seq && p0 >= 0 && p0 + kFa <= L;
        if (!good) hd->ok = 0;
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = hd->tmem_base;
    const bool ok = hd->ok != 0;
    if (h == 0 && threadIdx.x == 0) tile_ok[tile] = ok ? 1 : 0;
    const int n_kv = ok ? (p0 + kFa - 1) / kFa + 1 : 0;  // key/value tiles 0 .. n_kv-1
    const uint32_t sbase = ptx::smem_u32(smem);

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0 && ok) {
            const uint64_t pol = ptx::policy_evict_last();
            ptx::mbar_arrive_expect_tx(&hd->q_full, kTileBytes);
            for (int half = 0; half < 2; ++half)
                ptx::tma_load_2d(smem + kOffQ + half * kHalfBytes, &tmQ, h * 128 + half * 64, t0,
                                 &hd->q_full, pol);
            const int row0 = (sq * Hkv + g) * L;
            int issued = 0;
            for (int j = 0; j < n_kv; ++j) {
                const int b = j & 1;
                if (!ptx::mbar_wait(&hd->kv_empty[b], ((j >> 1) & 1) ^ 1, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->kv_full[b], 2 * kTileBytes);
                for (int half = 0; half < 2; ++half) {
                    ptx::tma_load_2d(smem + kOffK + b * kTileBytes + half * kHalfBytes, &tmK,
                                     half * 64, row0 + j * kFa, &hd->kv_full[b], pol);
                    ptx::tma_load_2d(smem + kOffV + b * kTileBytes + half * kHalfBytes, &tmV,
                                     half * 64, row0 + j * kFa, &hd->kv_full[b], pol);
                }
                issued = j + 1;
            }
            // let loads still in flight land before the block can exit
            ptx::mbar_wait(&hd->q_full, 0, err);
            for (int j = (issued > 2 ? issued - 2 : 0); j < issued; ++j)
                ptx::mbar_wait(&hd->kv_full[j & 1], (j >> 1) & 1, err);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && ok) {
            bool good = ptx::mbar_wait(&hd->q_full, 0, err);
            for (int j = 0; j <= n_kv && good; ++j) {
                if (j < n_kv) {  // S_j = Q K_j^T
                    const int b = j & 1;
                    if (!(good = ptx::mbar_wait(&hd->kv_full[b], (j >> 1) & 1, err))) break;
                    if (!(good = ptx::mbar_wait(&hd->s_free[b], ((j >> 1) & 1) ^ 1, err))) break;
                    tc_fence_after();
                    issue_128x128x128(tmem + b * kFa, sbase + kOffQ, sbase + kOffK + b * kTileBytes);
                    mma_commit(&hd->s_full[b]);
                }
                if (j >= 1) {  // O_{j-1} = P_{j-1} V_{j-1}
                    const int jp = j - 1;
                    if (!(good = ptx::mbar_wait(&hd->p_ready, jp & 1, err))) break;
                    tc_fence_after();
                    issue_128x128x128(tmem + 2 * kFa, sbase + kOffP, sbase + kOffVt);
                    mma_commit(&hd->o_full);
                    mma_commit(&hd->kv_empty[jp & 1]);
                }
            }
            mma_commit(&hd->done);
            ptx::mbar_wait(&hd->done, 0, err);
        }
        __syncwarp();
    } else if (ok) {
        // ------------------------------------------------------------ softmax
        const int q = warp & 3;             // tensor-memory lane quarter
        const int r = q * 32 + lane;        // query row of the tile
        const int st = (warp - 2) * 32 + lane;  // 0..127: the V^T row this thread writes
        const int qpos = p0 + r;
        const int last = p0 + kFa - 1;      // the tile's last query position
        const float sl2 = 1.4426950408889634f / sqrtf((float)kHeadDimFa);
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        float o[128];
#pragma unroll
        for (int i = 0; i < 128; ++i) o[i] = 0.f;
        float m = -INFINITY, l = 0.f, corr = 1.f;
        bool good = true;
        for (int j = 0; j < n_kv && good; ++j) {
            const int b = j & 1;
            if (j >= 1) {  // fold O_{j-1}; then P, V^T and the output tile are free
                if (!(good = ptx::mbar_wait(&hd->o_full, (j - 1) & 1, err))) break;
                tc_fence_after();
#pragma unroll
                for (int c = 0; c < 128; c += 32) {
                    float v[32];
                    tmem_ld32(tmem + lane_base + 2 * kFa + c, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[c + i] = fmaf(o[c + i], corr, v[i]);
                }
            }
            // V_j -> V^T (row = dim st, column = position), zero past `last`
            if (!(good = ptx::mbar_wait(&hd->kv_full[b], (j >> 1) & 1, err))) break;
            {
                const unsigned char *vs = smem + kOffV + b * kTileBytes;
                unsigned char *vt = smem + kOffVt;
                const int d = st;
#pragma unroll 2
                for (int p8 = 0; p8 < kFa; p8 += 8) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int pa = p8 + 2 * e, pb = pa + 1;
                        const uint16_t va = *reinterpret_cast<const uint16_t *>(vs + tile_offset(pa, d));
                        const uint16_t vb = *reinterpret_cast<const uint16_t *>(vs + tile_offset(pb, d));
                        const uint32_t lo = j * kFa + pa <= last ? va : 0u;
                        const uint32_t hi = j * kFa + pb <= last ? vb : 0u;
                        w[e] = lo | (hi << 16);
                    }
                    *reinterpret_cast<uint4 *>(vt + tile_offset(d, p8)) = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
            // scores of S_j: masked row max, then probabilities
            if (!(good = ptx::mbar_wait(&hd->s_full[b], (j >> 1) & 1, err))) break;
            tc_fence_after();
            const uint32_t sb = tmem + lane_base + b * kFa;
            float mx = m;
#pragma unroll
            for (int c = 0; c < 128; c += 32) {
                float v[32];
                tmem_ld32(sb + c, v);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; ++i)
                    if (j * kFa + c + i <= qpos) mx = fmaxf(mx, v[i] * sl2);
            }
            // mx is finite: position 128j <= qpos for every row of the tile
            float sum = 0.f;
            unsigned char *ps = smem + kOffP;
#pragma unroll
            for (int c = 0; c < 128; c += 32) {
                float v[32];
                tmem_ld32(sb + c, v);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; i += 8) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int ca = c + i + 2 * e;
                        const float pa = j * kFa + ca <= qpos ? exp2f(v[i + 2 * e] * sl2 - mx) : 0.f;
                        const float pb =
                            j * kFa + ca + 1 <= qpos ? exp2f(v[i + 2 * e + 1] * sl2 - mx) : 0.f;
                        const __nv_bfloat162 p2 = __floats2bfloat162_rn(pa, pb);
                        // the row sum takes the probabilities as stored
                        sum += __low2float(p2) + __high2float(p2);
                        w[e] = *reinterpret_cast<const uint32_t *>(&p2);
                    }
                    *reinterpret_cast<uint4 *>(ps + tile_offset(r, c + i)) = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->s_free[b]);
            fence_proxy_async_smem();  // P_j and V_j^T visible to the MMA
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->p_ready);
            corr = exp2f(m - mx);  // 0 on the first tile (m = -inf)
            l = l * corr + sum;
            m = mx;
        }
        if (good && n_kv > 0 && ptx::mbar_wait(&hd->o_full, (n_kv - 1) & 1, err)) {
            tc_fence_after();
            const float inv = l > 0.f ? 1.f / l : 0.f;
            bf16 *dst = ctx + ((size_t)(t0 + r) * Hq + h) * 128;
#pragma unroll
            for (int c = 0; c < 128; c += 32) {
                float v[32];
                tmem_ld32(tmem + lane_base + 2 * kFa + c, v);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; i += 8) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float a = fmaf(o[c + i + 2 * e], corr, v[i + 2 * e]) * inv;
                        const float bq = fmaf(o[c + i + 2 * e + 1], corr, v[i + 2 * e + 1]) * inv;
                        const __nv_bfloat162 p2 = __floats2bfloat162_rn(a, bq);
                        w[e] = *reinterpret_cast<const uint32_t *>(&p2);
                    }
                    *reinterpret_cast<uint4 *>(dst + c + i) = make_uint4(w[0], w[1], w[2], w[3]);
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kFaTmemCols);
}

}  // namespace

bool attn_prefill_tc_ok() { return encode_fn() != nullptr; }

cudaError_t launch_attn_prefill_tc(int T, int Hq, int Hkv, int n_seq, int L, const int32_t *seq,
                                   const int32_t *pos, const void *q16, const void *k_cache,
                                   const void *v_cache, void *ctx, int *tile_ok, cudaStream_t st) {
    CUtensorMap mq, mk, mv;
    const uint64_t rows = (uint64_t)n_seq * Hkv * L;
    if (!make_map(&mq, q16, (uint64_t)T, (uint64_t)Hq * 128, kFa) ||
        !make_map(&mk, k_cache, rows, 128, kFa) || !make_map(&mv, v_cache, rows, 128, kFa))
        return cudaErrorInvalidValue;
    const void *kern = (const void *)k_attn_prefill_tc;
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kFaSmem);
    if (e != cudaSuccess) return e;
    unsigned *err = device_info().err;
    bf16 *cp = static_cast<bf16 *>(ctx);
    void *args[] = {&mq, &mk, &mv, &T, &Hq, &Hkv, &n_seq, &L, &seq, &pos, &cp, &tile_ok, &err};
    LaunchScope ls("attention_tc", st);
    return launch_pdl(kern, dim3((T + kFa - 1) / kFa, Hq), dim3(kFaThreads), kFaSmem, st, args);
}

}  // namespace moe
