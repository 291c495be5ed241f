// Causal attention of prefill tiles on the tcgen05 tensor cores.
//
// A tile is 128 consecutive tokens of one call that are consecutive positions
// p0 .. p0+127 of one sequence (a prefill chunk).  One CTA per (tile, query
// head h), key/value head g = h / (Hq/Hkv), over cache positions 0 .. p0+127
// in key/value tiles of 128 positions:
//
//   warp 0      TMA: the tile's bf16 queries once, then the key and the value
//               tiles of positions [128j, 128j+128) into two-stage rings;
//   warp 1      tensor memory (512 columns: two score buffers and one output
//               tile) and the MMAs: S_j = Q K_j^T (M = 128 queries, N = 128
//               positions, K = 128 dims) into score buffer j % 2, and once
//               the softmax warps have written P_j,
//               O_j = P_j V_j (M = 128 queries, N = 128 dims, K = 128
//               positions) into the output tile, V_j read as it lies in the
//               cache: an MN-major operand (dims contiguous, 128-byte
//               swizzle), so no transpose;
//   warps 2-9   two threads per query row, each owning 64 of the 128 score
//               columns and of the 128 output dims: fold O_{j-1} into the
//               row's fp32 accumulator (registers), zero the rows of V_j past
//               the tile's last query (a key/value tile that runs past it:
//               those cache rows may hold anything, and 0 * NaN is NaN), then
//               the online softmax of S_j (causal mask, base-2 exponent of the
//               1/sqrt(128)-scaled scores; the two halves of a row exchange
//               their maxima through shared memory) and the bf16
//               probabilities P_j, written in the 128-byte-swizzled K-major
//               layout the MMA reads.
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
constexpr int kFaSoftmaxWarps = 8;       // two threads per query row
constexpr int kFaThreads = (2 + kFaSoftmaxWarps) * 32;
constexpr uint32_t kHalfBytes = kFa * 128;     // one 64-column half of a 128-row tile
constexpr uint32_t kTileBytes = 2 * kHalfBytes;  // 32 KB
// shared memory: Q, K[2], V[2], P (each a 32 KB tile), then the header
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kTileBytes;
constexpr uint32_t kOffV = 3 * kTileBytes;
constexpr uint32_t kOffP = 5 * kTileBytes;
constexpr uint32_t kOffHdr = 6 * kTileBytes;
constexpr uint32_t kOffRed = kOffHdr + 256;  // row max / sum exchange: [2][2][128] floats
constexpr size_t kFaSmem = 1024 + kOffRed + 2 * 2 * kFa * 4;
static_assert(kFaSmem <= 227 * 1024, "shared memory");
// kind::f16 instruction descriptor: bf16 A and B, fp32 D, K-major, N = M = 128
constexpr uint32_t kFaIdesc =
    (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kFa >> 3) << 17) | ((uint32_t)(kFa >> 4) << 24);
// the same with B MN-major (bit 16): O = P V with V as stored
constexpr uint32_t kFaIdescVmn = kFaIdesc | (1u << 16);
constexpr uint32_t kFaTmemCols = 512;  // S[0] 0..127, S[1] 128..255, O 256..383

struct FaHeader {
    uint64_t q_full;
    uint64_t kv_full[2];   // key tile j in stage j % 2
    uint64_t kv_empty[2];
    uint64_t v_full[2];    // value tile j in stage j % 2
    uint64_t v_empty[2];   // the MMA of O_j has read it
    uint64_t s_full[2];
    uint64_t s_free[2];  // the softmax warps have read score buffer b (one arrival each)
    uint64_t p_ready;    // P_j and V_j^T written (one arrival per softmax warp)
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

// 2^x on the special-function unit (the probabilities are rounded to bf16
// right after, far coarser than its error).
__device__ __forceinline__ float fast_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// Shared-memory descriptor of an MN-major operand written by TMA with the
// 128-byte swizzle: a row of 128 B holds 64 consecutive MN elements of one k,
// 8 rows (k) make a 1024-byte atom; the next 8 k follow 1024 B on (stride
// offset), the next 64 MN elements 16 KB on (leading offset: the second
// 64-column box of the tile).
__device__ __forceinline__ uint64_t smem_desc_mn(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(kHalfBytes >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// O (+)= P V: P [128 queries, 128 positions] K-major, V [128 positions,
// 128 dims] as stored (MN-major); K = 16 positions per instruction.
__device__ __forceinline__ void issue_pv(uint32_t d_tmem, uint32_t p_smem, uint32_t v_smem) {
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
        const uint64_t ad = smem_desc(p_smem + (ks >> 2) * kHalfBytes) + 2 * (ks & 3);
        const uint64_t bd = smem_desc_mn(v_smem + ks * 16 * 128);
        mma_bf16(d_tmem, ad, bd, kFaIdescVmn, ks != 0 ? 1u : 0u);
    }
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
            ptx::mbar_init(&hd->s_free[b], kFaSoftmaxWarps);
        }
        ptx::mbar_init(&hd->p_ready, kFaSoftmaxWarps);
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&hd->v_full[b], 1);
            ptx::mbar_init(&hd->v_empty[b], 1);
        }
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
            int v_issued = 0;
            for (int j = 0; j < n_kv; ++j) {
                const int b = j & 1;
                if (!ptx::mbar_wait(&hd->kv_empty[b], ((j >> 1) & 1) ^ 1, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->kv_full[b], kTileBytes);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kOffK + b * kTileBytes + half * kHalfBytes, &tmK,
                                     half * 64, row0 + j * kFa, &hd->kv_full[b], pol);
                issued = j + 1;
                if (!ptx::mbar_wait(&hd->v_empty[b], ((j >> 1) & 1) ^ 1, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->v_full[b], kTileBytes);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kOffV + b * kTileBytes + half * kHalfBytes, &tmV,
                                     half * 64, row0 + j * kFa, &hd->v_full[b], pol);
                v_issued = j + 1;
            }
            // let loads still in flight land before the block can exit
            ptx::mbar_wait(&hd->q_full, 0, err);
            for (int j = (issued > 2 ? issued - 2 : 0); j < issued; ++j)
                ptx::mbar_wait(&hd->kv_full[j & 1], (j >> 1) & 1, err);
            for (int j = (v_issued > 2 ? v_issued - 2 : 0); j < v_issued; ++j)
                ptx::mbar_wait(&hd->v_full[j & 1], (j >> 1) & 1, err);
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
                    mma_commit(&hd->kv_empty[b]);  // key tile j read once these finish
                }
                if (j >= 1) {  // O_{j-1} = P_{j-1} V_{j-1}
                    const int jp = j - 1;
                    if (!(good = ptx::mbar_wait(&hd->v_full[jp & 1], (jp >> 1) & 1, err))) break;
                    if (!(good = ptx::mbar_wait(&hd->p_ready, jp & 1, err))) break;
                    tc_fence_after();
                    issue_pv(tmem + 2 * kFa, sbase + kOffP, sbase + kOffV + (jp & 1) * kTileBytes);
                    mma_commit(&hd->o_full);
                    mma_commit(&hd->v_empty[jp & 1]);  // value tile jp read once these finish
                }
            }
            mma_commit(&hd->done);
            ptx::mbar_wait(&hd->done, 0, err);
        }
        __syncwarp();
    } else if (ok) {
        // ------------------------------------------------------------ softmax
        const int q = warp & 3;                  // tensor-memory lane quarter
        const int r = q * 32 + lane;             // query row of the tile
        const int w8 = warp - 2;                 // 0..7
        const int hf = w8 >> 2;                  // column half: scores and output dims
        const int c0 = hf * 64;
        const int qpos = p0 + r;
        const int last = p0 + kFa - 1;           // the tile's last query position
        const float sl2 = 1.4426950408889634f / sqrtf((float)kHeadDimFa);
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        float *red = reinterpret_cast<float *>(smem + kOffRed);  // [2 buffers][2 halves][128]
        float o[64];
#pragma unroll
        for (int i = 0; i < 64; ++i) o[i] = 0.f;
        float m = -INFINITY, l = 0.f, corr = 1.f;  // l: this half's share of the row sum
        // every softmax warp runs every iteration and reaches every named
        // barrier: a wait that gave up (recorded in err) turns the later waits
        // into no-ops instead of leaving the loop early
        bool good = true;
        for (int j = 0; j < n_kv; ++j) {
            const int b = j & 1;
            if (j >= 1) {  // fold O_{j-1}; then P, V^T and the output tile are free
                good = good && ptx::mbar_wait(&hd->o_full, (j - 1) & 1, err);
                tc_fence_after();
#pragma unroll
                for (int c = 0; c < 64; c += 32) {
                    float v[32];
                    tmem_ld32(tmem + lane_base + 2 * kFa + c0 + c, v);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) o[c + i] = fmaf(o[c + i], corr, v[i]);
                }
            }
            // a value tile that runs past the tile's last query: its rows past
            // `last` are zeroed before P_j V_j reads them (P is zero there, but
            // those cache rows may hold anything); thread (r, hf) clears half
            // hf of row r
            if (j * kFa + kFa - 1 > last) {
                good = good && ptx::mbar_wait(&hd->v_full[b], (j >> 1) & 1, err);
                if (j * kFa + r > last) {
                    unsigned char *vrow = smem + kOffV + b * kTileBytes + hf * kHalfBytes;
#pragma unroll
                    for (int c = 0; c < 64; c += 8)
                        *reinterpret_cast<uint4 *>(vrow + swizzle_offset((uint32_t)r, (uint32_t)c)) =
                            make_uint4(0u, 0u, 0u, 0u);
                }
            }
            // scores of S_j (this thread's 64 columns): masked max, exchanged
            // with the other half of the row, then probabilities
            good = good && ptx::mbar_wait(&hd->s_full[b], (j >> 1) & 1, err);
            tc_fence_after();
            const uint32_t sb = tmem + lane_base + b * kFa + c0;
            const bool full = j * kFa + kFa - 1 <= p0;  // no position of the tile is masked
            float v[64];
            tmem_ld32(sb, *reinterpret_cast<float(*)[32]>(&v[0]));
            tmem_ld32(sb + 32, *reinterpret_cast<float(*)[32]>(&v[32]));
            tmem_ld_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->s_free[b]);  // scores read
            float hm = -INFINITY;
            if (full) {
#pragma unroll
                for (int i = 0; i < 64; ++i) hm = fmaxf(hm, v[i]);
            } else {
#pragma unroll
                for (int i = 0; i < 64; ++i)
                    if (j * kFa + c0 + i <= qpos) hm = fmaxf(hm, v[i]);
            }
            red[(b * 2 + hf) * kFa + r] = hm;
            ptx::named_bar_sync(1, kFaSoftmaxWarps * 32);
            const float other = red[(b * 2 + (hf ^ 1)) * kFa + r];
            // finite: position 128j <= qpos for every row of the tile
            const float mx = fmaxf(m, fmaxf(hm, other) * sl2);
            float sum = 0.f;
            unsigned char *ps = smem + kOffP;
#pragma unroll
            for (int i = 0; i < 64; i += 8) {
                uint32_t w[4];
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    const int ca = c0 + i + 2 * e;
                    float pa = fast_exp2(fmaf(v[i + 2 * e], sl2, -mx));
                    float pb = fast_exp2(fmaf(v[i + 2 * e + 1], sl2, -mx));
                    if (!full) {
                        if (j * kFa + ca > qpos) pa = 0.f;
                        if (j * kFa + ca + 1 > qpos) pb = 0.f;
                    }
                    const __nv_bfloat162 p2 = __floats2bfloat162_rn(pa, pb);
                    // the row sum takes the probabilities as stored, so the
                    // weights P V is normalised by sum to exactly one
                    sum += __low2float(p2) + __high2float(p2);
                    w[e] = *reinterpret_cast<const uint32_t *>(&p2);
                }
                *reinterpret_cast<uint4 *>(ps + tile_offset(r, c0 + i)) = make_uint4(w[0], w[1], w[2], w[3]);
            }
            fence_proxy_async_smem();  // P_j (and a clipped V_j) visible to the MMA
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->p_ready);
            corr = exp2f(m - mx);  // 0 on the first tile (m = -inf)
            l = l * corr + sum;
            m = mx;
        }
        // the row sum: both halves' shares
        red[hf * kFa + r] = l;
        ptx::named_bar_sync(1, kFaSoftmaxWarps * 32);
        const float lt = l + red[(hf ^ 1) * kFa + r];
        if (good && n_kv > 0 && ptx::mbar_wait(&hd->o_full, (n_kv - 1) & 1, err)) {
            tc_fence_after();
            const float inv = lt > 0.f ? 1.f / lt : 0.f;
            bf16 *dst = ctx + ((size_t)(t0 + r) * Hq + h) * 128 + c0;
#pragma unroll
            for (int c = 0; c < 64; c += 32) {
                float vv[32];
                tmem_ld32(tmem + lane_base + 2 * kFa + c0 + c, vv);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; i += 8) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float a = fmaf(o[c + i + 2 * e], corr, vv[i + 2 * e]) * inv;
                        const float bq = fmaf(o[c + i + 2 * e + 1], corr, vv[i + 2 * e + 1]) * inv;
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
