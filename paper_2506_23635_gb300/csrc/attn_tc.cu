// Causal attention of prefill tiles on the tcgen05 tensor cores.
//
// A tile is 128 consecutive tokens of one call that are consecutive positions
// p0 .. p0+127 of one sequence (a prefill chunk).  One CTA per (tile, query
// head h), key/value head g = h / (Hq/Hkv), over cache positions 0 .. p0+127
// in key/value tiles of 128 positions.  The grid runs every head of the last
// (longest) tile first, so the short tiles fill the end of the launch:
//
//   warp 0      TMA: the tile's bf16 queries once, then the key and the value
//               tiles of positions [128j, 128j+128) into two-stage rings;
//   warp 1      tensor memory (512 columns: two score buffers and one output
//               tile) and the MMAs: S_j = Q K_j^T (M = 128 queries, N = 128
//               positions, K = 128 dims) into score buffer j % 2, and once
//               the softmax warps have written P_j,
//               O += P_j V_j (M = 128 queries, N = 128 dims, K = 128
//               positions) into the output tile, which accumulates over the
//               key/value tiles; V_j read as it lies in the cache: an
//               MN-major operand (dims contiguous, 128-byte swizzle), so no
//               transpose;
//   warps 2-9   two threads per query row, each owning 64 of the 128 score
//               columns and of the 128 output dims: zero the rows of V_j past
//               the tile's last query (a key/value tile that runs past it:
//               those cache rows may hold anything, and 0 * NaN is NaN), then
//               the online softmax of S_j (causal mask, base-2 exponent of the
//               1/sqrt(128)-scaled scores, two columns per packed fp32x2
//               instruction; the two threads of a row exchange their maxima
//               through shared memory at a barrier of their two warps) into
//               bf16 probabilities P_j, held in registers until
//               P_{j-1} V_{j-1} has finished and then written in the
//               128-byte-swizzled K-major layout the MMA reads.  The exponent
//               base of a row moves only when the row maximum passes it by
//               more than 8 (a factor of 2^8); then the same threads rescale
//               their half row of O in tensor memory first.
//
// At 2048 tokens, against 142 us for the form with O folded into registers
// after every tile and the heads of one query tile spread over the launch:
// longest tiles first 128 us, sleeping waits and split max/sum chains
// 124 us, O kept in tensor memory 118 us, packed fp32x2 arithmetic 108 us.
// What remains is latency along one chain per key/value tile (~2900 cycles:
// barrier waits, the max exchange, the exponentials, the P stores and the
// proxy fence) with the tensor pipe busy a third of it; more softmax warps
// (four threads per row) or P written to tensor memory did not shorten it.
//
// Every wait is bounded (ptx.cuh) and sleeps on its barrier (suspend-time
// hint) instead of spinning, which leaves issue slots to the softmax warps.
// Tiles that do not satisfy the layout condition record tile_ok = 0 and are
// left to the CUDA-core kernel.
#include <math.h>

#include "tc.cuh"

namespace moe {
namespace {

using namespace tc;

constexpr int kFa = 128;                 // queries per tile, positions per key/value tile
constexpr int kHeadDimFa = 128;
constexpr int kFaSoftmaxWarps = 8;       // two threads per query row
constexpr int kFaGroups = kFaSoftmaxWarps / 4;  // threads (column groups) per query row
constexpr int kFaCols = kFa / kFaGroups;        // score columns and output dims per thread
static_assert(kFaCols % 32 == 0, "tensor-memory loads of 32 columns");
// how far (base 2) the row maximum may pass the exponent base in use before
// the base moves and O is rescaled: probabilities up to 2^8, exact in bf16
constexpr float kFaRescale = 8.f;
constexpr int kFaThreads = (2 + kFaSoftmaxWarps) * 32;
constexpr uint32_t kHalfBytes = kFa * 128;     // one 64-column half of a 128-row tile
constexpr uint32_t kTileBytes = 2 * kHalfBytes;  // 32 KB
// shared memory: Q, K[2], V[2], P (each a 32 KB tile), then the header
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = kTileBytes;
constexpr uint32_t kOffV = 3 * kTileBytes;
constexpr uint32_t kOffP = 5 * kTileBytes;
constexpr uint32_t kOffHdr = 6 * kTileBytes;
// row maxima exchange [2 buffers][kFaGroups][128] floats, then the row sums
// [kFaGroups][128] in a region of their own (a slow thread of the row may still
// be reading the last tile's maxima)
constexpr uint32_t kOffRed = kOffHdr + 256;
constexpr size_t kFaSmem = 1024 + kOffRed + 3 * kFaGroups * kFa * 4;
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

// Wait for a barrier phase: a non-blocking test, then the bounded wait that
// sleeps on the barrier.  (Even on a phase that has completed, a wait costs
// ~200-600 cycles here, measured with clock stamps, whichever form it takes.)
__device__ __forceinline__ bool fa_wait(uint64_t *bar, uint32_t parity, unsigned *err) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(ptx::smem_u32(bar)), "r"(parity)
        : "memory");
    return done != 0 || ptx::mbar_wait_hint(bar, parity, err);
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
// 128 dims] as stored (MN-major); K = 16 positions per instruction.  The
// first key/value tile overwrites O, the later ones add to it.
__device__ __forceinline__ void issue_pv(uint32_t d_tmem, uint32_t p_smem, uint32_t v_smem,
                                         bool accumulate) {
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
        const uint64_t ad = smem_desc(p_smem + (ks >> 2) * kHalfBytes) + 2 * (ks & 3);
        const uint64_t bd = smem_desc_mn(v_smem + ks * 16 * 128);
        mma_bf16(d_tmem, ad, bd, kFaIdescVmn, (accumulate || ks != 0) ? 1u : 0u);
    }
}

// 32 columns of this warp's 32 tensor-memory lanes from registers.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const float (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "f"(v[0]), "f"(v[1]), "f"(v[2]), "f"(v[3]), "f"(v[4]), "f"(v[5]), "f"(v[6]), "f"(v[7]),
        "f"(v[8]), "f"(v[9]), "f"(v[10]), "f"(v[11]), "f"(v[12]), "f"(v[13]), "f"(v[14]),
        "f"(v[15]), "f"(v[16]), "f"(v[17]), "f"(v[18]), "f"(v[19]), "f"(v[20]), "f"(v[21]),
        "f"(v[22]), "f"(v[23]), "f"(v[24]), "f"(v[25]), "f"(v[26]), "f"(v[27]), "f"(v[28]),
        "f"(v[29]), "f"(v[30]), "f"(v[31])
        : "memory");
}

__device__ __forceinline__ void tmem_st_wait() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
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
    const int tile = n_tiles - 1 - (int)blockIdx.y;  // the longest tiles first
    const int h = blockIdx.x, g = h / (Hq / Hkv);
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
                if (!fa_wait(&hd->kv_empty[b], ((j >> 1) & 1) ^ 1, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->kv_full[b], kTileBytes);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kOffK + b * kTileBytes + half * kHalfBytes, &tmK,
                                     half * 64, row0 + j * kFa, &hd->kv_full[b], pol);
                issued = j + 1;
                if (!fa_wait(&hd->v_empty[b], ((j >> 1) & 1) ^ 1, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->v_full[b], kTileBytes);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kOffV + b * kTileBytes + half * kHalfBytes, &tmV,
                                     half * 64, row0 + j * kFa, &hd->v_full[b], pol);
                v_issued = j + 1;
            }
            // let loads still in flight land before the block can exit
            fa_wait(&hd->q_full, 0, err);
            for (int j = (issued > 2 ? issued - 2 : 0); j < issued; ++j)
                fa_wait(&hd->kv_full[j & 1], (j >> 1) & 1, err);
            for (int j = (v_issued > 2 ? v_issued - 2 : 0); j < v_issued; ++j)
                fa_wait(&hd->v_full[j & 1], (j >> 1) & 1, err);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && ok) {
            bool good = fa_wait(&hd->q_full, 0, err);
            for (int j = 0; j <= n_kv && good; ++j) {
                if (j < n_kv) {  // S_j = Q K_j^T
                    const int b = j & 1;
                    if (!(good = fa_wait(&hd->kv_full[b], (j >> 1) & 1, err))) break;
                    if (!(good = fa_wait(&hd->s_free[b], ((j >> 1) & 1) ^ 1, err))) break;
                    tc_fence_after();
                    issue_128x128x128(tmem + b * kFa, sbase + kOffQ, sbase + kOffK + b * kTileBytes);
                    mma_commit(&hd->s_full[b]);
                    mma_commit(&hd->kv_empty[b]);  // key tile j read once these finish
                }
                if (j >= 1) {  // O_{j-1} = P_{j-1} V_{j-1}
                    const int jp = j - 1;
                    if (!(good = fa_wait(&hd->v_full[jp & 1], (jp >> 1) & 1, err))) break;
                    if (!(good = fa_wait(&hd->p_ready, jp & 1, err))) break;
                    tc_fence_after();
                    issue_pv(tmem + 2 * kFa, sbase + kOffP, sbase + kOffV + (jp & 1) * kTileBytes,
                             jp != 0);
                    mma_commit(&hd->o_full);
                    mma_commit(&hd->v_empty[jp & 1]);  // value tile jp read once these finish
                }
            }
            mma_commit(&hd->done);
            fa_wait(&hd->done, 0, err);
        }
        __syncwarp();
    } else if (ok) {
        // ------------------------------------------------------------ softmax
        const int q = warp & 3;                  // tensor-memory lane quarter
        const int r = q * 32 + lane;             // query row of the tile
        const int cg = (warp - 2) >> 2;          // column group: scores and output dims
        const int c0 = cg * kFaCols;
        const int qpos = p0 + r;
        const int last = p0 + kFa - 1;           // the tile's last query position
        const float sl2 = 1.4426950408889634f / sqrtf((float)kHeadDimFa);
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        float *red = reinterpret_cast<float *>(smem + kOffRed);  // [2 buffers][kFaGroups][128]
        float *rsum = red + 2 * kFaGroups * kFa;                  // [kFaGroups][128]
        // the kFaGroups warps of lane quarter q hold the same rows: they alone
        // meet at named barrier 1 + q
        const int bar_id = 1 + q;
        // m: the exponent base of the row (scaled scores), which may trail the
        // row maximum by up to kFaRescale; l: this thread's share of the row sum
        float m = -INFINITY, l = 0.f;
        // every softmax warp runs every iteration and reaches every named
        // barrier: a wait that gave up (recorded in err) turns the later waits
        // into no-ops instead of leaving the loop early
        bool good = true;
        for (int j = 0; j < n_kv; ++j) {
            const int b = j & 1;
            // a value tile that runs past the tile's last query: its rows past
            // `last` are zeroed before P_j V_j reads them (P is zero there, but
            // those cache rows may hold anything); thread (r, cg) clears the
            // dims of its column group in row r
            if (j * kFa + kFa - 1 > last) {
                good = good && fa_wait(&hd->v_full[b], (j >> 1) & 1, err);
                if (j * kFa + r > last) {
                    unsigned char *vt = smem + kOffV + b * kTileBytes;
#pragma unroll
                    for (int c = 0; c < kFaCols; c += 8)
                        *reinterpret_cast<uint4 *>(vt + tile_offset((uint32_t)r, (uint32_t)(c0 + c))) =
                            make_uint4(0u, 0u, 0u, 0u);
                }
            }
            // scores of S_j (this thread's kFaCols columns): masked max,
            // exchanged with the row's other column groups, then probabilities
            good = good && fa_wait(&hd->s_full[b], (j >> 1) & 1, err);
            tc_fence_after();
            const uint32_t sb = tmem + lane_base + b * kFa + c0;
            const bool full = j * kFa + kFa - 1 <= p0;  // no position of the tile is masked
            float v[kFaCols];
#pragma unroll
            for (int c = 0; c < kFaCols; c += 32)
                tmem_ld32(sb + c, *reinterpret_cast<float(*)[32]>(&v[c]));
            tmem_ld_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->s_free[b]);  // scores read
            float hm4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            if (full) {
#pragma unroll
                for (int i = 0; i < kFaCols; ++i) hm4[i & 3] = fmaxf(hm4[i & 3], v[i]);
            } else {
#pragma unroll
                for (int i = 0; i < kFaCols; ++i)
                    if (j * kFa + c0 + i <= qpos) hm4[i & 3] = fmaxf(hm4[i & 3], v[i]);
            }
            const float hm = fmaxf(fmaxf(hm4[0], hm4[1]), fmaxf(hm4[2], hm4[3]));
            red[(b * kFaGroups + cg) * kFa + r] = hm;
            ptx::named_bar_sync(bar_id, kFaGroups * 32);
            // every thread of the row takes the groups' maxima in the same
            // order; finite: position 128j <= qpos for every row of the tile
            float rmax = red[(b * kFaGroups) * kFa + r];
#pragma unroll
            for (int g2 = 1; g2 < kFaGroups; ++g2) rmax = fmaxf(rmax, red[(b * kFaGroups + g2) * kFa + r]);
            const float mrow = rmax * sl2;
            // the base moves only when the row maximum passes it by more than
            // kFaRescale (the row's threads decide alike), so the
            // probabilities stay at most 2^kFaRescale and O is rarely rescaled
            const bool bump = mrow > m + kFaRescale;
            const float corr = bump ? exp2f(m - mrow) : 1.f;  // 0 on the first tile
            if (bump) m = mrow;
            // two columns per packed fp32x2 instruction
            float2 sum2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
            const float2 sl2x2 = make_float2(sl2, sl2), nm2 = make_float2(-m, -m);
            uint32_t pw[kFaCols / 2];
#pragma unroll
            for (int i = 0; i < kFaCols; i += 2) {
                const float2 x = __ffma2_rn(make_float2(v[i], v[i + 1]), sl2x2, nm2);
                float pa = fast_exp2(x.x);
                float pb = fast_exp2(x.y);
                if (!full) {
                    if (j * kFa + c0 + i > qpos) pa = 0.f;
                    if (j * kFa + c0 + i + 1 > qpos) pb = 0.f;
                }
                const __nv_bfloat162 p2 = __floats2bfloat162_rn(pa, pb);
                // the row sum takes the probabilities as stored, so the
                // weights P V is normalised by sum to exactly one
                sum2[(i >> 1) & 1] = __fadd2_rn(sum2[(i >> 1) & 1], __bfloat1622float2(p2));
                pw[i >> 1] = *reinterpret_cast<const uint32_t *>(&p2);
            }
            const float sum = (sum2[0].x + sum2[0].y) + (sum2[1].x + sum2[1].y);
            // P_{j-1} V_{j-1} has finished: the P buffer is free and the
            // output tile holds every earlier key/value tile
            if (j >= 1) {
                good = good && fa_wait(&hd->o_full, (j - 1) & 1, err);
                tc_fence_after();
                // the whole warp loads and stores (rows without a new base
                // scale by 1)
                if (__any_sync(0xffffffffu, bump) && __all_sync(0xffffffffu, good)) {
#pragma unroll
                    for (int c = 0; c < kFaCols; c += 32) {
                        float ov[32];
                        tmem_ld32(tmem + lane_base + 2 * kFa + c0 + c, ov);
                        tmem_ld_wait();
#pragma unroll
                        for (int i = 0; i < 32; ++i) ov[i] *= corr;
                        tmem_st32(tmem + lane_base + 2 * kFa + c0 + c, ov);
                    }
                    tmem_st_wait();
                }
            }
            unsigned char *ps = smem + kOffP;
#pragma unroll
            for (int i = 0; i < kFaCols; i += 8)
                *reinterpret_cast<uint4 *>(ps + tile_offset(r, c0 + i)) =
                    make_uint4(pw[i / 2], pw[i / 2 + 1], pw[i / 2 + 2], pw[i / 2 + 3]);
            fence_proxy_async_smem();  // P_j (and a clipped V_j) visible to the MMA
            tc_fence_before();         // and a rescaled O
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->p_ready);
            l = l * corr + sum;
        }
        // the row sum: the column groups' shares, in the same order for every
        // thread of the row
        rsum[cg * kFa + r] = l;
        ptx::named_bar_sync(bar_id, kFaGroups * 32);
        float lt = rsum[r];
#pragma unroll
        for (int g2 = 1; g2 < kFaGroups; ++g2) lt += rsum[g2 * kFa + r];
        bool fin = good && n_kv > 0;
        if (fin) fin = fa_wait(&hd->o_full, (n_kv - 1) & 1, err);
        if (__all_sync(0xffffffffu, fin)) {
            tc_fence_after();
            const float inv = lt > 0.f ? 1.f / lt : 0.f;
            bf16 *dst = ctx + ((size_t)(t0 + r) * Hq + h) * 128 + c0;
#pragma unroll
            for (int c = 0; c < kFaCols; c += 32) {
                float vv[32];
                tmem_ld32(tmem + lane_base + 2 * kFa + c0 + c, vv);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; i += 8) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float a = vv[i + 2 * e] * inv;
                        const float bq = vv[i + 2 * e + 1] * inv;
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
    return launch_pdl(kern, dim3(Hq, (T + kFa - 1) / kFa), dim3(kFaThreads), kFaSmem, st, args);
}

}  // namespace moe
