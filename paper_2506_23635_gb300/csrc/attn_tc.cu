// Causal attention of prefill tiles on the tcgen05 tensor cores.
//
// A tile is 128 consecutive tokens of one call that are consecutive positions
// p0 .. p0+127 of one sequence (a prefill chunk).  One CTA per (tile, pair of
// query heads hA, hB = hA + 1 of one key/value head g), over cache positions
// 0 .. p0+127 in key/value tiles of 128 positions; the two heads share every
// key and value tile and every causal mask, so one copy stream feeds two
// independent softmax chains that take turns on the tensor cores (a group
// with an odd number of query heads leaves its last head alone in a CTA).
// The grid runs every head pair of the last (longest) tile first, so the
// short tiles fill the end of the launch.
//
//   warp 0      TMA: both heads' bf16 query tiles once, then the key and
//               the value tiles of positions [128j, 128j+128) into
//               two-stage rings;
//   warp 1      tensor memory (512 columns: per head a score tile S and an
//               output tile O) and the MMAs, per head: S_j = Q K_j^T
//               (M = 128 queries, N = 128 positions, K = 128 dims), and once
//               the head's softmax warps have written P_j,
//               O += P_j V_j (M = 128 queries, N = 128 dims, K = 128
//               positions) with P_j read from tensor memory, where it
//               replaced S_j, and V_j as it lies in the cache (an MN-major
//               operand: dims contiguous, 128-byte swizzle); S_{j+1} of a
//               head is issued once its P_j V_j has finished;
//   warps 2-5   head A, warps 6-9 head B: one thread per query row owning
//               all 128 score columns and output dims: the online softmax
//               of S_j (causal mask, base-2 exponent of the
//               1/sqrt(128)-scaled scores, two columns per packed fp32x2
//               instruction) into bf16 probabilities written back over S_j.
//               The exponent base of a row moves only when the row maximum
//               passes it by more than 8 (a factor of 2^8); then the thread
//               first rescales its row of O in tensor memory.  Head A's
//               threads also zero the rows of V_j past the tile's last
//               query (a key/value tile that runs past it: those cache rows
//               may hold anything, and 0 * NaN is NaN) before its P_j is
//               announced, which comes before either head's P_j V_j.
//
// At 2048 tokens (48 query heads): 94-100 us, against 108-113 us for one head
// per CTA with eight softmax warps (two threads per row and a row-max
// exchange).  By clock stamps a key/value tile takes ~5250 cycles for the two
// heads: each head's softmax ~2000, and the MMA thread, which alternates
// between the heads and waits for a head's P_j V_j before its S_{j+1} (P_j
// lives in S_j's columns), is busy all of it -- every wait costs 200-600
// cycles even on a completed phase.  One issuing thread per head instead
// let the two heads fall into step (both softmaxes at once, then both heads'
// MMAs): 108-110 us.
//
// Every wait is bounded (ptx.cuh) and sleeps on its barrier (suspend-time
// hint) instead of spinning.  Tiles that do not satisfy the layout condition
// record tile_ok = 0 and are left to the CUDA-core kernel.
#include <math.h>

#include "tc.cuh"

namespace moe {
namespace {

using namespace tc;

constexpr int kFa = 128;                 // queries per tile, positions per key/value tile
constexpr int kHeadDimFa = 128;
constexpr int kFaHeads = 2;              // query heads per CTA
constexpr int kFaWarpsPerHead = 4;       // one thread per query row
constexpr int kFaThreads = (2 + kFaHeads * kFaWarpsPerHead) * 32;
// how far (base 2) the row maximum may pass the exponent base in use before
// the base moves and O is rescaled: probabilities up to 2^8, well inside the
// range of bf16 (which rounds them as it would any other value)
constexpr float kFaRescale = 8.f;
constexpr uint32_t kHalfBytes = kFa * 128;       // one 64-column half of a 128-row tile
constexpr uint32_t kTileBytes = 2 * kHalfBytes;  // 32 KB
// shared memory: Q[2], K[2], V[2] (each a 32 KB tile), then the header
constexpr uint32_t kOffQ = 0;
constexpr uint32_t kOffK = 2 * kTileBytes;
constexpr uint32_t kOffV = 4 * kTileBytes;
constexpr uint32_t kOffHdr = 6 * kTileBytes;
constexpr size_t kFaSmem = 1024 + kOffHdr + 256;
static_assert(kFaSmem <= 227 * 1024, "shared memory");
// kind::f16 instruction descriptor: bf16 A and B, fp32 D, K-major, N = M = 128
constexpr uint32_t kFaIdesc =
    (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(kFa >> 3) << 17) | ((uint32_t)(kFa >> 4) << 24);
// the same with B MN-major (bit 16): O = P V with V as stored
constexpr uint32_t kFaIdescVmn = kFaIdesc | (1u << 16);
// tensor memory: head x's S (and P over its first 64 columns) at 128 x, its O
// at 256 + 128 x
constexpr uint32_t kFaTmemCols = 512;
constexpr uint32_t kColS = 0, kColO = 2 * kFa;

struct FaHeader {
    uint64_t q_full;
    uint64_t kv_full[2];   // key tile j in stage j % 2
    uint64_t kv_empty[2];  // both heads' S MMAs have read it
    uint64_t v_full[2];    // value tile j in stage j % 2
    uint64_t v_empty[2];   // both heads' P V MMAs have read it
    uint64_t s_full[kFaHeads];
    uint64_t p_ready[kFaHeads];  // P_j written (one arrival per softmax warp of the head)
    uint64_t o_full[kFaHeads];   // P_j V_j finished
    uint64_t done;
    uint32_t tmem_base;
    int ok;
};
static_assert(sizeof(FaHeader) <= 256, "flash-attention header");

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

// S = Q K^T: 128 queries x 128 positions over 128 dims, both K-major.
__device__ __forceinline__ void issue_qk(uint32_t d_tmem, uint32_t q_smem, uint32_t k_smem) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const uint64_t ad = smem_desc(q_smem + half * kHalfBytes);
        const uint64_t bd = smem_desc(k_smem + half * kHalfBytes);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
            mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, kFaIdesc, (half | kk) != 0 ? 1u : 0u);
    }
}

// O (+)= P V: P [128 queries, 128 positions] in tensor memory (row r in lane
// r, two positions per 32-bit column), V [128 positions, 128 dims] as stored
// (MN-major); K = 16 positions (8 columns of P) per instruction.  The first
// key/value tile overwrites O, the later ones add to it.
__device__ __forceinline__ void issue_pv(uint32_t d_tmem, uint32_t p_tmem, uint32_t v_smem,
                                         bool accumulate) {
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
        const uint64_t bd = smem_desc_mn(v_smem + ks * 16 * 128);
        const uint32_t acc = (accumulate || ks != 0) ? 1u : 0u;
        asm volatile(
            "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
            "tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n\t}" ::"r"(d_tmem),
            "r"(p_tmem + ks * 8), "l"(bd), "r"(kFaIdescVmn), "r"(acc));
    }
}

// 32 columns of this warp's 32 tensor-memory lanes from registers.
__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t (&v)[32]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16,"
        "%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31,%32};" ::"r"(taddr),
        "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
        "r"(v[8]), "r"(v[9]), "r"(v[10]), "r"(v[11]), "r"(v[12]), "r"(v[13]), "r"(v[14]),
        "r"(v[15]), "r"(v[16]), "r"(v[17]), "r"(v[18]), "r"(v[19]), "r"(v[20]), "r"(v[21]),
        "r"(v[22]), "r"(v[23]), "r"(v[24]), "r"(v[25]), "r"(v[26]), "r"(v[27]), "r"(v[28]),
        "r"(v[29]), "r"(v[30]), "r"(v[31])
        : "memory");
}

__device__ __forceinline__ void tmem_st_wait() {
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// 320 threads: three warps share two of the four schedulers' 16K-register
// files, so at most 168 registers a thread
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
    const int G = Hq / Hkv, pairs = (G + 1) / 2;
    const int g = (int)blockIdx.x / pairs, hp = (int)blockIdx.x - g * pairs;
    const int h0 = g * G + 2 * hp;                // this CTA's first query head
    const int nh = 2 * hp + 1 < G ? 2 : 1;        // and how many it holds
    const int t0 = tile * kFa;

    if (threadIdx.x == 0) {
        ptx::mbar_init(&hd->q_full, 1);
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&hd->kv_full[b], 1);
            ptx::mbar_init(&hd->kv_empty[b], 1);
            ptx::mbar_init(&hd->v_full[b], 1);
            ptx::mbar_init(&hd->v_empty[b], 1);
        }
        for (int x = 0; x < kFaHeads; ++x) {
            ptx::mbar_init(&hd->s_full[x], 1);
            ptx::mbar_init(&hd->p_ready[x], kFaWarpsPerHead);
            ptx::mbar_init(&hd->o_full[x], 1);
        }
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
    if (blockIdx.x == 0 && threadIdx.x == 0) tile_ok[tile] = ok ? 1 : 0;
    const int n_kv = ok ? (p0 + kFa - 1) / kFa + 1 : 0;  // key/value tiles 0 .. n_kv-1
    const uint32_t sbase = ptx::smem_u32(smem);

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0 && ok) {
            const uint64_t pol = ptx::policy_evict_last();
            ptx::mbar_arrive_expect_tx(&hd->q_full, (uint32_t)nh * kTileBytes);
            for (int x = 0; x < nh; ++x)
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kOffQ + x * kTileBytes + half * kHalfBytes, &tmQ,
                                     (h0 + x) * 128 + half * 64, t0, &hd->q_full, pol);
            const int row0 = (sq * Hkv + g) * L;
            int issued = 0, v_issued = 0;
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
            bool good = fa_wait(&hd->q_full, 0, err) && fa_wait(&hd->kv_full[0], 0, err);
            if (good) {
                tc_fence_after();
                for (int x = 0; x < nh; ++x) {
                    issue_qk(tmem + kColS + x * kFa, sbase + kOffQ + x * kTileBytes, sbase + kOffK);
                    mma_commit(&hd->s_full[x]);
                }
                mma_commit(&hd->kv_empty[0]);  // key tile 0 read once these finish
            }
            for (int j = 0; j < n_kv && good; ++j) {
                const int b = j & 1;
                if (!(good = fa_wait(&hd->v_full[b], (j >> 1) & 1, err))) break;
                for (int x = 0; x < nh && good; ++x) {
                    // O += P_j V_j once the head's softmax warps have written P_j
                    if (!(good = fa_wait(&hd->p_ready[x], j & 1, err))) break;
                    tc_fence_after();
                    issue_pv(tmem + kColO + x * kFa, tmem + kColS + x * kFa,
                             sbase + kOffV + b * kTileBytes, j != 0);
                    mma_commit(&hd->o_full[x]);
                    if (x == nh - 1) mma_commit(&hd->v_empty[b]);  // value tile j read by both
                    if (j + 1 < n_kv) {
                        // S_{j+1} replaces P_j: only after P_j V_j has finished
                        const int b1 = (j + 1) & 1;
                        if (!(good = fa_wait(&hd->o_full[x], j & 1, err))) break;
                        // (head B follows head A, which has waited for key tile j+1)
                        if (x == 0 && !(good = fa_wait(&hd->kv_full[b1], ((j + 1) >> 1) & 1, err)))
                            break;
                        tc_fence_after();
                        issue_qk(tmem + kColS + x * kFa, sbase + kOffQ + x * kTileBytes,
                                 sbase + kOffK + b1 * kTileBytes);
                        mma_commit(&hd->s_full[x]);
                        if (x == nh - 1) mma_commit(&hd->kv_empty[b1]);
                    }
                }
            }
            mma_commit(&hd->done);
            fa_wait(&hd->done, 0, err);
        }
        __syncwarp();
    } else if (ok && (warp - 2) / kFaWarpsPerHead < nh) {
        // ------------------------------------------------------------ softmax
        const int x = (warp - 2) / kFaWarpsPerHead;  // head h0 + x of the CTA
        const int q = warp & 3;                      // tensor-memory lane quarter
        const int r = q * 32 + lane;                 // query row of the tile
        const int qpos = p0 + r;
        const int last = p0 + kFa - 1;               // the tile's last query position
        const float sl2 = 1.4426950408889634f / sqrtf((float)kHeadDimFa);
        const uint32_t lane_base = (uint32_t)(q * 32) << 16;
        const uint32_t s_col = tmem + lane_base + kColS + (uint32_t)x * kFa;
        const uint32_t o_col = tmem + lane_base + kColO + (uint32_t)x * kFa;
        // m: the exponent base of the row (scaled scores), which may trail the
        // row maximum by up to kFaRescale; l: the row sum relative to it
        float m = -INFINITY, l = 0.f;
        bool good = true;
        for (int j = 0; j < n_kv; ++j) {
            const int b = j & 1;
            // a value tile that runs past the tile's last query: head A's
            // thread r zeroes its row r past `last` before P_j V_j reads it
            // (P is zero there, but those cache rows may hold anything)
            const bool clip = j * kFa + kFa - 1 > last;
            if (x == 0 && clip) {
                good = good && fa_wait(&hd->v_full[b], (j >> 1) & 1, err);
                if (j * kFa + r > last) {
                    unsigned char *vt = smem + kOffV + b * kTileBytes;
#pragma unroll
                    for (int c = 0; c < kFa; c += 8)
                        *reinterpret_cast<uint4 *>(vt + (c >> 6) * kHalfBytes +
                                                   swizzle_offset((uint32_t)r, (uint32_t)(c & 63))) =
                            make_uint4(0u, 0u, 0u, 0u);
                }
            }
            // the row's 128 scores of S_j
            good = good && fa_wait(&hd->s_full[x], j & 1, err);
            tc_fence_after();
            float v[kFa];
#pragma unroll
            for (int c = 0; c < kFa; c += 32)
                tmem_ld32(s_col + c, *reinterpret_cast<float(*)[32]>(&v[c]));
            tmem_ld_wait();
            const bool full = j * kFa + kFa - 1 <= p0;  // no position of the tile is masked
            float hm4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
            if (full) {
#pragma unroll
                for (int i = 0; i < kFa; ++i) hm4[i & 3] = fmaxf(hm4[i & 3], v[i]);
            } else {
#pragma unroll
                for (int i = 0; i < kFa; ++i)
                    if (j * kFa + i <= qpos) hm4[i & 3] = fmaxf(hm4[i & 3], v[i]);
            }
            // finite: position 128j <= qpos for every row of the tile
            const float mrow = fmaxf(fmaxf(hm4[0], hm4[1]), fmaxf(hm4[2], hm4[3])) * sl2;
            const bool bump = mrow > m + kFaRescale;
            const float corr = bump ? exp2f(m - mrow) : 1.f;  // 0 on the first tile
            if (bump) m = mrow;
            // P_j in bf16 pairs over the first 64 columns of S_j, 64 positions
            // at a time; the row sum takes the probabilities as stored, so the
            // weights P V is normalised by sum to exactly one
            const float2 sl2x2 = make_float2(sl2, sl2), nm2 = make_float2(-m, -m);
            float2 sum2[2] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll
            for (int half = 0; half < 2; ++half) {
                uint32_t pw[32];
#pragma unroll
                for (int i = 0; i < 64; i += 2) {
                    const int c = half * 64 + i;
                    const float2 e = __ffma2_rn(make_float2(v[c], v[c + 1]), sl2x2, nm2);
                    float pa = fast_exp2(e.x);
                    float pb = fast_exp2(e.y);
                    if (!full) {
                        if (j * kFa + c > qpos) pa = 0.f;
                        if (j * kFa + c + 1 > qpos) pb = 0.f;
                    }
                    const __nv_bfloat162 p2 = __floats2bfloat162_rn(pa, pb);
                    sum2[(i >> 1) & 1] = __fadd2_rn(sum2[(i >> 1) & 1], __bfloat1622float2(p2));
                    pw[i >> 1] = *reinterpret_cast<const uint32_t *>(&p2);
                }
                tmem_st32(s_col + half * 32, pw);
            }
            // a new base rescales O (the scores are consumed by now): P_{j-1}
            // V_{j-1} finished before S_j was issued, and P_j V_j waits for
            // this warp's arrival; the whole warp loads and stores (rows
            // without a new base scale by 1)
            if (j >= 1 && __any_sync(0xffffffffu, bump) && __all_sync(0xffffffffu, good)) {
#pragma unroll 1
                for (int c = 0; c < kFa; c += 32) {
                    float ov[32];
                    uint32_t ow[32];
                    tmem_ld32(o_col + c, ov);
                    tmem_ld_wait();
#pragma unroll
                    for (int i = 0; i < 32; ++i) ow[i] = __float_as_uint(ov[i] * corr);
                    tmem_st32(o_col + c, ow);
                }
            }
            tmem_st_wait();
            if (x == 0 && clip) fence_proxy_async_smem();  // the zeroed value rows
            tc_fence_before();                             // P_j and a rescaled O
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->p_ready[x]);
            l = l * corr + ((sum2[0].x + sum2[0].y) + (sum2[1].x + sum2[1].y));
        }
        bool fin = good && n_kv > 0;
        if (fin) fin = fa_wait(&hd->o_full[x], (n_kv - 1) & 1, err);
        if (__all_sync(0xffffffffu, fin)) {
            tc_fence_after();
            const float inv = l > 0.f ? 1.f / l : 0.f;
            bf16 *dst = ctx + ((size_t)(t0 + r) * Hq + h0 + x) * 128;
#pragma unroll
            for (int c = 0; c < kFa; c += 32) {
                float vv[32];
                tmem_ld32(o_col + c, vv);
                tmem_ld_wait();
#pragma unroll
                for (int i = 0; i < 32; i += 8) {
                    uint32_t w[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const __nv_bfloat162 p2 =
                            __floats2bfloat162_rn(vv[i + 2 * e] * inv, vv[i + 2 * e + 1] * inv);
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
    // a CTA per (pair of query heads of one key/value head, tile)
    const int pairs = (Hq / Hkv + 1) / 2;
    LaunchScope ls("attention_tc", st);
    return launch_pdl(kern, dim3(Hkv * pairs, (T + kFa - 1) / kFa), dim3(kFaThreads), kFaSmem, st,
                      args);
}

}  // namespace moe
