// Decode attention on the tcgen05 tensor cores: tokens that attend to a key/
// value cache one by one (a decode step: one token per sequence).
//
// A decode token's grouped-query attention is small in the query dimension
// (the G <= 8 query heads that share one key/value head) and long in the
// position dimension, so the positions are the MMA's M and the heads its N:
//
//   S^T = K_j Q^T       M = 128 positions, N = 16 (the G heads, zero-
//                       padded), K = 128 dims; K_j and Q both K-major
//   O^T += V_j^T P_j^T  M = 128 dims, N = 16 heads, K = 128 positions; V_j
//                       as it lies in the cache (dims contiguous: an
//                       MN-major A operand), P_j K-major in shared memory
//
// with S^T and O^T in tensor memory (lane = position, resp. dim; column =
// head).  One CTA per (position split c, token t, key/value head g); the
// splits of (t, g) share the position tiles of t's sequence (128 positions
// each): split c takes tiles c, c + n_split, c + 2 n_split first, then one
// at a time from a counter in the cluster's CTA 0, so a split whose share
// of the memory bandwidth runs ahead takes more tiles.  A CTA's j-th tile
// goes to its stages in order and is published in a ring of tile indices
// (-1 after its last):
//
//   warp 0      TMA: the group's bf16 query rows once, then key and value
//               tiles into three-stage rings (each 32 KB: two boxes of 64
//               dims with the 128-byte swizzle), the first three before the
//               block-wide barrier of the set-up;
//   warp 1      tensor memory (S^T twice, O^T: 48 of 64 columns) and the
//               MMAs: S_{j+1} is issued as soon as its key tile has landed
//               and the softmax has read S_{j-1}, O += P_j V_j once P_j is
//               written;
//   warps 2-5   softmax, one thread per position of the tile (its tensor-
//               memory lane): the tile maximum of every head across the
//               128 positions (a warp maximum, then the four warps' through
//               shared memory), the base-2 exponent of the 1/sqrt(128)-
//               scaled scores against a per-head base that moves only when
//               the maximum passes it by more than 8 (then O^T is rescaled
//               in tensor memory, each thread its dim's row), bf16
//               probabilities written into P_j (rows = heads, positions
//               contiguous, 128-byte swizzle), rows of V_j past the
//               sequence's last position zeroed (0 * NaN is NaN; those cache
//               rows may hold anything).
//
// The end: each thread owns dim r of O^T; per head the row sums of the four
// warps are added.  A single split writes ctx.  Several splits of one
// (token, key/value head) are the CTAs of one thread-block cluster (at most
// 8), and CTA c owns the heads h = c, c + n_split, ...: every CTA stores its
// (base, sum) and O^T row of each head straight into the owner's shared
// memory with asynchronous stores that count their bytes on the owner's
// merge barrier (the owner expects all splits' bytes from its start), so
// no sender waits for its stores or fences them; the owner's acquire wait
// on the barrier sees every split's partials, then it combines its heads
// and writes their ctx.  (The stores wait until every CTA of the cluster
// has initialised its barriers: each arrives on the cluster barrier at its
// start and waits on it before storing, by when the wait is long
// satisfied.)
//
// Numerics as the prefill flash attention: bf16 queries and probabilities,
// fp32 scores and accumulation; the row sum takes the probabilities as
// stored.  Every wait is bounded (ptx.cuh); once one gives up the thread
// skips the later waits and the kernel ends.
#include <math.h>

#include <algorithm>

#include "tc.cuh"

namespace moe {
namespace {

using namespace tc;

constexpr int kDecPos = 128;   // positions per key/value tile: the MMA's M
constexpr int kDecN = 16;      // the MMA's N: the group's query heads, zero-padded
constexpr int kDecMaxG = 8;    // query heads per key/value head
constexpr int kDecThreads = 6 * 32;
constexpr int kDecStages = 3;     // key and value tiles in flight
constexpr int kDecMaxSplit = 8;   // splits of one (token, key/value head): a portable cluster
// the position tiles of a CTA are published in a ring: the producer
// publishes its tile j once S_{j-3} has been computed (after the softmax
// took S_{j-5}, so after it read tile j-5), so a slot is rewritten long
// after both its readers (issuer, softmax) took it
constexpr int kDecRing = 8;
constexpr uint32_t kDecHalf = kDecPos * 128;  // one 64-dim box of a key/value tile: 16 KB
constexpr uint32_t kDecTile = 2 * kDecHalf;   // 32 KB
constexpr uint32_t kDecNHalf = kDecN * 128;   // 16 rows x 64 elements: 2 KB
constexpr uint32_t kDecQ = 2 * kDecNHalf;     // query rows, 128 dims
constexpr uint32_t kDecP = 2 * kDecNHalf;     // probabilities, 128 positions
// shared memory (1024-byte aligned): K[3], V[3], Q, P[2], the O^T rows the
// splits store for the heads this CTA merges, header
constexpr uint32_t kDecOffK = 0;
constexpr uint32_t kDecOffV = kDecOffK + kDecStages * kDecTile;
constexpr uint32_t kDecOffQ = kDecOffV + kDecStages * kDecTile;
constexpr uint32_t kDecOffP = kDecOffQ + kDecQ;
constexpr uint32_t kDecOffX = kDecOffP + 2 * kDecP;
// [heads this CTA owns <= ceil(8 / n_split)][n_split][128] floats: at most
// 14 rows (8 heads over 7 splits)
constexpr uint32_t kDecXBytes = 14 * 128 * 4;
constexpr uint32_t kDecOffHdr = kDecOffX + kDecXBytes;
constexpr uint32_t kDecHdrBytes = 2048;
constexpr size_t kDecSmem = 1024 + kDecOffHdr + kDecHdrBytes;
static_assert(kDecSmem <= 227 * 1024, "shared memory");
// kind::f16: bf16 A and B, fp32 D, M = 128, N = 16; A and B K-major
constexpr uint32_t kDecIdescQK = (1u << 4) | (1u << 7) | (1u << 10) |
                                 ((uint32_t)(kDecN >> 3) << 17) | ((uint32_t)(kDecPos >> 4) << 24);
// the same with A MN-major (bit 15): O^T += V^T P^T with V as stored
constexpr uint32_t kDecIdescPV = kDecIdescQK | (1u << 15);
constexpr uint32_t kDecTmemCols = 64;
constexpr uint32_t kDecColS = 0, kDecColO = 2 * kDecN;
// base-2 distance the tile maximum may run ahead of a head's exponent base
constexpr float kDecRescale = 8.f;

struct DecHeader {
    uint64_t q_full;
    uint64_t k_full[kDecStages], k_empty[kDecStages];  // key tile j in stage j % 3
    uint64_t v_full[kDecStages], v_empty[kDecStages];  // value tile j in stage j % 3
    uint64_t s_full[2];              // S_j written (buffer j % 2)
    uint64_t s_empty[2];             // S_j read by the four softmax warps
    uint64_t p_ready[2];             // P_j written (four softmax warps)
    uint64_t p_empty[2];             // P_j V_j finished
    uint64_t t_full[kDecRing];       // tile index j of this CTA published (producer)
    uint64_t done;
    uint64_t merge_full;             // every split's partials stored here (their bytes)
    uint32_t tmem_base;
    uint32_t next_tile;              // the cluster's tile counter (in CTA 0)
    int tidx[kDecRing];              // position tile of this CTA's j-th tile, -1 past the last
    float red[2][4][kDecMaxG];  // the warps' tile maxima, by tile parity
    float lsum[4][kDecMaxG];    // the warps' row sums at the end
    alignas(8) float ml[kDecMaxG][kDecMaxSplit][2];  // (base, sum) of the owned heads, by split
};
static_assert(sizeof(DecHeader) <= kDecHdrBytes, "decode attention header");

// Waits spin on the non-blocking test (bounded by the wall-time limit of
// ptx.cuh): the pipeline is a chain of short steps, and a thread that
// suspends in try_wait resumes later than the phase completes.
__device__ __forceinline__ bool dec_test(uint64_t *bar, uint32_t parity) {
    uint32_t done;
    asm volatile(
        "{\n\t.reg .pred p;\n\tmbarrier.test_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(done)
        : "r"(ptx::smem_u32(bar)), "r"(parity)
        : "memory");
    return done != 0;
}

__device__ __forceinline__ bool dec_wait(uint64_t *bar, uint32_t parity, unsigned *err) {
    if (dec_test(bar, parity)) return true;
    const uint64_t t0 = ptx::globaltimer();
    for (uint32_t it = 1;; ++it) {
        if (dec_test(bar, parity)) return true;
        if ((it & 255u) == 0 && ptx::globaltimer() - t0 > ptx::kWaitLimitNs) {
            set_error(err, kErrTimeout);
            return false;
        }
    }
}

__device__ __forceinline__ float dec_exp2(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// 16 fp32 columns of this warp's 32 tensor-memory lanes.
__device__ __forceinline__ void tmem_ld16(uint32_t taddr, float (&v)[16]) {
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]),
          "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]),
          "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr)
        : "memory");
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

__device__ __forceinline__ void tmem_st16(uint32_t taddr, const float (&v)[16]) {
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x16.b32 [%0], "
        "{%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,%16};" ::"r"(taddr),
        "r"(__float_as_uint(v[0])), "r"(__float_as_uint(v[1])), "r"(__float_as_uint(v[2])),
        "r"(__float_as_uint(v[3])), "r"(__float_as_uint(v[4])), "r"(__float_as_uint(v[5])),
        "r"(__float_as_uint(v[6])), "r"(__float_as_uint(v[7])), "r"(__float_as_uint(v[8])),
        "r"(__float_as_uint(v[9])), "r"(__float_as_uint(v[10])), "r"(__float_as_uint(v[11])),
        "r"(__float_as_uint(v[12])), "r"(__float_as_uint(v[13])), "r"(__float_as_uint(v[14])),
        "r"(__float_as_uint(v[15]))
        : "memory");
    asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory");
}

// Asynchronous stores into CTA `rank`'s shared memory that count their bytes
// on that CTA's barrier `bar` (complete-tx, released at cluster scope): the
// receiver's acquire wait on `bar` sees them, and the sender waits for
// nothing.
__device__ __forceinline__ void st_async_f32(float *p, uint32_t rank, uint64_t *bar, float v) {
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.f32 [%0], %1, [%2];" ::"r"(
            ptx::map_rank(ptx::smem_u32(p), rank)),
        "f"(v), "r"(ptx::map_rank(ptx::smem_u32(bar), rank))
        : "memory");
}

__device__ __forceinline__ void st_async_v2f32(float *p, uint32_t rank, uint64_t *bar, float a,
                                               float b) {
    asm volatile(
        "st.async.shared::cluster.mbarrier::complete_tx::bytes.v2.f32 [%0], {%1, %2}, [%3];" ::"r"(
            ptx::map_rank(ptx::smem_u32(p), rank)),
        "f"(a), "f"(b), "r"(ptx::map_rank(ptx::smem_u32(bar), rank))
        : "memory");
}

__device__ __forceinline__ void cluster_arrive_release() {
    asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}
// Take the next value of a counter in a cluster CTA's shared memory.
__device__ __forceinline__ uint32_t dec_take(uint32_t cluster_addr) {
    uint32_t old;
    asm volatile("atom.shared::cluster.add.u32 %0, [%1], 1;" : "=r"(old) : "r"(cluster_addr)
                 : "memory");
    return old;
}
__device__ __forceinline__ void cluster_wait() {
    asm volatile("barrier.cluster.wait.aligned;" ::: "memory");
}

// MN-major operand written by TMA with the 128-byte swizzle (the value tile
// as A = V^T): a 128-byte row holds 64 consecutive dims of one position, 8
// positions make a 1024-byte atom (stride offset), the next 64 dims are the
// second box, 16 KB on (leading offset).
__device__ __forceinline__ uint64_t dec_desc_mn(uint32_t saddr) {
    return (uint64_t)((saddr & 0x3FFFFu) >> 4) | ((uint64_t)(kDecHalf >> 4) << 16) |
           ((uint64_t)(1024 >> 4) << 32) | ((uint64_t)1 << 46) | ((uint64_t)2 << 61);
}

// S^T = K Q^T: 128 positions x 16 heads over 128 dims.
__device__ __forceinline__ void dec_issue_qk(uint32_t d_tmem, uint32_t k_smem, uint32_t q_smem) {
#pragma unroll
    for (int half = 0; half < 2; ++half) {
        const uint64_t ad = smem_desc(k_smem + half * kDecHalf);
        const uint64_t bd = smem_desc(q_smem + half * kDecNHalf);
#pragma unroll
        for (int kk = 0; kk < 4; ++kk)
            mma_bf16(d_tmem, ad + 2 * kk, bd + 2 * kk, kDecIdescQK, (half | kk) != 0 ? 1u : 0u);
    }
}

// O^T (+)= V^T P^T: 128 dims x 16 heads over 128 positions, 16 a step.
__device__ __forceinline__ void dec_issue_pv(uint32_t d_tmem, uint32_t v_smem, uint32_t p_smem,
                                             bool accumulate) {
#pragma unroll
    for (int ks = 0; ks < 8; ++ks) {
        const uint64_t ad = dec_desc_mn(v_smem + ks * 16 * 128);
        const uint64_t bd = smem_desc(p_smem + (ks >> 2) * kDecNHalf) + 2 * (ks & 3);
        mma_bf16(d_tmem, ad, bd, kDecIdescPV, (accumulate || ks != 0) ? 1u : 0u);
    }
}

template <int G>
__global__ void __launch_bounds__(kDecThreads, 1)
k_attn_decode_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                 const __grid_constant__ CUtensorMap tmV, int Hq, int Hkv, int n_seq, int L,
                 int n_split, const int32_t *__restrict__ seq, const int32_t *__restrict__ pos,
                 bf16 *__restrict__ ctx, unsigned *err) {
    static_assert(G >= 1 && G <= kDecMaxG, "query heads per key/value head");
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    DecHeader *hd = reinterpret_cast<DecHeader *>(smem + kDecOffHdr);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int s = blockIdx.x, tg = blockIdx.y;
    const int t = tg / Hkv, g = tg - t * Hkv;
    // the token's sequence and position are inputs of the call, complete
    // before it in stream order (no kernel of the library writes them): read
    // first, their latency behind the set-up
    const int sq = seq[t], p = pos[t];

    const int c = s;  // rank in the cluster (the splits of one pair)

    if (threadIdx.x == 0) {
        ptx::mbar_init(&hd->q_full, 1);
        for (int b = 0; b < kDecStages; ++b) {
            ptx::mbar_init(&hd->k_full[b], 1);
            ptx::mbar_init(&hd->k_empty[b], 1);
            ptx::mbar_init(&hd->v_full[b], 1);
            ptx::mbar_init(&hd->v_empty[b], 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&hd->s_full[b], 1);
            ptx::mbar_init(&hd->s_empty[b], 4);
            ptx::mbar_init(&hd->p_ready[b], 4);
            ptx::mbar_init(&hd->p_empty[b], 1);
        }
        for (int b = 0; b < kDecRing; ++b) ptx::mbar_init(&hd->t_full[b], 1);
        ptx::mbar_init(&hd->done, 1);
        ptx::mbar_init(&hd->merge_full, 1);
        hd->next_tile = 0u;
        if (n_split > 1) {
            // the bytes every split stores here: an O^T row and (base, sum)
            // for each head this CTA merges
            const int owned = c < G ? (G - 1 - c) / n_split + 1 : 0;
            ptx::mbar_arrive_expect_tx(&hd->merge_full,
                                       (uint32_t)(n_split * owned * (kDecPos * 4 + 8)));
        }
        ptx::fence_barrier_init();
        ptx::prefetch_tmap(&tmQ);
        ptx::prefetch_tmap(&tmK);
        ptx::prefetch_tmap(&tmV);
    }
    if (n_split > 1) {
        // this CTA's barriers and tile counter are initialised: the
        // cluster's other CTAs may use them once they pass the matching wait
        // (the arrival releases thread 0's stores at cluster scope)
        __syncthreads();
        cluster_arrive_release();
    }
    if (warp == 1) tmem_alloc(&hd->tmem_base, kDecTmemCols);
    // the output projection may launch now: it streams its weights into the
    // SMs this grid leaves free while the attention runs
    ptx::launch_dependents();
    ptx::grid_dependency_wait();  // queries and caches come from the previous kernel
    const bool ok = sq >= 0 && sq < n_seq && p >= 0 && p < L;
    // the position tiles of the sequence: the splits share them, the first
    // kDecStages of each split fixed (tile c + i n_split for split c), the
    // rest taken one by one from a counter in CTA 0 of the cluster by
    // whichever split frees a stage first (the splits' shares of the memory
    // bandwidth differ); only the last tile of the sequence is partial
    const int n = ok ? p + 1 : 0;
    const int n_all = (n + kDecPos - 1) / kDecPos;
    const int row0 = (sq * Hkv + g) * L;
    int n_first = 0;  // fixed tiles of this split that exist
    for (int i = 0; i < kDecStages; ++i) n_first += c + i * n_split < n_all ? 1 : 0;
    // the producer (thread 0, which initialised the barriers) sends the
    // query rows and the fixed tiles before the block-wide barrier: their
    // stages are empty yet
    if (threadIdx.x == 0) {
        if (n_first > 0) {
            const uint64_t pol_kv = ptx::policy_evict_first();  // read once
            ptx::mbar_arrive_expect_tx(&hd->q_full, kDecQ);
            for (int half = 0; half < 2; ++half)
                ptx::tma_load_2d(smem + kDecOffQ + half * kDecNHalf, &tmQ, half * 64,
                                 t * Hq + g * G, &hd->q_full, ptx::policy_evict_normal());
            for (int j = 0; j < n_first; ++j) {
                const int row = row0 + (c + j * n_split) * kDecPos;
                ptx::mbar_arrive_expect_tx(&hd->k_full[j], kDecTile);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kDecOffK + j * kDecTile + half * kDecHalf, &tmK,
                                     half * 64, row, &hd->k_full[j], pol_kv);
                ptx::mbar_arrive_expect_tx(&hd->v_full[j], kDecTile);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kDecOffV + j * kDecTile + half * kDecHalf, &tmV,
                                     half * 64, row, &hd->v_full[j], pol_kv);
                hd->tidx[j] = c + j * n_split;
                ptx::mbar_arrive(&hd->t_full[j]);
            }
        }
        if (n_first < kDecStages) {
            // no tile past these: the end is published now
            hd->tidx[n_first] = -1;
            ptx::mbar_arrive(&hd->t_full[n_first]);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = hd->tmem_base;
    const uint32_t sbase = ptx::smem_u32(smem);

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        // (CTA 0's counter is initialised before the first take)
        if (n_split > 1) cluster_wait();
        if (lane == 0 && n_first == kDecStages) {
            const uint64_t pol_kv = ptx::policy_evict_first();
            const uint32_t counter = ptx::map_rank(ptx::smem_u32(&hd->next_tile), 0u);
            // the next tile is taken one ahead: its counter round trip runs
            // while the stage it goes to frees
            int taken = 0;  // (a single split counts alone)
            auto take = [&]() -> int {
                return kDecStages * n_split +
                       (n_split > 1 ? (int)dec_take(counter) : taken++);
            };
            int nxt = take();
            int k_issued = kDecStages, v_issued = kDecStages;
            for (int j = kDecStages;; ++j) {
                const int tile = nxt;
                if (tile >= n_all) {
                    hd->tidx[j % kDecRing] = -1;
                    ptx::mbar_arrive(&hd->t_full[j % kDecRing]);
                    break;
                }
                nxt = take();
                const int b = j % kDecStages;
                const uint32_t ph = ((j / kDecStages) & 1) ^ 1;
                const int row = row0 + tile * kDecPos;
                if (!dec_wait(&hd->k_empty[b], ph, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->k_full[b], kDecTile);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kDecOffK + b * kDecTile + half * kDecHalf, &tmK,
                                     half * 64, row, &hd->k_full[b], pol_kv);
                k_issued = j + 1;
                hd->tidx[j % kDecRing] = tile;
                ptx::mbar_arrive(&hd->t_full[j % kDecRing]);
                if (!dec_wait(&hd->v_empty[b], ph, err)) break;
                ptx::mbar_arrive_expect_tx(&hd->v_full[b], kDecTile);
                for (int half = 0; half < 2; ++half)
                    ptx::tma_load_2d(smem + kDecOffV + b * kDecTile + half * kDecHalf, &tmV,
                                     half * 64, row, &hd->v_full[b], pol_kv);
                v_issued = j + 1;
            }
            // copies still in flight land before the block can exit
            dec_wait(&hd->q_full, 0, err);
            for (int j = std::max(0, k_issued - kDecStages); j < k_issued; ++j)
                dec_wait(&hd->k_full[j % kDecStages], (j / kDecStages) & 1, err);
            for (int j = std::max(0, v_issued - kDecStages); j < v_issued; ++j)
                dec_wait(&hd->v_full[j % kDecStages], (j / kDecStages) & 1, err);
        } else if (lane == 0 && n_first > 0) {
            dec_wait(&hd->q_full, 0, err);
            for (int j = 0; j < n_first; ++j) {
                dec_wait(&hd->k_full[j], 0, err);
                dec_wait(&hd->v_full[j], 0, err);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0 && n_first > 0) {
            bool good = dec_wait(&hd->q_full, 0, err) && dec_wait(&hd->k_full[0], 0, err);
            if (good) {
                tc_fence_after();
                dec_issue_qk(tmem + kDecColS, sbase + kDecOffK, sbase + kDecOffQ);
                mma_commit(&hd->s_full[0]);
                mma_commit(&hd->k_empty[0]);
            }
            for (int j = 0; good; ++j) {
                // is there a tile j + 1 (published by the producer)?
                const int r1 = (j + 1) % kDecRing;
                if (!(good = dec_wait(&hd->t_full[r1], ((j + 1) / kDecRing) & 1, err))) break;
                const bool more = hd->tidx[r1] >= 0;
                if (more) {
                    // S_{j+1} into the buffer of S_{j-1}, once the softmax has read it
                    const int sb1 = (j + 1) & 1, kb1 = (j + 1) % kDecStages;
                    good = dec_wait(&hd->k_full[kb1], ((j + 1) / kDecStages) & 1, err) &&
                           (j < 1 || dec_wait(&hd->s_empty[sb1], ((j - 1) >> 1) & 1, err));
                    if (!good) break;
                    tc_fence_after();
                    dec_issue_qk(tmem + kDecColS + sb1 * kDecN, sbase + kDecOffK + kb1 * kDecTile,
                                 sbase + kDecOffQ);
                    mma_commit(&hd->s_full[sb1]);
                    mma_commit(&hd->k_empty[kb1]);
                }
                const int pb = j & 1, vb = j % kDecStages;
                good = dec_wait(&hd->v_full[vb], (j / kDecStages) & 1, err) &&
                       dec_wait(&hd->p_ready[pb], (j >> 1) & 1, err);
                if (!good) break;
                tc_fence_after();
                dec_issue_pv(tmem + kDecColO, sbase + kDecOffV + vb * kDecTile,
                             sbase + kDecOffP + pb * kDecP, j != 0);
                mma_commit(&hd->p_empty[pb]);
                mma_commit(&hd->v_empty[vb]);
                if (!more) break;
            }
            mma_commit(&hd->done);
            dec_wait(&hd->done, 0, err);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ softmax
        {
            // probability rows G..15 of both buffers stay zero (the MMA's
            // padding heads; no thread writes them later, and each thread's
            // proxy fence before it releases P_0 covers its zeros)
            constexpr int kPadRow = G * 8;  // 16-byte chunks before row G of a half
            constexpr int kPad = 16 * 8 - kPadRow;
            for (int i = threadIdx.x - 64; i < 4 * kPad; i += 128) {
                uint4 *half = reinterpret_cast<uint4 *>(smem + kDecOffP) + (i / kPad) * (kDecNHalf / 16);
                half[kPadRow + i % kPad] = make_uint4(0u, 0u, 0u, 0u);
            }
        }
        // every CTA of the cluster has initialised its barriers before this
        // one's merge stores (waited here, long before they are needed)
        if (n_split > 1) cluster_wait();
        const int qd = warp & 3;       // tensor-memory lane quarter
        const int r = qd * 32 + lane;  // position of the tile; dim of O^T
        const uint32_t lane_base = (uint32_t)(qd * 32) << 16;
        const float sl2 = 1.4426950408889634f / sqrtf(128.f);
        float base[G], l[G];
#pragma unroll
        for (int h = 0; h < G; ++h) {
            base[h] = -INFINITY;
            l[h] = 0.f;
        }
        bool good = true;
        int had = 0;  // tiles this split has had
        for (int j = 0;; ++j) {
            const int b = j & 1;
            good = good && dec_wait(&hd->t_full[j % kDecRing], (j / kDecRing) & 1, err);
            // (lane 0's reading steers the warp: its loop stays converged)
            const int tile =
                __shfl_sync(0xffffffffu, good ? hd->tidx[j % kDecRing] : -1, 0);
            if (tile < 0) break;
            had = j + 1;
            const int pj = tile * kDecPos + r;
            const bool valid = pj < n;
            // (the load runs on every lane whatever its waits returned: it is
            // warp-collective; after a failed wait the values are not used)
            float v[16];
            good = good && dec_wait(&hd->s_full[b], (j >> 1) & 1, err);
            tc_fence_after();
            tmem_ld16(tmem + lane_base + kDecColS + b * kDecN, v);
            tmem_ld_wait();
            tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->s_empty[b]);
            // the tile maximum of every head (finite: the tile has a valid position)
            float x[G];
#pragma unroll
            for (int h = 0; h < G; ++h) {
                x[h] = valid ? v[h] * sl2 : -INFINITY;
                float m = x[h];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
                if (lane == 0) hd->red[b][qd][h] = m;
            }
            ptx::named_bar_sync(1, 128);
            float corr[G];
            bool bump_any = false;
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float tm = fmaxf(fmaxf(hd->red[b][0][h], hd->red[b][1][h]),
                                       fmaxf(hd->red[b][2][h], hd->red[b][3][h]));
                const bool bump = tm > base[h] + kDecRescale;
                corr[h] = bump ? exp2f(base[h] - tm) : 1.f;  // 0 on the first tile
                if (bump) base[h] = tm;
                bump_any |= bump;
            }
            // P_j into buffer b, free once P_{j-2} V_{j-2} has finished
            good = good && (j < 2 || dec_wait(&hd->p_empty[b], ((j - 2) >> 1) & 1, err));
            unsigned char *pb = smem + kDecOffP + b * kDecP + (r >> 6) * kDecNHalf;
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float pv = valid ? dec_exp2(x[h] - base[h]) : 0.f;
                const bf16 pq = __float2bfloat16_rn(pv);
                if (good)
                    *reinterpret_cast<bf16 *>(pb + swizzle_offset((uint32_t)h,
                                                                  (uint32_t)(r & 63))) = pq;
                l[h] = fmaf(l[h], corr[h], __bfloat162float(pq));
            }
            // a value tile that runs past the sequence's last position: its
            // rows there are zeroed before P_j V_j reads them
            if (tile * kDecPos + kDecPos > n) {
                const int vb = j % kDecStages;
                good = good && dec_wait(&hd->v_full[vb], (j / kDecStages) & 1, err);
                if (good && !valid) {
                    unsigned char *vt = smem + kDecOffV + vb * kDecTile;
#pragma unroll
                    for (int c = 0; c < 128; c += 8)
                        *reinterpret_cast<uint4 *>(
                            vt + (c >> 6) * kDecHalf +
                            swizzle_offset((uint32_t)r, (uint32_t)(c & 63))) =
                            make_uint4(0u, 0u, 0u, 0u);
                }
            }
            // a moved base rescales O^T (each thread its dim's row) once
            // P_{j-1} V_{j-1} has finished; P_j V_j waits for this warp
            if (j >= 1 && bump_any) {
                good = good && dec_wait(&hd->p_empty[(j - 1) & 1], ((j - 1) >> 1) & 1, err);
                if (__all_sync(0xffffffffu, good)) {
                    tc_fence_after();
                    float o[16];
                    tmem_ld16(tmem + lane_base + kDecColO, o);
                    tmem_ld_wait();
#pragma unroll
                    for (int h = 0; h < G; ++h) o[h] *= corr[h];
                    tmem_st16(tmem + lane_base + kDecColO, o);
                }
            }
            fence_proxy_async_smem();  // P_j and the zeroed value rows
            tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->p_ready[b]);
        }
        // the split's result: O^T row r (dim r) of every head, the row sums
        // of the four warps added in warp order
        bool fin = good && had > 0;
        if (fin) fin = dec_wait(&hd->p_empty[(had - 1) & 1], ((had - 1) >> 1) & 1, err);
        fin = __all_sync(0xffffffffu, fin);
#pragma unroll
        for (int h = 0; h < G; ++h) {
            const float ws = warp_sum(l[h]);
            if (lane == 0) hd->lsum[qd][h] = ws;
        }
        ptx::named_bar_sync(1, 128);
        float o[16];
#pragma unroll
        for (int h = 0; h < 16; ++h) o[h] = 0.f;
        if (fin) {
            tc_fence_after();
            tmem_ld16(tmem + lane_base + kDecColO, o);
            tmem_ld_wait();
        }
        if (n_split == 1) {
#pragma unroll
            for (int h = 0; h < G; ++h) {
                const float Ls = fin ? (hd->lsum[0][h] + hd->lsum[1][h]) +
                                           (hd->lsum[2][h] + hd->lsum[3][h])
                                     : 0.f;
                ctx[((size_t)t * Hq + g * G + h) * 128 + r] =
                    __float2bfloat16_rn(Ls > 0.f ? __fdividef(o[h], Ls) : 0.f);
            }
        } else {
            float *xo = reinterpret_cast<float *>(smem + kDecOffX);
#pragma unroll
            for (int h = 0; h < G; ++h) {
                // head h belongs to CTA h % n_split, row slot h / n_split;
                // the stores count their bytes on the owner's merge barrier
                const uint32_t owner = (uint32_t)(h % n_split);
                const int slot = h / n_split;
                st_async_f32(&xo[((size_t)slot * n_split + c) * 128 + r], owner, &hd->merge_full,
                             fin ? o[h] : 0.f);
                if (r == 0) {
                    const float Ls = fin ? (hd->lsum[0][h] + hd->lsum[1][h]) +
                                               (hd->lsum[2][h] + hd->lsum[3][h])
                                         : 0.f;
                    st_async_v2f32(&hd->ml[slot][c][0], owner, &hd->merge_full,
                                   fin ? base[h] : -INFINITY, Ls);
                }
            }
            // the heads this CTA owns (base 2: split weight 2^(base_s - M)),
            // once every split's bytes have landed
            const bool got = ptx::mbar_wait_cluster(&hd->merge_full, 0, err);
            // (unrolled to the bounds and predicated, so that the heads' and
            // the splits' loads go out together: n_split >= 2 leaves at most
            // (G + 1) / 2 heads to a CTA)
#pragma unroll
            for (int slot = 0; slot < (G + 1) / 2; ++slot) {
                const int h = (int)c + slot * n_split;
                if (!got || h >= G) continue;
                float bq[kDecMaxSplit], M = -INFINITY;
#pragma unroll
                for (int q = 0; q < kDecMaxSplit; ++q) {
                    bq[q] = q < n_split ? hd->ml[slot][q][0] : -INFINITY;
                    M = fmaxf(M, bq[q]);
                }
                float A = 0.f, Ls = 0.f;
                if (M != -INFINITY) {
#pragma unroll
                    for (int q = 0; q < kDecMaxSplit; ++q) {
                        if (q < n_split) {
                            const float w = dec_exp2(bq[q] - M);
                            Ls = fmaf(w, hd->ml[slot][q][1], Ls);
                            A = fmaf(w, xo[(slot * n_split + q) * 128 + r], A);
                        }
                    }
                }
                // (Ls is a sum of probabilities of at most 2^8 each: far
                // inside the fast division's range)
                ctx[((size_t)t * Hq + g * G + h) * 128 + r] =
                    __float2bfloat16_rn(Ls > 0.f ? __fdividef(A, Ls) : 0.f);
            }
        }
    }
    // (the aligned wait of every thread: producer and softmax warps waited
    // at their start)
    if (n_split > 1 && warp == 1) cluster_wait();
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, kDecTmemCols);
}

}  // namespace

bool attn_decode_tc_ok() { return encode_fn() != nullptr; }

int attn_decode_tc_splits(int T, int Hkv, int max_len) {
    // one wave of one-CTA-per-SM blocks, at least one position tile a
    // split, at most a portable cluster of splits
    const int tg = std::max(1, T * Hkv);
    int ns = std::max(1, device_info().sm_count / tg);
    ns = std::min(ns, (max_len + kDecPos - 1) / kDecPos);
    return std::max(1, std::min(ns, kDecMaxSplit));
}

cudaError_t launch_attn_decode_tc(int T, int Hq, int Hkv, int n_seq, int L, int n_split,
                                  const int32_t *seq, const int32_t *pos, const void *q16,
                                  const void *k_cache, const void *v_cache, void *ctx,
                                  cudaStream_t st) {
    const int G = Hq / Hkv;
    if (G < 1 || G > kDecMaxG || G * Hkv != Hq || n_split < 1 || n_split > kDecMaxSplit)
        return cudaErrorInvalidValue;
    CUtensorMap mq, mk, mv;
    const uint64_t rows = (uint64_t)n_seq * Hkv * L;
    if (!make_map(&mq, q16, (uint64_t)T * Hq, 128, kDecN) ||
        !make_map(&mk, k_cache, rows, 128, kDecPos) || !make_map(&mv, v_cache, rows, 128, kDecPos))
        return cudaErrorInvalidValue;
    const void *kern = nullptr;
    switch (G) {
        case 1: kern = (const void *)k_attn_decode_tc<1>; break;
        case 2: kern = (const void *)k_attn_decode_tc<2>; break;
        case 3: kern = (const void *)k_attn_decode_tc<3>; break;
        case 4: kern = (const void *)k_attn_decode_tc<4>; break;
        case 5: kern = (const void *)k_attn_decode_tc<5>; break;
        case 6: kern = (const void *)k_attn_decode_tc<6>; break;
        case 7: kern = (const void *)k_attn_decode_tc<7>; break;
        default: kern = (const void *)k_attn_decode_tc<8>; break;
    }
    cudaError_t e =
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kDecSmem);
    if (e != cudaSuccess) return e;
    unsigned *err = device_info().err;
    bf16 *cp = static_cast<bf16 *>(ctx);
    int Hqv = Hq, Hkvv = Hkv, ns = n_seq, Lv = L, nsp = n_split;
    void *args[] = {&mq, &mk, &mv, &Hqv, &Hkvv, &ns, &Lv, &nsp, &seq, &pos, &cp, &err};
    // the splits of a (token, key/value head) form one cluster
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(n_split, T * Hkv);
    cfg.blockDim = dim3(kDecThreads);
    cfg.dynamicSmemBytes = kDecSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = n_split;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    LaunchScope ls("attention_decode_tc", st);
    return cudaLaunchKernelExC(&cfg, kern, args);
}

}  // namespace moe
