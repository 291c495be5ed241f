// Grouped expert GEMMs for prefill with the expert weights as the MMA's M
// operand and the sorted slots as N: tcgen05, bf16 operands, fp32
// accumulators in tensor memory, on one SM per tile (CG = 1) or on a CTA
// pair that shares every MMA (CG = 2, cta_group::2).
//
// Table 1 notes (d),(e) of arxiv 2506.23635: every expert is three
// D_embed x D_ffn matrices.  With the slots sorted by expert (moe_dispatch)
// the expert FFN is two grouped GEMMs with a variable number of slots per
// expert:
//
//   UP   (GLU):  h[j, f] = SiLU(x_j . W1[e,f,:]) * (x_j . V1[e,f,:])   -> bf16
//   DOWN:        y[j, d] = h[j, :] . W2[e,d,:]                          -> fp32
//
// A unit of work is (expert e, weight tile, slot tile).
//  * Weight tile: 128 A rows per CTA.  UP: 64 rows of W1 and the same 64
//    rows of V1 (one 3-D copy over the two tensors when their distance
//    allows it, else two copies), so tensor-memory lanes 0-63 hold one of
//    a = x.W1, b = x.V1 and lanes 64-127 the other, for the same f; DOWN:
//    128 rows of W2.  A pair covers twice that (the odd CTA the next 64 f /
//    128 d).
//  * Slot tile: the n_e slots of expert e are cut into ceil(n_e / 256)
//    near-equal runs; each run is the MMA's N, rounded up to 16 (32 for a
//    pair, whose CTAs hold N/2 slots each).  N is a field of the instruction
//    descriptor, set per tile, so a ragged expert wastes at most 15 (31)
//    columns per run rather than up to 127 rows of a fixed 128-slot tile.
// Units are numbered expert by expert, weight tile outer and slot tile inner
// (units running at the same time share weight tiles in L2); CTA (pair) b of
// G takes units b, b+G, ... in full rounds, and a piece of one of the last
// round's units (wm_item).
//
// Per CTA, 6 warps:
//   warp 0     TMA producer (one lane): the A tile and the run's slot rows
//              (N, or N/2 per CTA of a pair, as one box: a tensor map per box
//              height) into a ring of stages -- a copy instruction costs more
//              than its bytes: two per stage ran 1.2-1.3x faster than one per
//              16-128-row piece;
//              in a pair both CTAs' copies complete on the even CTA's
//              barrier of the stage (cta_group::2 copies), which expects the
//              bytes of both;
//   warp 1     tensor-memory allocation; one lane of the even CTA (or of
//              the only CTA) issues the MMAs;
//   warps 2-5  epilogue: tcgen05.ld of their 32 lanes; UP exchanges half of
//              a and b with the partner warp through shared memory (warps of
//              lanes 0-31 and 64-95, 32-63 and 96-127) and writes bf16 h,
//              DOWN writes fp32 y.
// A pair's MMAs free a stage in both CTAs and hand a finished accumulator to
// both epilogues (multicast commit); both epilogues release it to the even
// CTA.  (Relaying "stage landed" from a thread of the odd CTA instead took
// 2.3x longer per stage.)  Every mbarrier wait is bounded (ptx.cuh); an epilogue warp whose
// wait gave up keeps stepping through its named barriers without loading, so
// its partner never waits on it.
#include <cuda.h>
#include <cudaTypedefs.h>

#include <stdlib.h>

#include <mutex>

#include "tc.cuh"

namespace moe {
namespace {

using namespace tc;

constexpr int kWmBK = 64;          // reduction columns per stage (128 B rows)
constexpr int kWmMaxN = 256;       // slots per tile (the MMA's N)
constexpr int kWmThreads = 192;
constexpr int kWmMaxStages = 8;
constexpr size_t kWmHeaderBytes = 2048;
constexpr uint32_t kWmTmemCols = 512;  // two 256-column accumulators

enum WmMode { kWmUp = 0, kWmDown = 1 };

template <int MODE, int CG>
struct WmCfg {
    static constexpr uint32_t kStageA = 128 * kWmBK * 2;           // 16 KB
    static constexpr int kRowsB = kWmMaxN / CG;                    // slot rows per CTA
    static constexpr uint32_t kStageB = kRowsB * kWmBK * 2;        // 32 / 16 KB
    static constexpr uint32_t kStageBytes = kStageA + kStageB;
    static constexpr int kStages = CG == 1 ? 4 : 6;
    static constexpr int kOutPerCta = MODE == kWmUp ? 64 : 128;    // f or d values per CTA
    static constexpr uint32_t kXchgBytes = MODE == kWmUp ? 16384 : 0;
    static constexpr size_t kSmem =
        1024 /*align slack*/ + kStages * kStageBytes + kXchgBytes + kWmHeaderBytes;
    // kind::f16: bf16 A and B, fp32 D, both K-major, M = 128 per CTA; the
    // N field (bits 17-22, N >> 3) is added per tile
    static constexpr uint32_t kIdescBase =
        (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)((128 * CG) >> 4) << 24);
    static constexpr int kGran = 16 * CG;
    static_assert(kStages <= kWmMaxStages, "stages");
    static_assert(kStageBytes % 1024 == 0, "stages stay 1024-byte aligned");
    static_assert(kSmem <= 227 * 1024, "shared memory");
};

// The slot rows [S, Kdim] with box heights 16, 32, ..., 256 rows: map i
// loads 16 (i + 1) rows.  A pair uses the first 8.
struct SlotMaps {
    CUtensorMap m[16];
};

struct WmHeader {
    uint64_t full[kWmMaxStages];
    uint64_t empty[kWmMaxStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t done;
    uint32_t tmem_base;
    int tprefix[257];  // unit prefix over experts
};
static_assert(sizeof(WmHeader) <= kWmHeaderBytes, "header");

// tprefix[e] = sum over earlier experts of n_wt * ceil(n_e / 256).
__device__ void wm_prefix(const int32_t *offsets, int E, int S, int nwt, int *tprefix,
                          unsigned *err) {
    const int lane = threadIdx.x & 31;
    int run = 0;
    for (int base = 0; base < E; base += 32) {
        const int e = base + lane;
        int c = 0;
        if (e < E) {
            const int lo = offsets[e], hi = offsets[e + 1];
            if (lo < 0 || hi < lo || hi > S) set_error(err, kErrIndex);
            else c = ((hi - lo + kWmMaxN - 1) / kWmMaxN) * nwt;
        }
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (e < E) tprefix[e] = run + incl - c;
        run += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) tprefix[E] = run;
}

struct WmTile {
    int e, wt;  // expert, weight tile
    int s0;     // first sorted slot of the run
    int cnt;    // slots in the run (<= 256)
    int n;      // the MMA's N: cnt rounded up to the granule
};

__device__ __forceinline__ WmTile wm_tile(const int *tprefix, const int32_t *offsets, int E, int u,
                                          int gran) {
    WmTile t;
    t.e = chunk_expert(tprefix, E, u);
    const int r = u - tprefix[t.e];
    const int lo = offsets[t.e], n_e = offsets[t.e + 1] - lo;
    const int nst = (n_e + kWmMaxN - 1) / kWmMaxN;
    t.wt = r / nst;
    const int st = r - t.wt * nst;
    const int a = (int)((long long)st * n_e / nst);
    const int b = (int)((long long)(st + 1) * n_e / nst);
    t.s0 = lo + a;
    t.cnt = b - a;
    t.n = (t.cnt + gran - 1) / gran * gran;
    return t;
}

// The work of pair (or CTA) `pair` of n_pairs, item i: units pair,
// pair + n_pairs, ... in full rounds; the units of a last, partial round are
// cut into pieces along their slot run (granules of `gran` slots) so that
// the pairs the round would leave idle share them -- each piece keeps the
// whole reduction, so every output element is still computed once, by one
// MMA chain.  (768 down-projection units on 76 pairs of a 2048-token
// prefill: the eleventh round held 8 units, now 64 pieces of 32 slots.)
// False once the pair has no item i.  Items of zero width are skipped by
// the caller (cnt == 0).
__device__ __forceinline__ bool wm_item(const int *tprefix, const int32_t *offsets, int E,
                                        int n_units, int pair, int n_pairs, int i, int gran,
                                        WmTile &t) {
    const int rounds = n_units / n_pairs, full = rounds * n_pairs;
    if (i < rounds) {
        t = wm_tile(tprefix, offsets, E, pair + i * n_pairs, gran);
        return true;
    }
    const int rem = n_units - full;
    if (i > rounds || rem == 0) return false;
    // the tail round: pair -> (tail unit, piece)
    const int max_pieces = kWmMaxN / gran;
    const int P = max(1, min(max_pieces, n_pairs / rem));
    const int tu = pair / P, q = pair - tu * P;
    if (tu >= rem) return false;
    t = wm_tile(tprefix, offsets, E, full + tu, gran);
    const int g = t.n / gran;                      // granules of the run
    const int a = g * q / P, b = g * (q + 1) / P;  // this piece's granules
    const int s_a = a * gran;
    t.s0 += s_a;
    t.cnt = max(0, min(t.cnt, b * gran) - s_a);
    t.n = (b - a) * gran;
    if (t.n == 0) t.cnt = 0;
    return true;
}

// A tensor copy that completes on the mbarrier at cluster address `bar` --
// this CTA's or, in a CTA pair, the peer's (cta_group::2).
template <int CG>
__device__ __forceinline__ void wm_tma(void *dst_smem, const CUtensorMap *tmap, int32_t x, int32_t y,
                                       uint64_t *bar, uint32_t bar_cluster, uint64_t policy) {
    if (CG == 2)
        asm volatile(
            "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            ".cta_group::2.L2::cache_hint [%0], [%1, {%2, %3}], [%4], %5;" ::"r"(
                ptx::smem_u32(dst_smem)),
            "l"(tmap), "r"(x), "r"(y), "r"(bar_cluster), "l"(policy)
            : "memory");
    else
        ptx::tma_load_2d(dst_smem, tmap, x, y, bar, policy);
}

// The UP A tile as one 3-D copy: 64 rows of each of the two weight tensors
// (coordinate 0 of the third dimension first).
template <int CG>
__device__ __forceinline__ void wm_tma3(void *dst_smem, const CUtensorMap *tmap, int32_t x,
                                        int32_t y, uint64_t *bar, uint32_t bar_cluster,
                                        uint64_t policy) {
    if (CG == 2)
        asm volatile(
            "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            ".cta_group::2.L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(
                ptx::smem_u32(dst_smem)),
            "l"(tmap), "r"(x), "r"(y), "r"(0), "r"(bar_cluster), "l"(policy)
            : "memory");
    else
        asm volatile(
            "cp.async.bulk.tensor.3d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
            ".L2::cache_hint [%0], [%1, {%2, %3, %4}], [%5], %6;" ::"r"(ptx::smem_u32(dst_smem)),
            "l"(tmap), "r"(x), "r"(y), "r"(0), "r"(ptx::smem_u32(bar)), "l"(policy)
            : "memory");
}

template <int MODE, int CG>
__global__ void __launch_bounds__(kWmThreads, 1)
k_gemm_wm(const __grid_constant__ CUtensorMap tmA0, const __grid_constant__ CUtensorMap tmA1,
          const __grid_constant__ SlotMaps tmB, int a_mode, const int32_t *__restrict__ offsets,
          int E, int S, int Kdim, int Nw, bf16 *__restrict__ h_out, float *__restrict__ y_out,
          unsigned *err) {
    // DOWN: tmA0 = W2 [E*D, F] (128-row box).  UP, a_mode 0: tmA0 = W1 and
    // tmA1 = V1, [E*F, D] each (64-row boxes); a_mode 1 / 2: tmA0 = both as
    // one 3-D tensor [2][E*F][D] (box 64 rows x 2), W1 first (1) or V1
    // first (2).  tmB: the sorted slot rows [S, Kdim] (x_sorted for UP, h
    // for DOWN).  Kdim: reduction length; Nw: output width
    // (F for UP, D for DOWN).
    using C = WmCfg<MODE, CG>;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    constexpr int kStages = C::kStages;
    constexpr uint32_t kStageBytes = C::kStageBytes, kStageA = C::kStageA;
    float *xchg = reinterpret_cast<float *>(smem + kStages * kStageBytes);
    WmHeader *hd = reinterpret_cast<WmHeader *>(smem + kStages * kStageBytes + C::kXchgBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = CG == 2 ? ptx::cluster_ctarank() : 0u;
    const bool issuer = rank == 0;  // the CTA that issues the MMAs
    const int nwt = (Nw + C::kOutPerCta * CG - 1) / (C::kOutPerCta * CG);
    const int nk = (Kdim + kWmBK - 1) / kWmBK;
    const int unit0 = blockIdx.x / CG, ustride = gridDim.x / CG;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&hd->full[s], 1);
            ptx::mbar_init(&hd->empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&hd->tfull[b], 1);
            ptx::mbar_init(&hd->tempty[b], 4 * CG);
        }
        ptx::mbar_init(&hd->done, 1);
        ptx::fence_barrier_init();
        ptx::prefetch_tmap(&tmA0);
        if (MODE == kWmUp && a_mode == 0) ptx::prefetch_tmap(&tmA1);
        ptx::prefetch_tmap(&tmB.m[C::kRowsB / 16 - 1]);
    }
    if (warp == 1) {
        if (CG == 2) tmem_alloc_pair(&hd->tmem_base, kWmTmemCols);
        else tmem_alloc(&hd->tmem_base, kWmTmemCols);
    }
    ptx::grid_dependency_wait();  // offsets and the slot rows come from earlier kernels
    if (warp == 2) wm_prefix(offsets, E, S, nwt, hd->tprefix, err);
    tc_fence_before();
    if (CG == 2) ptx::cluster_sync_all();  // barriers initialised in both CTAs
    else __syncthreads();
    tc_fence_after();
    const uint32_t tmem = hd->tmem_base;
    const int n_units = hd->tprefix[E];

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            // a weight tile serves the 2-3 slot runs of its expert on
            // neighbouring pairs: normal priority keeps it in L2 between them
            // (evict-first: 2-3% slower, DRAM reads 14% above the weights)
            const uint64_t pol_w = ptx::policy_evict_normal();
            const uint64_t pol_x = ptx::policy_evict_last();
            uint32_t it = 0;
            bool ok = true;
            WmTile t;
            for (int i = 0; ok && wm_item(hd->tprefix, offsets, E, n_units, unit0, ustride, i,
                                          C::kGran, t);
                 ++i) {
                if (t.cnt == 0) continue;
                const uint32_t rows_b = (uint32_t)(t.n / CG);  // a multiple of 16, <= kRowsB
                const int brow = t.s0 + (int)(rank * rows_b);
                const int arow = t.e * Nw + (t.wt * CG + (int)rank) * C::kOutPerCta;

                for (int kb = 0; kb < nk; ++kb, ++it) {
                    const uint32_t s = it % kStages, ph = (it / kStages) & 1;
                    if (!(ok = ptx::mbar_wait_hint(&hd->empty[s], ph ^ 1, err))) break;
                    unsigned char *sa = smem + s * kStageBytes;
                    unsigned char *sb = sa + kStageA;
                    const int kx = kb * kWmBK;
                    uint64_t *fb = &hd->full[s];
                    const uint32_t fbc = CG == 2 ? ptx::map_rank(ptx::smem_u32(fb), 0) : 0u;
                    // the even CTA expects the bytes of both CTAs of the pair
                    if (issuer) ptx::mbar_arrive_expect_tx(fb, (kStageA + rows_b * (kWmBK * 2)) * CG);
                    if (MODE == kWmUp && a_mode != 0) {
                        wm_tma3<CG>(sa, &tmA0, kx, arow, fb, fbc, pol_w);
                    } else {
                        wm_tma<CG>(sa, &tmA0, kx, arow, fb, fbc, pol_w);
                        if (MODE == kWmUp)
                            wm_tma<CG>(sa + kStageA / 2, &tmA1, kx, arow, fb, fbc, pol_w);
                    }
                    wm_tma<CG>(sb, &tmB.m[rows_b / 16 - 1], kx, brow, fb, fbc, pol_x);
                }
            }
            // let copies still in flight land before the block can exit: the
            // even CTA sees its stages fill; the odd CTA, whose copies complete
            // on the even CTA's barriers, sees its stages consumed
            for (uint32_t k = (it > kStages ? it - kStages : 0); k < it; ++k) {
                if (issuer) ptx::mbar_wait_hint(&hd->full[k % kStages], (k / kStages) & 1, err);
                else ptx::mbar_wait_hint(&hd->empty[k % kStages], (k / kStages) & 1, err);
            }
        }
        __syncwarp();
    } else if (warp == 1) {
        if (issuer) {
            // -------------------------------------------------------- MMA issuer
            if (lane == 0) {
                uint32_t it = 0, tl = 0;
                bool ok = true;
                WmTile t;
                for (int i = 0; ok && wm_item(hd->tprefix, offsets, E, n_units, unit0, ustride,
                                              i, C::kGran, t);
                     ++i) {
                    if (t.cnt == 0) continue;
                    const uint32_t acc = tl & 1, aph = (tl >> 1) & 1;
                    ++tl;
                    // released by both CTAs' epilogues
                    if (!(ok = CG == 2 ? ptx::mbar_wait_cluster(&hd->tempty[acc], aph ^ 1, err)
                                       : ptx::mbar_wait(&hd->tempty[acc], aph ^ 1, err)))
                        break;
                    tc_fence_after();
                    const uint32_t d_tmem = tmem + acc * 256;
                    const uint32_t idesc = C::kIdescBase | ((uint32_t)(t.n >> 3) << 17);
                    for (int kb = 0; kb < nk; ++kb, ++it) {
                        const uint32_t s = it % kStages, ph = (it / kStages) & 1;
                        if (!(ok = ptx::mbar_wait_hint(&hd->full[s], ph, err))) break;
                        tc_fence_after();
                        const uint32_t sa = ptx::smem_u32(smem + s * kStageBytes);
                        const uint64_t adesc = smem_desc(sa), bdesc = smem_desc(sa + kStageA);
#pragma unroll
                        for (int kk = 0; kk < kWmBK / 16; ++kk) {
                            const uint32_t accum = (kb | kk) != 0 ? 1u : 0u;
                            if (CG == 2)
                                mma_bf16_pair(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, idesc, accum);
                            else
                                mma_bf16(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, idesc, accum);
                        }
                        // the stage is free (in both CTAs) once these MMAs finish
                        if (CG == 2) mma_commit_pair(&hd->empty[s], 3);
                        else mma_commit(&hd->empty[s]);
                    }
                    if (ok) {
                        if (CG == 2) mma_commit_pair(&hd->tfull[acc], 3);
                        else mma_commit(&hd->tfull[acc]);
                    }
                }
                // every MMA issued by this thread has completed once `done` flips
                if (CG == 2) mma_commit_pair(&hd->done, 1);
                else mma_commit(&hd->done);
                ptx::mbar_wait(&hd->done, 0, err);
            }
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int q = warp & 3;  // tensor-memory lane quarter of this warp
        bool dead = false;       // a wait gave up: keep the barrier sequence, skip the work
        uint32_t tl = 0, chunk = 0;
        const uint32_t tempty_issuer0 =
            CG == 2 ? ptx::map_rank(ptx::smem_u32(&hd->tempty[0]), 0) : 0u;
        WmTile t;
        for (int i = 0; wm_item(hd->tprefix, offsets, E, n_units, unit0, ustride, i, C::kGran, t);
             ++i) {
            if (t.cnt == 0) continue;
            const uint32_t acc = tl & 1, aph = (tl >> 1) & 1;
            ++tl;
            if (!dead && !ptx::mbar_wait_hint(&hd->tfull[acc], aph, err)) dead = true;
            tc_fence_after();
            const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + acc * 256;
            const size_t j0 = (size_t)t.s0;
            if (MODE == kWmUp) {
                // lanes 0-63: a (W1 rows), lanes 64-127: b (V1 rows) of the
                // same 64 f (the other way round for a_mode 2); partner warps
                // q and q+2 swap half a chunk each
                const int p = q & 1;
                const bool is_a = (q < 2) != (a_mode == 2);
                const int f = (t.wt * CG + (int)rank) * C::kOutPerCta + p * 32 + lane;
                const bool f_ok = f < Nw;
#pragma unroll 1
                for (int c = 0; c < t.n; c += 32, ++chunk) {
                    float v[32];
                    if (!dead) {
                        tmem_ld32(base + c, v);
                        tmem_ld_wait();
                    } else {
#pragma unroll
                        for (int i = 0; i < 32; ++i) v[i] = 0.f;
                    }
                    float *buf = xchg + (size_t)((p * 2 + (chunk & 1)) * 2) * 512;
                    float *mine = buf + (is_a ? 0 : 512), *theirs = buf + (is_a ? 512 : 0);
                    // a warp keeps columns [0,16) (a side) or [16,32) (b side)
                    // of the chunk and sends the other half
#pragma unroll
                    for (int i = 0; i < 16; ++i) mine[i * 32 + lane] = is_a ? v[16 + i] : v[i];
                    ptx::named_bar_sync(1 + p, 64);
                    const int col0 = c + (is_a ? 0 : 16);
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        const float o = theirs[i * 32 + lane];
                        const float hv = is_a ? silu(v[i]) * o : silu(o) * v[16 + i];
                        const int col = col0 + i;
                        if (!dead && f_ok && col < t.cnt)
                            h_out[(j0 + col) * Nw + f] = __float2bfloat16_rn(hv);
                    }
                }
            } else {
                const int dcol = (t.wt * CG + (int)rank) * C::kOutPerCta + q * 32 + lane;
                const bool d_ok = dcol < Nw && !dead;
#pragma unroll 1
                for (int c = 0; c < t.n; c += 32) {
                    float v[32];
                    if (!dead) {
                        tmem_ld32(base + c, v);
                        tmem_ld_wait();
                    }
                    if (d_ok) {
#pragma unroll
                        for (int i = 0; i < 32; ++i)
                            if (c + i < t.cnt) y_out[(j0 + c + i) * Nw + dcol] = v[i];
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) {
                if (CG == 2 && !issuer)
                    ptx::mbar_arrive_cluster(tempty_issuer0 + acc * (uint32_t)sizeof(uint64_t));
                else
                    ptx::mbar_arrive(&hd->tempty[acc]);
            }
        }
    }
    __syncwarp();
    tc_fence_before();
    if (CG == 2) ptx::cluster_sync_all();  // no CTA leaves while its pair may touch it
    else __syncthreads();
    tc_fence_after();
    if (warp == 1) {
        if (CG == 2) tmem_dealloc_pair(tmem, kWmTmemCols);
        else tmem_dealloc(tmem, kWmTmemCols);
    }
}

template <int MODE, int CG>
cudaError_t launch_wm_cg(const CUtensorMap &a0, const CUtensorMap &a1, const SlotMaps &b,
                         int a_mode, const int32_t *offsets, int E, int S, int Kdim, int Nw,
                         bf16 *h, float *y, int grid, cudaStream_t st, const char *name) {
    using C = WmCfg<MODE, CG>;
    const void *kern = (const void *)k_gemm_wm<MODE, CG>;
    unsigned *err = device_info().err;
    CUtensorMap m0 = a0, m1 = a1;
    SlotMaps mb = b;
    void *args[] = {&m0, &m1, &mb, &a_mode, &offsets, &E, &S, &Kdim, &Nw, &h, &y, &err};
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid);
    cfg.blockDim = dim3(kWmThreads);
    cfg.dynamicSmemBytes = C::kSmem;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = CG;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = 1;
    cfg.attrs = attr;
    cfg.numAttrs = CG == 2 ? 2 : 1;
    LaunchScope ls(name, st);
    return cudaLaunchKernelExC(&cfg, kern, args);
}

// The first n maps of the slot rows [S, Kdim] (box heights 16, ..., 16 n).
bool slot_maps(SlotMaps &b, const void *base, int S, int Kdim, int n) {
    for (int i = 0; i < n; ++i)
        if (!make_map(&b.m[i], base, (uint64_t)S, (uint64_t)Kdim, 16u * (i + 1))) return false;
    for (int i = n; i < 16; ++i) b.m[i] = b.m[n - 1];
    return true;
}

// CTA pairs when the device can keep pairs resident (one per two SMs), else
// one CTA per SM.  Per device: the number of resident pairs.
template <int MODE>
int wm_pairs() {
    static int cached[64];
    static std::once_flag once[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 0;
    std::call_once(once[dev], [] {
        using C = WmCfg<MODE, 2>;
        const void *kern = (const void *)k_gemm_wm<MODE, 2>;
        int pairs = 0;
        if (cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                 (int)C::kSmem) == cudaSuccess) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(device_info().sm_count & ~1);
            cfg.blockDim = dim3(kWmThreads);
            cfg.dynamicSmemBytes = C::kSmem;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = 2;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            if (cudaOccupancyMaxActiveClusters(&pairs, kern, &cfg) != cudaSuccess) pairs = 0;
        }
        (void)cudaGetLastError();
        int dv = 0;
        cudaGetDevice(&dv);
        cached[dv] = std::min(pairs, device_info().sm_count / 2);
    });
    return cached[dev];
}

// The single-CTA form serves devices that cannot keep CTA pairs resident;
// MOE_WM_SINGLE_CTA=1 in the environment (read on every call) selects it
// anyway, so that it can be tested where pairs are available.
bool single_cta_forced() {
    const char *v = getenv("MOE_WM_SINGLE_CTA");
    return v && v[0] == '1' && v[1] == 0;
}

template <int MODE>
cudaError_t launch_wm(const CUtensorMap (&a)[2], const void *slots, int a_mode,
                      const int32_t *offsets, int E, int S, int Kdim, int Nw, bf16 *h, float *y,
                      cudaStream_t st, const char *name) {
    const int pairs = single_cta_forced() ? 0 : wm_pairs<MODE>();
    SlotMaps b;
    if (!slot_maps(b, slots, S, Kdim, pairs > 0 ? 8 : 16)) return cudaErrorInvalidValue;
    if (pairs > 0)
        return launch_wm_cg<MODE, 2>(a[0], a[1], b, a_mode, offsets, E, S, Kdim, Nw, h, y,
                                     2 * pairs, st, name);
    const void *kern = (const void *)k_gemm_wm<MODE, 1>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)WmCfg<MODE, 1>::kSmem);
    if (e != cudaSuccess) return e;
    return launch_wm_cg<MODE, 1>(a[0], a[1], b, a_mode, offsets, E, S, Kdim, Nw, h, y,
                                 device_info().sm_count, st, name);
}


// W1 and V1 [rows, cols] as one 3-D tensor [2][rows][cols] based at the
// lower address, the higher one a stride away (box 64 columns x 64 rows x
// 2); false when the distance is not a valid stride.  *v1_first tells which
// tensor comes first.
bool weight_pair_map(CUtensorMap *m, const void *w1, const void *v1, uint64_t rows,
                     uint64_t cols, bool *v1_first) {
    auto fn = encode_fn();
    if (!fn) return false;
    const uintptr_t a = reinterpret_cast<uintptr_t>(w1), b = reinterpret_cast<uintptr_t>(v1);
    *v1_first = b < a;
    const uintptr_t lo = *v1_first ? b : a, dist = *v1_first ? a - b : b - a;
    if (dist < rows * cols * 2 || dist % 16 != 0 || dist >= (uintptr_t(1) << 40)) return false;
    cuuint64_t dims[3] = {cols, rows, 2};
    cuuint64_t strides[2] = {cols * 2, (cuuint64_t)dist};
    cuuint32_t box[3] = {64u, 64u, 2u};
    cuuint32_t estr[3] = {1, 1, 1};
    return fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, reinterpret_cast<void *>(lo), dims, strides,
              box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

cudaError_t launch_gemm_up_wm(const moe_dims &d, int T, const void *x_sorted,
                              const int32_t *offsets, const void *w1, const void *v1, void *h,
                              cudaStream_t st) {
    const int S = T * d.top_k, D = d.d_model, F = d.ffn_hidden, E = d.n_experts;
    CUtensorMap a[2];
    bool v1_first = false;
    int a_mode;
    if (weight_pair_map(&a[0], w1, v1, (uint64_t)E * F, (uint64_t)D, &v1_first)) {
        a[1] = a[0];
        a_mode = v1_first ? 2 : 1;
    } else {
        if (!make_map(&a[0], w1, (uint64_t)E * F, (uint64_t)D, 64) ||
            !make_map(&a[1], v1, (uint64_t)E * F, (uint64_t)D, 64))
            return cudaErrorInvalidValue;
        a_mode = 0;
    }
    return launch_wm<kWmUp>(a, x_sorted, a_mode, offsets, E, S, D, F, static_cast<bf16 *>(h), nullptr, st,
                            "gemm_up_glu_tc");
}

cudaError_t launch_gemm_down_wm(const moe_dims &d, int T, const void *h, const int32_t *offsets,
                                const void *w2, float *y_sorted, cudaStream_t st,
                                const char *name) {
    const int S = T * d.top_k, D = d.d_model, F = d.ffn_hidden, E = d.n_experts;
    CUtensorMap a[2];
    if (!make_map(&a[0], w2, (uint64_t)E * D, (uint64_t)F, 128)) return cudaErrorInvalidValue;
    a[1] = a[0];
    return launch_wm<kWmDown>(a, h, 0, offsets, E, S, F, D, nullptr, y_sorted, st,
                              name ? name : "gemm_down_tc");
}

}  // namespace moe
