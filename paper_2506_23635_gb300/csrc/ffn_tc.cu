// Grouped expert GEMMs on the tcgen05 tensor cores (prefill and larger
// decode batches), bf16 inputs, fp32 accumulation in tensor memory.
//
// Table 1 notes (d),(e) of arxiv 2506.23635: every expert is three
// D_embed x D_ffn matrices.  With the slots sorted by expert (moe_dispatch),
// the expert FFN is two grouped GEMMs with a variable number of rows per
// expert:
//
//   UP   (GLU):  h[j, f] = SiLU(x_j . W1[e,f,:]) * (x_j . V1[e,f,:])   -> bf16
//   DOWN:        y[j, d] = h[j, :] . W2[e,d,:]                          -> fp32
//
// for the sorted slots j of expert e (x_j = the gathered token rows).
// Tile = 128 slots (M, the A operand, K-major) x BN = 256 weight rows (N, the
// B operand, K-major) x 64 of the reduction dimension per pipeline stage
// (Cfg keeps BN and the stage count template parameters).  In UP the BN
// weight rows are BN/2 rows of W1 followed by the same BN/2 rows of V1, so
// one accumulator holds a (first half of the columns) and b (second half)
// for the same f, and the GLU runs in the epilogue straight from tensor
// memory.
//
// Per CTA (one per SM, persistent), 6 warps:
//   warp 0     TMA producer (one lane): A and B tiles into a 4-stage ring,
//              128-byte swizzle, completion on mbarriers;
//   warp 1     tensor-memory allocator and MMA issuer (one lane):
//              tcgen05.mma kind::f16, M=128, N=BN, K=16, into one of two
//              BN-column fp32 accumulators; tcgen05.commit frees a stage
//              and hands a finished accumulator to the epilogue;
//   warps 2-5  epilogue: tcgen05.ld of their 32 tensor-memory lanes, GLU or
//              plain copy, stores to global memory.
// Tiles are numbered expert by expert (weight tile outer, slot tile inner, so
// CTAs working at the same time share weight tiles in L2) from the device
// resident dispatch offsets; CTA b takes tiles b, b+G, ...  No host sync.
// Every mbarrier wait is bounded (see ptx.cuh).
#include <cuda.h>
#include <cudaTypedefs.h>

#include <mutex>

#include "tc.cuh"

namespace moe {
namespace {

using namespace tc;

constexpr int BM = 128, BK = 64;
constexpr int kMaxStages = 8;
constexpr int kThreadsTc = 192;
constexpr uint32_t kStageA = BM * BK * 2;  // 16 KB
constexpr size_t kTcHeaderBytes = 2048;
constexpr int kMaxSwapStages = 12;

enum Mode { kUp = 0, kDown = 1 };

// Tile shape of one instantiation: BN weight rows per tile (UP: BN/2 rows of
// W1 and the same BN/2 rows of V1), STAGES pipeline stages.
template <int MODE, int BN_, int STAGES_>
struct Cfg {
    static constexpr int BN = BN_;
    static constexpr int kStages = STAGES_;
    static constexpr int kCols = MODE == kUp ? BN / 2 : BN;  // output columns per tile
    static constexpr uint32_t kStageB = BN * BK * 2;
    static constexpr uint32_t kStageBytes = kStageA + kStageB;
    static constexpr uint32_t kTmemCols = 2 * BN;  // two accumulators
    static constexpr size_t kSmem = 1024 /*align slack*/ + kStages * kStageBytes + kTcHeaderBytes;
    // kind::f16 instruction descriptor: bf16 A and B, fp32 D, both K-major,
    // N = BN, M = 128
    static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                                       ((uint32_t)(BN >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
    static_assert(kStages <= kMaxStages, "too many stages");
    static_assert(kCols % 32 == 0, "epilogue works in 32-column steps");
    static_assert((kTmemCols & (kTmemCols - 1)) == 0 && kTmemCols >= 32 && kTmemCols <= 512,
                  "tensor memory is allocated in powers of two");
    static_assert(kSmem <= 227 * 1024, "shared memory");
};

struct TcHeader {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t done;
    uint32_t tmem_base;
    int tprefix[257];  // tile prefix over experts
};
static_assert(sizeof(TcHeader) <= kTcHeaderBytes, "tcgen05 kernel header too large");

// ---- tile schedule -------------------------------------------------------------

// tprefix[e] = sum over earlier experts of ceil(n_e / BM) * n_tiles_n.
__device__ void tile_prefix(const int32_t *offsets, int E, int S, int ntn, int *tprefix,
                            unsigned *err) {
    const int lane = threadIdx.x & 31;
    int run = 0;
    for (int base = 0; base < E; base += 32) {
        const int e = base + lane;
        int c = 0;
        if (e < E) {
            const int lo = offsets[e], hi = offsets[e + 1];
            if (lo < 0 || hi < lo || hi > S) set_error(err, kErrIndex);
            else c = ((hi - lo + BM - 1) / BM) * ntn;
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

struct Tile {
    int e, mt, nt, row0, rows;  // rows: valid slots in this M tile
};

__device__ __forceinline__ Tile tile_of(const int *tprefix, const int32_t *offsets, int E, int ntn,
                                        int u) {
    Tile t;
    t.e = chunk_expert(tprefix, E, u);
    const int r = u - tprefix[t.e];
    const int n_e = offsets[t.e + 1] - offsets[t.e];
    const int mtiles = (n_e + BM - 1) / BM;
    t.nt = r / mtiles;
    t.mt = r - t.nt * mtiles;
    t.row0 = offsets[t.e] + t.mt * BM;
    t.rows = min(BM, n_e - t.mt * BM);
    return t;
}

// The CTA's work as segments (unit u, k-blocks [kb0, kb1)).  Standard: units
// b, b+G, ... whole.  Stream-K (down projection with a tail buffer, at least
// as many units as CTAs): CTA b takes the contiguous share [W b/G, W (b+1)/G)
// of the W = units x nk (unit, k-block) pairs, so every CTA does the same
// amount of work; a share is at least nk long, so a unit is split at most
// once -- into a head (k-block 0 on) and a tail (ending at nk).
struct SegIter {
    bool sk;
    int nk, G;
    long long pos, end;
    __device__ __forceinline__ bool next(int n_units, int &u, int &kb0, int &kb1) {
        if (sk) {
            if (pos >= end) return false;
            u = (int)(pos / nk);
            kb0 = (int)(pos - (long long)u * nk);
            kb1 = (int)min((long long)nk, kb0 + (end - pos));
            pos += kb1 - kb0;
            return true;
        }
        if (pos >= n_units) return false;
        u = (int)pos;
        kb0 = 0;
        kb1 = nk;
        pos += G;
        return true;
    }
};

__device__ __forceinline__ SegIter make_segs(bool sk, int n_units, int nk) {
    SegIter it;
    it.sk = sk;
    it.nk = nk;
    it.G = gridDim.x;
    if (sk) {
        const long long W = (long long)n_units * nk;
        it.pos = W * blockIdx.x / gridDim.x;
        it.end = W * (blockIdx.x + 1) / gridDim.x;
    } else {
        it.pos = blockIdx.x;
        it.end = 0;
    }
    return it;
}

// ---- the kernel ------------------------------------------------------------------

template <int MODE, class C>
__global__ void __launch_bounds__(kThreadsTc, 1)
k_gemm_tc(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB0,
          const __grid_constant__ CUtensorMap tmB1, const int32_t *__restrict__ offsets, int E,
          int S, int Kdim, int Nw, uint32_t a_bytes, bf16 *__restrict__ h_out,
          float *__restrict__ y_out, float *__restrict__ y_tail, unsigned *err) {
    // Kdim: reduction length (D for UP, F for DOWN); Nw: weight rows per
    // expert (F for UP, D for DOWN) = the output width.  a_bytes: bytes of
    // the A box (rows x 128 B).  y_tail (DOWN, optional): the second output
    // buffer of the stream-K schedule (SegIter): heads go to y_out, tails to
    // y_tail, and a unit done whole zeroes its part of y_tail, so the caller
    // adds y_out + y_tail.  In a decode batch an expert holds at most T
    // slots, so only ceil(T/16)*16 rows are loaded; the MMA still reads 128
    // rows and the rows past the box give accumulator rows nobody stores.
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    constexpr int kStages = C::kStages, BN = C::BN, kCols = C::kCols;
    constexpr uint32_t kStageBytes = C::kStageBytes, kStageB = C::kStageB;
    TcHeader *hd = reinterpret_cast<TcHeader *>(smem + kStages * kStageBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int ntn = (Nw + kCols - 1) / kCols;
    const int nk = (Kdim + BK - 1) / BK;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&hd->full[s], 1);
            ptx::mbar_init(&hd->empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            ptx::mbar_init(&hd->tfull[b], 1);
            ptx::mbar_init(&hd->tempty[b], 4);
        }
        ptx::mbar_init(&hd->done, 1);
        ptx::fence_barrier_init();
        ptx::prefetch_tmap(&tmA);
        ptx::prefetch_tmap(&tmB0);
        if (MODE == kUp) ptx::prefetch_tmap(&tmB1);
    }
    if (warp == 1) tmem_alloc(&hd->tmem_base, C::kTmemCols);
    ptx::grid_dependency_wait();  // offsets and the A operand come from earlier kernels
    if (warp == 2) tile_prefix(offsets, E, S, ntn, hd->tprefix, err);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = hd->tmem_base;
    const int n_tiles = hd->tprefix[E];
    const bool sk = MODE == kDown && y_tail != nullptr && n_tiles >= (int)gridDim.x;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            const uint64_t pol_a = ptx::policy_evict_last();
            const uint64_t pol_b = ptx::policy_evict_first();
            uint32_t it = 0;
            bool ok = true;
            SegIter segs = make_segs(sk, n_tiles, nk);
            int u, kb0, kb1;
            while (ok && segs.next(n_tiles, u, kb0, kb1)) {
                const Tile t = tile_of(hd->tprefix, offsets, E, ntn, u);
                const int brow = t.e * Nw + t.nt * kCols;
                for (int kb = kb0; kb < kb1; ++kb, ++it) {
                    const uint32_t s = it % kStages, ph = (it / kStages) & 1;
                    if (!(ok = ptx::mbar_wait(&hd->empty[s], ph ^ 1, err))) break;
                    unsigned char *sa = smem + s * kStageBytes;
                    unsigned char *sb = sa + kStageA;
                    ptx::mbar_arrive_expect_tx(&hd->full[s], a_bytes + kStageB);
                    ptx::tma_load_2d(sa, &tmA, kb * BK, t.row0, &hd->full[s], pol_a);
                    if (MODE == kUp) {
                        ptx::tma_load_2d(sb, &tmB0, kb * BK, brow, &hd->full[s], pol_b);
                        ptx::tma_load_2d(sb + kStageB / 2, &tmB1, kb * BK, brow, &hd->full[s],
                                         pol_b);
                    } else {
                        ptx::tma_load_2d(sb, &tmB0, kb * BK, brow, &hd->full[s], pol_b);
                    }
                }
            }
            // let loads still in flight land before the block can exit
            for (uint32_t k = (it > kStages ? it - kStages : 0); k < it; ++k)
                ptx::mbar_wait(&hd->full[k % kStages], (k / kStages) & 1, err);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            uint32_t it = 0, tl = 0;
            bool ok = true;
            SegIter segs = make_segs(sk, n_tiles, nk);
            int u, kb0, kb1;
            for (; ok && segs.next(n_tiles, u, kb0, kb1); ++tl) {
                const uint32_t acc = tl & 1, aph = (tl >> 1) & 1;
                if (!(ok = ptx::mbar_wait(&hd->tempty[acc], aph ^ 1, err))) break;
                tc_fence_after();
                const uint32_t d_tmem = tmem + acc * BN;
                for (int kb = kb0; kb < kb1; ++kb, ++it) {
                    const uint32_t s = it % kStages, ph = (it / kStages) & 1;
                    if (!(ok = ptx::mbar_wait(&hd->full[s], ph, err))) break;
                    tc_fence_after();
                    const uint32_t sa = ptx::smem_u32(smem + s * kStageBytes);
                    const uint64_t adesc = smem_desc(sa), bdesc = smem_desc(sa + kStageA);
#pragma unroll
                    for (int kk = 0; kk < BK / 16; ++kk)
                        mma_bf16(d_tmem, adesc + 2 * kk, bdesc + 2 * kk, C::kIdesc,
                                 (kb != kb0 || kk != 0) ? 1u : 0u);
                    mma_commit(&hd->empty[s]);  // stage free once these MMAs finish
                }
                if (ok) mma_commit(&hd->tfull[acc]);
            }
            // every MMA issued by this thread has completed once `done` flips
            mma_commit(&hd->done);
            ptx::mbar_wait(&hd->done, 0, err);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        const int q = warp & 3;          // tensor-memory lane quarter of this warp
        const int m = q * 32 + lane;     // row of the tile = slot offset
        uint32_t tl = 0;
        SegIter segs = make_segs(sk, n_tiles, nk);
        int u, kb0, kb1;
        for (; segs.next(n_tiles, u, kb0, kb1); ++tl) {
            const Tile t = tile_of(hd->tprefix, offsets, E, ntn, u);
            const uint32_t acc = tl & 1, aph = (tl >> 1) & 1;
            float *ydst = kb0 == 0 ? y_out : y_tail;          // head / tail of the unit
            float *yzero = (y_tail && kb0 == 0 && kb1 == nk) ? y_tail : nullptr;
            if (!ptx::mbar_wait(&hd->tfull[acc], aph, err)) break;
            tc_fence_after();
            const uint32_t base = tmem + ((uint32_t)(q * 32) << 16) + acc * BN;
            const bool row_ok = m < t.rows;
            const size_t j = (size_t)t.row0 + m;
            if (MODE == kUp) {
                const int f0 = t.nt * kCols;
#pragma unroll 1
                for (int c = 0; c < kCols; c += 32) {
                    float a[32], b[32];
                    tmem_ld32(base + c, a);
                    tmem_ld32(base + kCols + c, b);
                    tmem_ld_wait();
                    if (row_ok) {
                        uint32_t pk[16];
#pragma unroll
                        for (int i = 0; i < 16; ++i) {
                            const float h0 = silu(a[2 * i]) * b[2 * i];
                            const float h1 = silu(a[2 * i + 1]) * b[2 * i + 1];
                            const __nv_bfloat162 p2 = __floats2bfloat162_rn(h0, h1);
                            pk[i] = *reinterpret_cast<const uint32_t *>(&p2);
                        }
                        bf16 *dst = h_out + j * Nw + f0 + c;
#pragma unroll
                        for (int g = 0; g < 4; ++g)  // 8 columns per 16-byte store
                            if (f0 + c + g * 8 < Nw)
                                *reinterpret_cast<uint4 *>(dst + g * 8) =
                                    make_uint4(pk[4 * g], pk[4 * g + 1], pk[4 * g + 2], pk[4 * g + 3]);
                    }
                }
            } else {
                const int d0 = t.nt * BN;
#pragma unroll 1
                for (int c = 0; c < BN; c += 32) {
                    float v[32];
                    tmem_ld32(base + c, v);
                    tmem_ld_wait();
                    if (row_ok) {
                        float *dst = ydst + j * Nw + d0 + c;
#pragma unroll
                        for (int g = 0; g < 8; ++g)  // 4 columns per 16-byte store
                            if (d0 + c + g * 4 < Nw)
                                *reinterpret_cast<float4 *>(dst + g * 4) =
                                    make_float4(v[4 * g], v[4 * g + 1], v[4 * g + 2], v[4 * g + 3]);
                        if (yzero) {
                            float *z = yzero + j * Nw + d0 + c;
#pragma unroll
                            for (int g = 0; g < 8; ++g)
                                if (d0 + c + g * 4 < Nw)
                                    *reinterpret_cast<float4 *>(z + g * 4) =
                                        make_float4(0.f, 0.f, 0.f, 0.f);
                        }
                    }
                }
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->tempty[acc]);
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, C::kTmemCols);
}

// ---- one weight matrix against a few token rows (weights as the M operand) -------
//
// y[j, n] = x[j, :] . W[n, :] for j < T <= 128 tokens and the Nw rows of one
// matrix W [Nw, Kdim].  A decode batch fills few of the 128 slot rows of the
// MMA above, and a single matrix has few 256-row tiles; here the weights are
// the A operand instead (128 rows per tile) and the tokens the B operand
// (NTOK = 16, 32, 64 or 128 columns), so every stage is 16 KB of weights
// plus NTOK x 128 B of tokens and 6-12 stages stay in flight.
// Loaded HBM latency is ~3.5 us, so streaming at the HBM rate needs ~25 MB in
// flight: the reduction is split over gridDim.y CTAs per tile (split z writes
// its partial sums to y_out + z*T*Nw; the caller adds the parts in order).
// The weight loads of the first stages are issued before the kernel waits
// for the previous grid (weights do not depend on it).
template <int NTOK>
struct SwapCfg {
    static constexpr uint32_t kStageW = BM * BK * 2;     // 16 KB of weights
    static constexpr uint32_t kStageX = NTOK * BK * 2;   // token rows
    static constexpr uint32_t kStageBytes = kStageW + kStageX;
    static constexpr int kStages =
        (int)((227 * 1024 - 1024 - kTcHeaderBytes) / kStageBytes) < 12
            ? (int)((227 * 1024 - 1024 - kTcHeaderBytes) / kStageBytes)
            : 12;
    static constexpr size_t kSmem = 1024 + (size_t)kStages * kStageBytes + kTcHeaderBytes;
    static constexpr uint32_t kTmemCols = NTOK < 32 ? 32 : NTOK;
    // kind::f16: bf16 A and B, fp32 D, both K-major, N = NTOK, M = 128
    static constexpr uint32_t kIdesc = (1u << 4) | (1u << 7) | (1u << 10) |
                                       ((uint32_t)(NTOK >> 3) << 17) | ((uint32_t)(BM >> 4) << 24);
    static_assert(NTOK % 16 == 0 && NTOK >= 16 && NTOK <= 128, "token columns");
    static_assert(kStageBytes % 1024 == 0, "stages stay 1024-byte aligned");
    static_assert(kStages >= 4 && kStages <= kMaxSwapStages, "stages");
    static_assert((kTmemCols & (kTmemCols - 1)) == 0, "tensor memory is allocated in powers of two");
    static_assert(kSmem <= 227 * 1024, "shared memory");
};

struct SwapHeader {
    uint64_t full[kMaxSwapStages];
    uint64_t empty[kMaxSwapStages];
    uint64_t tfull;
    uint32_t tmem_base;
};
static_assert(sizeof(SwapHeader) <= kTcHeaderBytes, "swap kernel header too large");

template <int NTOK>
__global__ void __launch_bounds__(kThreadsTc, 1)
k_gemm_swap(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
            int T, int Kdim, int Nw, float *__restrict__ y_out, unsigned *err) {
    using C = SwapCfg<NTOK>;
    extern __shared__ unsigned char smem_raw[];
    unsigned char *smem = reinterpret_cast<unsigned char *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    constexpr int kStages = C::kStages;
    SwapHeader *hd = reinterpret_cast<SwapHeader *>(smem + kStages * C::kStageBytes);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nk_all = (Kdim + BK - 1) / BK;
    const int kb0 = (int)((long long)nk_all * blockIdx.y / gridDim.y);
    const int nk = (int)((long long)nk_all * (blockIdx.y + 1) / gridDim.y) - kb0;
    const int n0 = blockIdx.x * BM;  // first weight row of this CTA's tile
    y_out += (size_t)blockIdx.y * T * Nw;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            ptx::mbar_init(&hd->full[s], 1);
            ptx::mbar_init(&hd->empty[s], 1);
        }
        ptx::mbar_init(&hd->tfull, 1);
        ptx::fence_barrier_init();
        ptx::prefetch_tmap(&tmW);
        ptx::prefetch_tmap(&tmX);
    }
    if (warp == 1) tmem_alloc(&hd->tmem_base, C::kTmemCols);
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = hd->tmem_base;

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        if (lane == 0) {
            const uint64_t pol_w = ptx::policy_evict_first();
            const uint64_t pol_x = ptx::policy_evict_last();
            const int early = nk < kStages ? nk : kStages;
            // weights of the first stages: independent of earlier kernels
            for (int kb = 0; kb < early; ++kb) {
                ptx::mbar_arrive_expect_tx(&hd->full[kb], C::kStageBytes);
                ptx::tma_load_2d(smem + kb * C::kStageBytes, &tmW, (kb0 + kb) * BK, n0, &hd->full[kb],
                                 pol_w);
            }
            ptx::grid_dependency_wait();  // the token rows come from the previous kernel
            for (int kb = 0; kb < early; ++kb)
                ptx::tma_load_2d(smem + kb * C::kStageBytes + C::kStageW, &tmX, (kb0 + kb) * BK, 0,
                                 &hd->full[kb], pol_x);
            int issued = early;
            for (int kb = early; kb < nk; ++kb) {
                const uint32_t s = kb % kStages, ph = (kb / kStages) & 1;
                if (!ptx::mbar_wait(&hd->empty[s], ph ^ 1, err)) break;
                unsigned char *st = smem + s * C::kStageBytes;
                ptx::mbar_arrive_expect_tx(&hd->full[s], C::kStageBytes);
                ptx::tma_load_2d(st, &tmW, (kb0 + kb) * BK, n0, &hd->full[s], pol_w);
                ptx::tma_load_2d(st + C::kStageW, &tmX, (kb0 + kb) * BK, 0, &hd->full[s], pol_x);
                issued = kb + 1;
            }
            // let loads still in flight land before the block can exit
            for (int k = (issued > kStages ? issued - kStages : 0); k < issued; ++k)
                ptx::mbar_wait(&hd->full[k % kStages], (k / kStages) & 1, err);
        }
    } else if (warp == 1) {
        // ------------------------------------------------------------ MMA issuer
        if (lane == 0) {
            bool ok = true;
            for (int kb = 0; kb < nk; ++kb) {
                const uint32_t s = kb % kStages, ph = (kb / kStages) & 1;
                if (!(ok = ptx::mbar_wait(&hd->full[s], ph, err))) break;
                tc_fence_after();
                const uint32_t sa = ptx::smem_u32(smem + s * C::kStageBytes);
                const uint64_t adesc = smem_desc(sa), bdesc = smem_desc(sa + C::kStageW);
#pragma unroll
                for (int kk = 0; kk < BK / 16; ++kk)
                    mma_bf16(tmem, adesc + 2 * kk, bdesc + 2 * kk, C::kIdesc,
                             (kb | kk) != 0 ? 1u : 0u);
                mma_commit(&hd->empty[s]);
            }
            // tfull flips once every MMA issued here has completed; wait for it
            // here too, so tensor memory is never freed under a running MMA
            mma_commit(&hd->tfull);
            (void)ok;
            ptx::mbar_wait(&hd->tfull, 0, err);
        }
        __syncwarp();
    } else {
        // ------------------------------------------------------------ epilogue
        ptx::grid_dependency_wait();
        const int q = warp & 3;
        const int n = n0 + q * 32 + lane;  // weight row = output column
        if (nk <= 0) {  // an empty share of the reduction: its part is zero
            if (n < Nw)
                for (int j = 0; j < T; ++j) y_out[(size_t)j * Nw + n] = 0.f;
        } else if (ptx::mbar_wait(&hd->tfull, 0, err)) {
            tc_fence_after();
            const uint32_t base = tmem + ((uint32_t)(q * 32) << 16);
#pragma unroll 1
            for (int c = 0; c < NTOK; c += 32) {
                float v[32];
                tmem_ld32(base + c, v);
                tmem_ld_wait();
                if (n < Nw) {
#pragma unroll
                    for (int j = 0; j < 32; ++j)
                        if (c + j < NTOK && c + j < T) y_out[(size_t)(c + j) * Nw + n] = v[j];
                }
            }
        }
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem, C::kTmemCols);
}

// ---- gather of the A operand: x_sorted[j, :] = x[perm[j] / K, :] ----------------

__global__ void __launch_bounds__(256)
k_gather_rows(int S, int D, int K, int n_chunk, const bf16 *__restrict__ x,
              const int32_t *__restrict__ perm, bf16 *__restrict__ xs,
              const int32_t *__restrict__ range, int n_range, unsigned *err) {
    ptx::grid_dependency_wait();
    const int nv = D >> 3;  // 16-byte vectors per row
    // sorted positions [range[0], range[n_range]) only, when a range of
    // experts is given (one node's share of an expert-parallel layer)
    const int j_lo = range ? max(0, min(S, range[0])) : 0;
    const int j_hi = range ? max(j_lo, min(S, range[n_range])) : S;
    // a warp per (sorted row, chunk of the row): n_chunk chunks a row, so
    // that few rows still spread over the SMs; eight 16-byte loads of each
    // lane in flight (2048-token prefill: 31 -> 27.5 us against four)
    const int lane = threadIdx.x & 31, wpb = blockDim.x >> 5;
    const int per = (nv + n_chunk - 1) / n_chunk;
    const long long n_items = (long long)(j_hi - j_lo) * n_chunk;
    for (long long i = (long long)blockIdx.x * wpb + (threadIdx.x >> 5); i < n_items;
         i += (long long)gridDim.x * wpb) {
        const int j = j_lo + (int)(i / n_chunk), c = (int)(i % n_chunk);
        int slot = perm[j];
        if (slot < 0 || slot >= S) {
            if (lane == 0) set_error(err, kErrIndex);
            slot = 0;
        }
        const uint4 *src = reinterpret_cast<const uint4 *>(x + (size_t)(slot / K) * D);
        uint4 *dst = reinterpret_cast<uint4 *>(xs + (size_t)j * D);
        const int v1 = min(nv, (c + 1) * per);
        int v = c * per + lane;
        for (; v + 224 < v1; v += 256) {
            uint4 a[8];
#pragma unroll
            for (int u = 0; u < 8; ++u) a[u] = __ldg(src + v + 32 * u);
#pragma unroll
            for (int u = 0; u < 8; ++u) dst[v + 32 * u] = a[u];
        }
        for (; v + 96 < v1; v += 128) {
            const uint4 a0 = __ldg(src + v), a1 = __ldg(src + v + 32);
            const uint4 a2 = __ldg(src + v + 64), a3 = __ldg(src + v + 96);
            dst[v] = a0;
            dst[v + 32] = a1;
            dst[v + 64] = a2;
            dst[v + 96] = a3;
        }
        for (; v < v1; v += 32) dst[v] = __ldg(src + v);
    }
}

template <int MODE, class C>
cudaError_t launch_gemm(const CUtensorMap &a, const CUtensorMap &b0, const CUtensorMap &b1,
                        const int32_t *offsets, int E, int S, int Kdim, int Nw, uint32_t a_bytes,
                        bf16 *h_out, float *y_out, cudaStream_t st, const char *name = nullptr,
                        float *y_tail = nullptr) {
    const void *kern = (const void *)k_gemm_tc<MODE, C>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::kSmem);
    if (e != cudaSuccess) return e;
    unsigned *err = device_info().err;
    CUtensorMap ma = a, mb0 = b0, mb1 = b1;
    void *args[] = {&ma, &mb0, &mb1, &offsets, &E, &S, &Kdim, &Nw, &a_bytes, &h_out, &y_out,
                    &y_tail, &err};
    LaunchScope ls(name ? name : MODE == kUp ? "gemm_up_glu_tc" : "gemm_down_tc", st);
    return launch_pdl(kern, dim3(device_info().sm_count), dim3(kThreadsTc), C::kSmem, st, args);
}

// Both projections use 256-row weight tiles with 4 stages: narrower tiles
// balance the SMs better when few experts are selected, but hold too few
// weight bytes in flight per SM to stream at the HBM rate (measured: 64-row
// down-projection tiles ran 1.6x slower at 64 tokens).
using UpWide = Cfg<kUp, 256, 4>;
using DownWide = Cfg<kDown, 256, 4>;

// Rows of the A box: a whole 128-row slot tile, or for batches under 128
// tokens (an expert then holds at most T slots, all in one slot tile) just
// T rounded up to 16.
uint32_t a_box_rows(int T) {
    if (T >= BM) return BM;
    return (uint32_t)((T + 15) / 16 * 16);
}

template <int NTOK>
cudaError_t launch_swap(const CUtensorMap &w, const CUtensorMap &x, int T, int Kdim, int Nw,
                        int parts, float *y, cudaStream_t st, const char *name) {
    using C = SwapCfg<NTOK>;
    const void *kern = (const void *)k_gemm_swap<NTOK>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::kSmem);
    if (e != cudaSuccess) return e;
    unsigned *err = device_info().err;
    CUtensorMap mw = w, mx = x;
    void *args[] = {&mw, &mx, &T, &Kdim, &Nw, &y, &err};
    LaunchScope ls(name ? name : "gemm_rows_tc", st);
    return launch_pdl(kern, dim3((Nw + BM - 1) / BM, parts), dim3(kThreadsTc), C::kSmem, st,
                      args);
}

}  // namespace

bool tc_path_ok(const moe_dims &d) {
    return d.w_dtype == MOE_BF16 && d.x_dtype == MOE_BF16 && encode_fn() != nullptr;
}

cudaError_t launch_gather_rows(const moe_dims &d, int T, const void *x, const int32_t *perm,
                               void *x_sorted, cudaStream_t st, const int32_t *range,
                               int n_range) {
    const int S = T * d.top_k;
    // 8 warps a block, at most 8 blocks per SM; a row in chunks of at least
    // 32 vectors when there are fewer rows than 64 warps per SM
    const int warps = device_info().sm_count * 64;
    int n_chunk = std::max(1, std::min(d.d_model / 8 / 32, warps / std::max(1, S)));
    const long long items = (long long)S * n_chunk;
    const int grid = (int)std::max(1LL, std::min((items + 7) / 8, (long long)warps / 8));
    int Sv = S, D = d.d_model, K = d.top_k;
    const bf16 *xp = static_cast<const bf16 *>(x);
    bf16 *xs = static_cast<bf16 *>(x_sorted);
    unsigned *err = device_info().err;
    void *args[] = {&Sv, &D, &K, &n_chunk, &xp, &perm, &xs, &range, &n_range, &err};
    LaunchScope ls("gather_rows", st);
    return launch_pdl((const void *)k_gather_rows, dim3(grid), dim3(256), 0, st, args);
}

cudaError_t launch_gemm_up_tc(const moe_dims &d, int T, const void *x_sorted, const int32_t *offsets,
                              const void *w1, const void *v1, void *h, cudaStream_t st) {
    if (use_wm(d, T)) return launch_gemm_up_wm(d, T, x_sorted, offsets, w1, v1, h, st);
    const int S = T * d.top_k, D = d.d_model, F = d.ffn_hidden, E = d.n_experts;
    const uint32_t arows = a_box_rows(T);
    CUtensorMap a, b0, b1;
    if (!make_map(&a, x_sorted, (uint64_t)S, (uint64_t)D, arows) ||
        !make_map(&b0, w1, (uint64_t)E * F, (uint64_t)D, UpWide::kCols) ||
        !make_map(&b1, v1, (uint64_t)E * F, (uint64_t)D, UpWide::kCols))
        return cudaErrorInvalidValue;
    return launch_gemm<kUp, UpWide>(a, b0, b1, offsets, E, S, D, F, arows * BK * 2,
                                    static_cast<bf16 *>(h), nullptr, st);
}

cudaError_t launch_gemm_down_tc(const moe_dims &d, int T, const void *h, const int32_t *offsets,
                                const void *w2, float *y_sorted, cudaStream_t st,
                                const char *name, float *y_tail) {
    if (use_wm(d, T) && y_tail == nullptr)
        return launch_gemm_down_wm(d, T, h, offsets, w2, y_sorted, st, name);
    const int S = T * d.top_k, D = d.d_model, F = d.ffn_hidden, E = d.n_experts;
    const uint32_t arows = a_box_rows(T);
    CUtensorMap a, b0;
    if (!make_map(&a, h, (uint64_t)S, (uint64_t)F, arows) ||
        !make_map(&b0, w2, (uint64_t)E * D, (uint64_t)F, DownWide::BN))
        return cudaErrorInvalidValue;
    return launch_gemm<kDown, DownWide>(a, b0, b0, offsets, E, S, F, D, arows * BK * 2, nullptr,
                                        y_sorted, st, name, y_tail);
}

int gemm_rows_parts(int Kdim, int Nw) {
    const int tiles = (Nw + BM - 1) / BM, nk = (Kdim + BK - 1) / BK;
    const int by_sms = std::max(1, device_info().sm_count / std::max(1, tiles));
    return std::max(1, std::min({kRowsMaxParts, by_sms, nk}));
}

cudaError_t launch_gemm_rows_tc(int T, int Kdim, int Nw, const void *x, const void *w, int parts,
                                float *y, cudaStream_t st, const char *name) {
    if (T < 1 || T > kRowsMaxTokens || parts < 1 || parts > kRowsMaxParts)
        return cudaErrorInvalidValue;
    const int ntok = (T + 15) / 16 * 16;
    const uint32_t xrows = ntok <= 16 ? 16 : ntok <= 32 ? 32 : ntok <= 64 ? 64 : 128;
    CUtensorMap mw, mx;
    if (!make_map(&mw, w, (uint64_t)Nw, (uint64_t)Kdim, BM) ||
        !make_map(&mx, x, (uint64_t)T, (uint64_t)Kdim, xrows))
        return cudaErrorInvalidValue;
    if (xrows == 16) return launch_swap<16>(mw, mx, T, Kdim, Nw, parts, y, st, name);
    if (xrows == 32) return launch_swap<32>(mw, mx, T, Kdim, Nw, parts, y, st, name);
    if (xrows == 64) return launch_swap<64>(mw, mx, T, Kdim, Nw, parts, y, st, name);
    return launch_swap<128>(mw, mx, T, Kdim, Nw, parts, y, st, name);
}

}  // namespace moe
