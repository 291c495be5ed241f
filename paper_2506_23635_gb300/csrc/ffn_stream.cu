// Bulk-copy pipelined expert FFN for a few tokens per expert (decode, bf16).
//
// Sec. 4.4 of arxiv 2506.23635 bounds token generation by the time to load
// the selected experts' weights.  These kernels stream every selected weight
// row exactly once from HBM, with enough bytes in flight per SM to run at the
// copy rate:
//
//   * one CTA per SM (persistent), W consumer warps and a producer warp;
//   * the producer's lane 0 issues cp.async.bulk copies of whole weight rows
//     (W1 row + V1 row, or one W2 row) into W shared-memory stages,
//     completing on mbarriers; weights use an L2 evict-first policy;
//   * task i goes to consumer warp i % W and stage i % W: every stage belongs
//     to one warp and is used in task order, so a warp never waits on a
//     barrier phase other than the next one (a parity wait two phases ahead
//     would pass at once); the producer also tags each stage with its task
//     number and the consumer checks the tag;
//   * the consumer dots the row with the token vectors of the current
//     (expert, slot chunk), which the producer bulk-copies into a
//     double-buffered area;
//   * every CTA owns an equal contiguous share of the work, so the 152 SMs
//     finish together.
//
// k_up_glu_stream:  h[j,f] = bf16( SiLU(W1[e,f,:] . x_j) * (V1[e,f,:] . x_j) )
//   tasks = (chunk of <= NS slots of one expert, row f), split evenly over CTAs.
// k_down_stream:    y[j,d] = W2[e,d,:] . h[j,:] for the CTA's rows d and every
//   slot j, kept in shared memory; then either the gated combine
//   out[t,d] = residual + sum_k gate[t,k] y[inv_perm[t*K+k], d]  (k ascending)
//   or the ungated y_sorted rows are written.
#include "ptx.cuh"

namespace moe {
namespace {

constexpr int kMaxStages = 8;  // = the most consumer warps
constexpr int kMaxThreads = (kMaxStages + 1) * 32;
constexpr int kHeaderBytes = 2048;  // barriers, tags, chunk prefix
constexpr size_t kSmemBudget = 227 * 1024;

struct Header {
    uint64_t full[kMaxStages];
    uint64_t empty[kMaxStages];
    uint64_t vfull[2];   // token vectors (x or h) of a chunk
    uint64_t vempty[2];
    long long tag[kMaxStages];  // task number of the data in each stage
    int prefix[257];
    // one token, rows shared out: each chunk's expert and h row
    int q_e[kStreamMaxSlots], q_j[kStreamMaxSlots];
};
static_assert(sizeof(Header) <= kHeaderBytes, "header too large");

__device__ __forceinline__ void init_header(Header *hd, int n_stages) {
    for (int i = 0; i < n_stages; ++i) {
        ptx::mbar_init(&hd->full[i], 1);
        ptx::mbar_init(&hd->empty[i], 1);
        hd->tag[i] = -1;
    }
    for (int b = 0; b < 2; ++b) {
        ptx::mbar_init(&hd->vfull[b], 1);
        ptx::mbar_init(&hd->vempty[b], n_stages);
    }
    ptx::fence_barrier_init();
}

// 8 bf16 from shared memory -> float[8]
__device__ __forceinline__ void sm8(const bf16 *p, float (&o)[8]) {
    const uint4 u = *reinterpret_cast<const uint4 *>(p);
    unpack_bf16x2(u.x, o[0], o[1]);
    unpack_bf16x2(u.y, o[2], o[3]);
    unpack_bf16x2(u.z, o[4], o[5]);
    unpack_bf16x2(u.w, o[6], o[7]);
}

// Chunk q of the per-expert chunk list: expert, first sorted slot, slots.
template <int NS>
__device__ __forceinline__ void chunk_info(const int *prefix, const int32_t *offsets, int E, int q,
                                           int &e, int &j0, int &ns) {
    e = chunk_expert(prefix, E, q);
    j0 = offsets[e] + (q - prefix[e]) * NS;
    ns = min(NS, offsets[e + 1] - j0);
}

// ---------------------------------------------------------------------------
template <int NS>
__global__ void __launch_bounds__(kMaxThreads, 1)
k_up_glu_stream(int D, int F, int E, int K, int T, const bf16 *__restrict__ x,
                const int32_t *__restrict__ perm, const int32_t *__restrict__ offsets,
                const bf16 *__restrict__ w1, const bf16 *__restrict__ v1, bf16 *__restrict__ h,
                int n_stages, int *ctr, unsigned *err) {
    extern __shared__ __align__(1024) unsigned char smem[];
    Header *hd = reinterpret_cast<Header *>(smem);
    bf16 *xbuf = reinterpret_cast<bf16 *>(smem + kHeaderBytes);  // [2][NS][D]
    bf16 *ring = xbuf + (size_t)2 * NS * D;                        // [n_stages][2][D]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = T * K;
    const int W = n_stages;  // consumer warps; warp W is the producer

    if (threadIdx.x == 0) init_header(hd, n_stages);
    ptx::grid_dependency_wait();  // perm/offsets come from the previous kernel
    // the next kernel's CTAs may launch now (they take the SMs this grid
    // leaves); triggered after the wait, so a CTA of it that starts finds
    // the kernels before this one complete (the down projection reads the
    // dispatch offsets before its own wait)
    ptx::launch_dependents();
    if (warp == 0) chunk_prefix<NS>(offsets, E, S, hd->prefix, err);
    __syncthreads();

    const int Q = hd->prefix[E];
    const long long N = (long long)Q * F;
    if (NS == 1 && T == 1 && ctr != nullptr && Q <= kStreamMaxSlots) {
        // one token, rows shared out as they go: task g = (chunk g / F, row
        // g % F) in batches of n_stages consecutive tasks taken from a
        // counter (zeroed by the routing kernel), the next batch taken while
        // the current one streams -- each SM's share of the memory bandwidth
        // differs by a few percent, and equal static shares left the last
        // SM ~10 us behind the first.  Every chunk holds the same token.
        const uint32_t row_bytes = (uint32_t)D * 2u;
        for (int q = threadIdx.x; q < Q; q += blockDim.x) {
            const int e = chunk_expert(hd->prefix, E, q);
            hd->q_e[q] = e;
            hd->q_j[q] = offsets[e];
        }
        __syncthreads();
        if (warp == W) {
            if (lane != 0) return;
            const uint64_t pol_w = ptx::policy_evict_first();
            ptx::mbar_arrive_expect_tx(&hd->vfull[0], row_bytes);
            ptx::bulk_g2s(xbuf, x, row_bytes, &hd->vfull[0], ptx::policy_evict_last());
            long long i = 0;
            bool ok = true;
            int nxt = atomicAdd(ctr, 1);
            for (;;) {
                const long long g0 = (long long)nxt * n_stages;
                if (g0 >= N) break;
                nxt = atomicAdd(ctr, 1);
                for (int u = 0; u < n_stages && g0 + u < N && ok; ++u, ++i) {
                    const int st = (int)(i % n_stages);
                    if (!(ok = ptx::mbar_wait(&hd->empty[st],
                                              (uint32_t)((i / n_stages) & 1) ^ 1, err)))
                        break;
                    const long long g = g0 + u;
                    const int q = (int)(g / F), f = (int)(g - (long long)q * F);
                    const int e = hd->q_e[q];
                    bf16 *dst = ring + (size_t)st * 2 * D;
                    hd->tag[st] = g;
                    ptx::mbar_arrive_expect_tx(&hd->full[st], 2 * row_bytes);
                    ptx::bulk_g2s(dst, w1 + ((size_t)e * F + f) * D, row_bytes, &hd->full[st],
                                  pol_w);
                    ptx::bulk_g2s(dst + D, v1 + ((size_t)e * F + f) * D, row_bytes,
                                  &hd->full[st], pol_w);
                }
                if (!ok) break;
            }
            // the end, one marker for each consumer warp (its next task)
            for (int w = 0; w < W && ok; ++w, ++i) {
                const int st = (int)(i % n_stages);
                if (!(ok = ptx::mbar_wait(&hd->empty[st], (uint32_t)((i / n_stages) & 1) ^ 1,
                                          err)))
                    break;
                hd->tag[st] = -1;
                ptx::mbar_arrive(&hd->full[st]);
            }
            ptx::mbar_wait(&hd->vfull[0], 0, err);
            return;
        }
        if (!ptx::mbar_wait(&hd->vfull[0], 0, err)) return;
        const int nv = D >> 3;
        for (long long i = warp;; i += W) {
            const int st = warp;
            if (!ptx::mbar_wait(&hd->full[st], (uint32_t)((i / n_stages) & 1), err)) return;
            const long long g = hd->tag[st];
            if (g < 0) return;
            const int q = (int)(g / F), f = (int)(g - (long long)q * F);
            const int jq = hd->q_j[q];
            const bf16 *wr = ring + (size_t)st * 2 * D;
            const bf16 *vr = wr + D;
            float a = 0.f, bb = 0.f;
#pragma unroll 2
            for (int v = lane; v < nv; v += 32) {
                float wv[8], vv[8], xv[8];
                sm8(wr + v * 8, wv);
                sm8(vr + v * 8, vv);
                sm8(xbuf + v * 8, xv);
#pragma unroll
                for (int k = 0; k < 8; ++k) {
                    a = fmaf(wv[k], xv[k], a);
                    bb = fmaf(vv[k], xv[k], bb);
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->empty[st]);
            const float as = warp_sum(a), bs = warp_sum(bb);
            if (lane == 0) h[(size_t)jq * F + f] = __float2bfloat16_rn(silu(as) * bs);
        }
    }
    const long long lo = N * blockIdx.x / gridDim.x;
    const long long hi = N * (blockIdx.x + 1) / gridDim.x;
    if (lo >= hi) return;
    const int q_first = (int)(lo / F), q_last = (int)((hi - 1) / F);
    const uint32_t row_bytes = (uint32_t)D * 2u;

    if (warp == W) {
        if (lane != 0) return;
        const uint64_t pol_w = ptx::policy_evict_first();
        const uint64_t pol_x = ptx::policy_evict_last();
        long long i = 0;
        bool ok = true;
        for (int q = q_first; q <= q_last && ok; ++q) {
            int e, j0, ns;
            chunk_info<NS>(hd->prefix, offsets, E, q, e, j0, ns);
            const int qi = q - q_first, b = qi & 1;
            if (!(ok = ptx::mbar_wait(&hd->vempty[b], ((qi >> 1) & 1) ^ 1, err))) break;
            ptx::mbar_arrive_expect_tx(&hd->vfull[b], (uint32_t)ns * row_bytes);
            for (int s = 0; s < ns; ++s) {
                int slot = perm[j0 + s];
                if (slot < 0 || slot >= S) { set_error(err, kErrIndex); slot = 0; }
                ptx::bulk_g2s(xbuf + ((size_t)b * NS + s) * D, x + (size_t)(slot / K) * D,
                              row_bytes, &hd->vfull[b], pol_x);
            }
            const long long f_lo = max(lo, (long long)q * F) - (long long)q * F;
            const long long f_hi = min(hi, (long long)(q + 1) * F) - (long long)q * F;
            for (long long f = f_lo; f < f_hi; ++f, ++i) {
                const int st = (int)(i % n_stages);
                if (!(ok = ptx::mbar_wait(&hd->empty[st], (uint32_t)((i / n_stages) & 1) ^ 1, err)))
                    break;
                bf16 *dst = ring + (size_t)st * 2 * D;
                hd->tag[st] = i;
                ptx::mbar_arrive_expect_tx(&hd->full[st], 2 * row_bytes);
                ptx::bulk_g2s(dst, w1 + ((size_t)e * F + f) * D, row_bytes, &hd->full[st], pol_w);
                ptx::bulk_g2s(dst + D, v1 + ((size_t)e * F + f) * D, row_bytes, &hd->full[st], pol_w);
            }
        }
        // Before leaving, let every copy still in flight land (on the normal
        // path the consumers have already waited for all of them).
        const long long n_issued = i;
        for (long long k = (n_issued > n_stages ? n_issued - n_stages : 0); k < n_issued; ++k)
            ptx::mbar_wait(&hd->full[k % n_stages], (uint32_t)((k / n_stages) & 1), err);
        return;
    }

    // consumer warps
    long long i = 0;
    const int nv = D >> 3;
    for (int q = q_first; q <= q_last; ++q) {
        int e, j0, ns;
        chunk_info<NS>(hd->prefix, offsets, E, q, e, j0, ns);
        const int qi = q - q_first, b = qi & 1;
        if (!ptx::mbar_wait(&hd->vfull[b], (qi >> 1) & 1, err)) return;
        const bf16 *xs = xbuf + (size_t)b * NS * D;
        const long long f_lo = max(lo, (long long)q * F) - (long long)q * F;
        const long long f_hi = min(hi, (long long)(q + 1) * F) - (long long)q * F;
        for (long long f = f_lo; f < f_hi; ++f, ++i) {
            if ((int)(i % W) != warp) continue;
            const int st = warp;
            if (!ptx::mbar_wait(&hd->full[st], (uint32_t)((i / n_stages) & 1), err)) return;
            if (hd->tag[st] != i) {  // pipeline out of step: record and stop
                set_error(err, kErrTimeout);
                return;
            }
            const bf16 *wr = ring + (size_t)st * 2 * D;
            const bf16 *vr = wr + D;
            float a[NS], bb[NS];
#pragma unroll
            for (int s = 0; s < NS; ++s) a[s] = bb[s] = 0.f;
#pragma unroll 2
            for (int v = lane; v < nv; v += 32) {
                float wv[8], vv[8];
                sm8(wr + v * 8, wv);
                sm8(vr + v * 8, vv);
#pragma unroll
                for (int s = 0; s < NS; ++s) {
                    if (s < ns) {
                        float xv[8];
                        sm8(xs + (size_t)s * D + v * 8, xv);
#pragma unroll
                        for (int k = 0; k < 8; ++k) {
                            a[s] = fmaf(wv[k], xv[k], a[s]);
                            bb[s] = fmaf(vv[k], xv[k], bb[s]);
                        }
                    }
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->empty[st]);
#pragma unroll
            for (int s = 0; s < NS; ++s) {
                if (s < ns) {
                    const float as = warp_sum(a[s]), bs = warp_sum(bb[s]);
                    if (lane == 0) h[(size_t)(j0 + s) * F + f] = __float2bfloat16_rn(silu(as) * bs);
                }
            }
        }
        __syncwarp();
        if (lane == 0) ptx::mbar_arrive(&hd->vempty[b]);
    }
}

// ---------------------------------------------------------------------------
template <int NS, typename TO, typename TR, bool FUSED>
__global__ void __launch_bounds__(kMaxThreads, 1)
k_down_stream(int D, int F, int E, int K, int T, const bf16 *__restrict__ h,
              const int32_t *__restrict__ offsets, const int32_t *__restrict__ inv_perm,
              const bf16 *__restrict__ w2, const float *__restrict__ gate,
              const TR *__restrict__ residual, TO *__restrict__ out, float *__restrict__ y_sorted,
              int n_stages, int rows_max, unsigned *err) {
    extern __shared__ __align__(1024) unsigned char smem[];
    Header *hd = reinterpret_cast<Header *>(smem);
    bf16 *hbuf = reinterpret_cast<bf16 *>(smem + kHeaderBytes);  // [2][NS][F]
    bf16 *ring = hbuf + (size_t)2 * NS * F;                        // [n_stages][F]
    float *ylocal = reinterpret_cast<float *>(ring + (size_t)n_stages * F);  // [S][rows_max]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = T * K;
    const int W = n_stages;  // consumer warps; warp W is the producer

    if (threadIdx.x == 0) init_header(hd, n_stages);
    ptx::launch_dependents();  // as in k_up_glu_stream
    // the dispatch offsets come from a kernel before the previous one (the
    // up projection lets this grid launch only after its own dependency
    // wait), W2 from none: half the stages' weight rows go out before the
    // wait for the hidden vectors (all of them queue the hidden vectors
    // behind more weight bytes than the overlap gains: one-token layer step
    // 237.3 / 236.0 / 235.8 / 236.0 us for 0 / 2 / 4 / 8 stages, same box)
    if (warp == 0) chunk_prefix<NS>(offsets, E, S, hd->prefix, err);
    __syncthreads();

    const int Q = hd->prefix[E];
    const int r0 = (int)((long long)D * blockIdx.x / gridDim.x);
    const int r1 = (int)((long long)D * (blockIdx.x + 1) / gridDim.x);
    const int R = r1 - r0;
    const uint32_t row_bytes = (uint32_t)F * 2u;
    long long n_pre = 0;  // tasks whose weight row was sent before the wait
    if (warp == W && lane == 0 && R > 0) {
        const uint64_t pol_w = ptx::policy_evict_first();
        for (int q = 0; q < Q && n_pre < n_stages / 2; ++q) {
            int e, j0, ns;
            chunk_info<NS>(hd->prefix, offsets, E, q, e, j0, ns);
            for (int r = 0; r < R && n_pre < n_stages / 2; ++r, ++n_pre) {
                const int st = (int)n_pre;
                hd->tag[st] = n_pre;
                ptx::mbar_arrive_expect_tx(&hd->full[st], row_bytes);
                ptx::bulk_g2s(ring + (size_t)st * F, w2 + ((size_t)e * D + r0 + r) * F, row_bytes,
                              &hd->full[st], pol_w);
            }
        }
    }
    ptx::grid_dependency_wait();  // h comes from the previous kernel
    if (R <= 0) return;

    if (warp == W) {
        if (lane != 0) return;
        const uint64_t pol_w = ptx::policy_evict_first();
        const uint64_t pol_h = ptx::policy_evict_last();
        long long i = 0;
        bool ok = true;
        for (int q = 0; q < Q && ok; ++q) {
            int e, j0, ns;
            chunk_info<NS>(hd->prefix, offsets, E, q, e, j0, ns);
            const int b = q & 1;
            if (!(ok = ptx::mbar_wait(&hd->vempty[b], ((q >> 1) & 1) ^ 1, err))) break;
            ptx::mbar_arrive_expect_tx(&hd->vfull[b], (uint32_t)ns * row_bytes);
            ptx::bulk_g2s(hbuf + (size_t)b * NS * F, h + (size_t)j0 * F, (uint32_t)ns * row_bytes,
                          &hd->vfull[b], pol_h);
            for (int r = 0; r < R; ++r, ++i) {
                if (i < n_pre) continue;  // sent before the dependency wait
                const int st = (int)(i % n_stages);
                if (!(ok = ptx::mbar_wait(&hd->empty[st], (uint32_t)((i / n_stages) & 1) ^ 1, err)))
                    break;
                hd->tag[st] = i;
                ptx::mbar_arrive_expect_tx(&hd->full[st], row_bytes);
                ptx::bulk_g2s(ring + (size_t)st * F, w2 + ((size_t)e * D + r0 + r) * F, row_bytes,
                              &hd->full[st], pol_w);
            }
        }
        const long long n_issued = i;
        for (long long k = (n_issued > n_stages ? n_issued - n_stages : 0); k < n_issued; ++k)
            ptx::mbar_wait(&hd->full[k % n_stages], (uint32_t)((k / n_stages) & 1), err);
        return;
    }

    long long i = 0;
    const int nv = F >> 3;
    bool ok = true;
    for (int q = 0; q < Q && ok; ++q) {
        int e, j0, ns;
        chunk_info<NS>(hd->prefix, offsets, E, q, e, j0, ns);
        const int b = q & 1;
        if (!(ok = ptx::mbar_wait(&hd->vfull[b], (q >> 1) & 1, err))) break;
        const bf16 *hs = hbuf + (size_t)b * NS * F;
        for (int r = 0; r < R; ++r, ++i) {
            if ((int)(i % W) != warp) continue;
            const int st = warp;
            if (!(ok = ptx::mbar_wait(&hd->full[st], (uint32_t)((i / n_stages) & 1), err))) break;
            if (hd->tag[st] != i) {  // pipeline out of step: record and stop
                set_error(err, kErrTimeout);
                ok = false;
                break;
            }
            const bf16 *wr = ring + (size_t)st * F;
            float acc[NS];
#pragma unroll
            for (int s = 0; s < NS; ++s) acc[s] = 0.f;
#pragma unroll 2
            for (int v = lane; v < nv; v += 32) {
                float wv[8];
                sm8(wr + v * 8, wv);
#pragma unroll
                for (int s = 0; s < NS; ++s) {
                    if (s < ns) {
                        float hv[8];
                        sm8(hs + (size_t)s * F + v * 8, hv);
#pragma unroll
                        for (int k = 0; k < 8; ++k) acc[s] = fmaf(wv[k], hv[k], acc[s]);
                    }
                }
            }
            __syncwarp();
            if (lane == 0) ptx::mbar_arrive(&hd->empty[st]);
#pragma unroll
            for (int s = 0; s < NS; ++s) {
                if (s < ns) {
                    const float y = warp_sum(acc[s]);
                    if (lane == 0) ylocal[(size_t)(j0 + s) * rows_max + r] = y;
                }
            }
        }
        __syncwarp();
        if (ok && lane == 0) ptx::mbar_arrive(&hd->vempty[b]);
    }
    // all consumer warps have written their rows of ylocal
    ptx::named_bar_sync(1, W * 32);
    if (!ok) return;
    const int tid = threadIdx.x;
    if (FUSED) {
        // only the slots of this launch's experts (sorted positions
        // [offsets[0], offsets[E]): all of them for the whole layer, one
        // node's share for an expert range) hold a row of ylocal
        const int j_lo = offsets[0], j_hi = offsets[E];
        for (int idx = tid; idx < T * R; idx += W * 32) {
            const int t = idx / R, r = idx - t * R;
            float v = 0.f;
            for (int k = 0; k < K; ++k) {
                const int j = inv_perm[(size_t)t * K + k];
                if (j < j_lo || j >= j_hi || j < 0 || j >= S) continue;
                v = fmaf(gate[(size_t)t * K + k], ylocal[(size_t)j * rows_max + r], v);
            }
            if (residual) v += to_f(residual[(size_t)t * D + r0 + r]);
            out[(size_t)t * D + r0 + r] = from_f<TO>(v);
        }
    } else {
        for (int idx = tid; idx < S * R; idx += W * 32) {
            const int j = idx / R, r = idx - j * R;
            y_sorted[(size_t)j * D + r0 + r] = ylocal[(size_t)j * rows_max + r];
        }
    }
}

// ---- host side ---------------------------------------------------------------

template <typename Kern>
cudaError_t set_smem(Kern kern, size_t bytes) {
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes);
}

struct UpPlan { int ns, n_stages; size_t smem; };
struct DownPlan { int ns, n_stages, rows_max; size_t smem; };

// Slots per chunk: an expert holds at most T slots (a token picks distinct
// experts), so a batch of at most kStreamMaxTokens tokens needs a token-vector
// buffer of kStreamMaxTokens rows and leaves the rest of shared memory for
// weight stages.
constexpr int kNs = kStreamMaxTokens;

bool plan_up(const moe_dims &d, int T, UpPlan &p) {
    (void)T;
    p.ns = kNs;
    const size_t fixed = kHeaderBytes + (size_t)2 * p.ns * d.d_model * 2;
    const size_t stage = (size_t)2 * d.d_model * 2;
    if (fixed + 2 * stage > kSmemBudget) return false;
    p.n_stages = (int)std::min<size_t>(kMaxStages, (kSmemBudget - fixed) / stage);
    p.smem = fixed + p.n_stages * stage;
    return true;
}

bool plan_down(const moe_dims &d, int T, int grid, DownPlan &p) {
    const int S = T * d.top_k;
    p.ns = kNs;
    p.rows_max = (d.d_model + grid - 1) / grid;
    const size_t fixed = kHeaderBytes + (size_t)2 * p.ns * d.ffn_hidden * 2 +
                         (((size_t)S * p.rows_max * 4 + 15) & ~size_t(15));
    const size_t stage = (size_t)d.ffn_hidden * 2;
    if (fixed + 2 * stage > kSmemBudget) return false;
    p.n_stages = (int)std::min<size_t>(kMaxStages, (kSmemBudget - fixed) / stage);
    p.smem = fixed + p.n_stages * stage;
    return true;
}

}  // namespace

bool stream_path_ok(const moe_dims &d, int T) {
    if (d.w_dtype != MOE_BF16 || d.x_dtype != MOE_BF16) return false;
    if (T < 1 || T > kStreamMaxTokens || T * d.top_k > kStreamMaxSlots) return false;
    const int grid = device_info().sm_count;
    UpPlan up;
    DownPlan dn;
    return plan_up(d, T, up) && plan_down(d, T, std::min(grid, d.d_model), dn);
}

cudaError_t launch_up_glu_stream(const moe_dims &d, int T, const void *x, const int32_t *perm,
                                 const int32_t *offsets, const void *w1, const void *v1, void *h,
                                 cudaStream_t st, int *ctr) {
    UpPlan p;
    if (!plan_up(d, T, p)) return cudaErrorInvalidValue;
    const void *kern = (const void *)k_up_glu_stream<kNs>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)p.smem);
    if (e != cudaSuccess) return e;
    int D = d.d_model, F = d.ffn_hidden, E = d.n_experts, K = d.top_k, Tv = T, ns = p.n_stages;
    const bf16 *xp = static_cast<const bf16 *>(x);
    const bf16 *w1p = static_cast<const bf16 *>(w1);
    const bf16 *v1p = static_cast<const bf16 *>(v1);
    bf16 *hp = static_cast<bf16 *>(h);
    unsigned *err = device_info().err;
    int *cp = T == 1 ? ctr : nullptr;
    void *args[] = {&D, &F, &E, &K, &Tv, &xp, &perm, &offsets, &w1p, &v1p, &hp, &ns, &cp, &err};
    LaunchScope ls("up_glu_stream", st);
    return launch_pdl(kern, dim3(device_info().sm_count), dim3((p.n_stages + 1) * 32), p.smem, st,
                      args);
}

template <typename TO, typename TR, bool FUSED>
cudaError_t down_stream_impl(const moe_dims &d, int T, const void *h, const int32_t *offsets,
                             const int32_t *inv_perm, const void *w2, const float *gate,
                             const void *residual, void *out, float *y_sorted, cudaStream_t st) {
    const int grid = std::min(device_info().sm_count, d.d_model);
    DownPlan p;
    if (!plan_down(d, T, grid, p)) return cudaErrorInvalidValue;
    const void *kern = (const void *)k_down_stream<kNs, TO, TR, FUSED>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)p.smem);
    if (e != cudaSuccess) return e;
    int D = d.d_model, F = d.ffn_hidden, E = d.n_experts, K = d.top_k, Tv = T;
    int ns = p.n_stages, rows_max = p.rows_max;
    const bf16 *hp = static_cast<const bf16 *>(h);
    const bf16 *w2p = static_cast<const bf16 *>(w2);
    const TR *rp = static_cast<const TR *>(residual);
    TO *op = static_cast<TO *>(out);
    unsigned *err = device_info().err;
    void *args[] = {&D, &F, &E, &K, &Tv, &hp, &offsets, &inv_perm, &w2p, &gate, &rp, &op,
                    &y_sorted, &ns, &rows_max, &err};
    LaunchScope ls(FUSED ? "down_combine_stream" : "down_stream", st);
    return launch_pdl(kern, dim3(grid), dim3((p.n_stages + 1) * 32), p.smem, st, args);
}

cudaError_t launch_down_stream(const moe_dims &d, int T, const void *h, const int32_t *offsets,
                               const int32_t *inv_perm, const void *w2, const float *gate,
                               const void *residual, void *out, float *y_sorted, bool fused,
                               cudaStream_t st) {
    if (!fused)
        return down_stream_impl<float, bf16, false>(d, T, h, offsets, inv_perm, w2, gate, nullptr,
                                                    nullptr, y_sorted, st);
    if (d.out_dtype == MOE_BF16)
        return down_stream_impl<bf16, bf16, true>(d, T, h, offsets, inv_perm, w2, gate, residual,
                                                  out, nullptr, st);
    return down_stream_impl<float, float, true>(d, T, h, offsets, inv_perm, w2, gate, residual, out,
                                               nullptr, st);
}

}  // namespace moe
