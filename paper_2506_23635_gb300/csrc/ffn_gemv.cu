// Weight-streaming expert FFN for few tokens per expert (decode).
//
// Table 1 notes (d),(e) of arxiv 2506.23635: an expert is three
// D_embed x D_ffn matrices (w1, v1, w2); Sec. 4.4 observes that for token
// generation the time is the weight load, not the arithmetic.  So these
// kernels read every selected expert's weights exactly once per call, with
// 16-byte streaming loads, and apply each weight row to all the slots routed
// to that expert:
//
//   k_up_glu_gemv:  h[j,f] = SiLU(W1[e,f,:] . x_j) * (V1[e,f,:] . x_j)
//   k_down_gemv:    y[j,d] = W2[e,d,:] . h[j,:]           (unfused), or
//                   out[t,d] = residual + sum over t's slots of gate * y
//                                                        (fused combine)
//
// j runs over the sorted slots of expert e (offsets[e] <= j < offsets[e+1]),
// x_j = x[perm[j] / K].  Accumulation is fp32; a row is split across the 32
// lanes of a warp and reduced with shuffles.
#include "moe_internal.cuh"

namespace moe {
namespace {

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kRowsPerWarp = 2;                   // up kernel: rows per warp
constexpr int kRowsPerUnit = kWarps * kRowsPerWarp;  // up kernel: rows per work unit

// Exclusive scan over experts of ceil(n_e / NS), written to prefix[0..E].
// Executed by warp 0 of the block; E <= 256.
template <typename TX, typename TW, int NS>
__global__ void __launch_bounds__(kThreads)
k_up_glu_gemv(int D, int F, int E, int K, int T, const TX *__restrict__ x,
              const int32_t *__restrict__ perm, const int32_t *__restrict__ offsets,
              const TW *__restrict__ w1, const TW *__restrict__ v1,
              float *__restrict__ h, unsigned *err) {
    extern __shared__ float4 smem_f4[];
    float *xs = reinterpret_cast<float *>(smem_f4);  // [NS][D] fp32 token vectors
    __shared__ int prefix[257];

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int S = T * K;
    if (warp == 0) chunk_prefix<NS>(offsets, E, S, prefix, err);
    __syncthreads();

    const int n_fb = (F + kRowsPerUnit - 1) / kRowsPerUnit;
    const long long total = (long long)prefix[E] * n_fb;
    const int nv = D >> 3;  // 8-element vectors per row
    int cur_chunk = -1, e = 0, j0 = 0, ns = 0;

    for (long long u = blockIdx.x; u < total; u += gridDim.x) {
        const int chunk = (int)(u / n_fb);
        const int fb = (int)(u - (long long)chunk * n_fb);
        if (chunk != cur_chunk) {  // uniform across the block
            int lo = 0, hi = E - 1;  // largest e with prefix[e] <= chunk
            while (lo < hi) {
                int mid = (lo + hi + 1) >> 1;
                if (prefix[mid] <= chunk) lo = mid; else hi = mid - 1;
            }
            e = lo;
            j0 = offsets[e] + (chunk - prefix[e]) * NS;
            ns = min(NS, offsets[e + 1] - j0);
            __syncthreads();  // previous token vectors no longer in use
            for (int s = 0; s < ns; ++s) {
                int slot = perm[j0 + s];
                if (slot < 0 || slot >= S) {
                    set_error(err, kErrIndex);
                    slot = 0;
                }
                const TX *xr = x + (size_t)(slot / K) * D;
                for (int v = threadIdx.x; v < nv; v += kThreads) {
                    float t8[8];
                    load8(xr + (size_t)v * 8, t8);
                    float4 *dst = reinterpret_cast<float4 *>(xs + (size_t)s * D + v * 8);
                    dst[0] = make_float4(t8[0], t8[1], t8[2], t8[3]);
                    dst[1] = make_float4(t8[4], t8[5], t8[6], t8[7]);
                }
            }
            __syncthreads();
            cur_chunk = chunk;
        }

        const int f0 = fb * kRowsPerUnit + warp * kRowsPerWarp;
        if (f0 >= F) continue;
        const bool two = (f0 + 1) < F;
        const TW *a0 = w1 + ((size_t)e * F + f0) * D;
        const TW *b0 = v1 + ((size_t)e * F + f0) * D;
        const TW *a1 = two ? a0 + D : a0;
        const TW *b1 = two ? b0 + D : b0;

        float acc_a0[NS], acc_a1[NS], acc_b0[NS], acc_b1[NS];
#pragma unroll
        for (int s = 0; s < NS; ++s) acc_a0[s] = acc_a1[s] = acc_b0[s] = acc_b1[s] = 0.f;

#pragma unroll 2
        for (int v = lane; v < nv; v += 32) {
            float wa0[8], wa1[8], wb0[8], wb1[8];
            stream8(a0 + (size_t)v * 8, wa0);
            stream8(b0 + (size_t)v * 8, wb0);
            stream8(a1 + (size_t)v * 8, wa1);
            stream8(b1 + (size_t)v * 8, wb1);
#pragma unroll
            for (int s = 0; s < NS; ++s) {
                if (s < ns) {
                    const float4 *xp = reinterpret_cast<const float4 *>(xs + (size_t)s * D + v * 8);
                    const float4 p = xp[0], q = xp[1];
                    const float xv[8] = {p.x, p.y, p.z, p.w, q.x, q.y, q.z, q.w};
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        acc_a0[s] = fmaf(wa0[i], xv[i], acc_a0[s]);
                        acc_b0[s] = fmaf(wb0[i], xv[i], acc_b0[s]);
                        acc_a1[s] = fmaf(wa1[i], xv[i], acc_a1[s]);
                        acc_b1[s] = fmaf(wb1[i], xv[i], acc_b1[s]);
                    }
                }
            }
        }
#pragma unroll
        for (int s = 0; s < NS; ++s) {
            if (s < ns) {
                const float a0s = warp_sum(acc_a0[s]), b0s = warp_sum(acc_b0[s]);
                const float a1s = warp_sum(acc_a1[s]), b1s = warp_sum(acc_b1[s]);
                if (lane == 0) {
                    float *hr = h + (size_t)(j0 + s) * F + f0;
                    hr[0] = silu(a0s) * b0s;
                    if (two) hr[1] = silu(a1s) * b1s;
                }
            }
        }
    }
}

// One warp per output row d; the block owns kWarps consecutive rows and
// visits every expert in ascending order, so each token's sum has a fixed
// order.  FUSED: out[t,d] = residual[t,d] + sum gate * y (T <= 64 tokens).
template <typename TW, typename TO, typename TR, int NS, bool FUSED>
__global__ void __launch_bounds__(kThreads)
k_down_gemv(int D, int F, int E, int K, int T, const float *__restrict__ h,
            const int32_t *__restrict__ perm, const int32_t *__restrict__ offsets,
            const TW *__restrict__ w2, const float *__restrict__ gate,
            float *__restrict__ y_sorted, const TR *__restrict__ residual,
            TO *__restrict__ out, unsigned *err) {
    __shared__ float oacc[kWarps][FUSED ? kFusedCombineMaxTokens : 1];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int d = blockIdx.x * kWarps + warp;
    if (d >= D) return;  // whole warp leaves; no block-wide sync below
    if (FUSED)
        for (int t = lane; t < T; t += 32) oacc[warp][t] = 0.f;
    __syncwarp();
    const int nv = F >> 3;
    const int S = T * K;
    for (int e = 0; e < E; ++e) {
        const int jb = offsets[e], je = offsets[e + 1];
        if (jb < 0 || je < jb || je > S) {  // corrupt offsets: record, skip
            if (lane == 0) set_error(err, kErrIndex);
            continue;
        }
        if (jb == je) continue;
        const TW *row = w2 + ((size_t)e * D + d) * F;
        for (int j0 = jb; j0 < je; j0 += NS) {
            const int ns = min(NS, je - j0);
            float acc[NS];
#pragma unroll
            for (int s = 0; s < NS; ++s) acc[s] = 0.f;
#pragma unroll 2
            for (int v = lane; v < nv; v += 32) {
                float w[8];
                stream8(row + (size_t)v * 8, w);
#pragma unroll
                for (int s = 0; s < NS; ++s) {
                    if (s < ns) {
                        float hv[8];
                        load8(h + (size_t)(j0 + s) * F + (size_t)v * 8, hv);
#pragma unroll
                        for (int i = 0; i < 8; ++i) acc[s] = fmaf(w[i], hv[i], acc[s]);
                    }
                }
            }
#pragma unroll
            for (int s = 0; s < NS; ++s) {
                if (s < ns) {
                    const float y = warp_sum(acc[s]);
                    if (lane == 0) {
                        if (FUSED) {
                            const int slot = perm[j0 + s];
                            if (slot >= 0 && slot < S) oacc[warp][slot / K] += gate[slot] * y;
                            else set_error(err, kErrIndex);
                        } else {
                            y_sorted[(size_t)(j0 + s) * D + d] = y;
                        }
                    }
                }
            }
        }
    }
    if (FUSED) {
        __syncwarp();
        for (int t = lane; t < T; t += 32) {
            float v = oacc[warp][t];
            if (residual) v += to_f(residual[(size_t)t * D + d]);
            out[(size_t)t * D + d] = from_f<TO>(v);
        }
    }
}

constexpr int kUpSlots = 4;    // slots sharing one pass over an up-projection row
constexpr size_t kUpSmemBudget = 200 * 1024;
constexpr int kDownSlots = 4;  // slots sharing one pass over a down-projection row

template <typename TX, typename TW, int NS>
cudaError_t up_impl(const moe_dims &d, int T, const void *x, const int32_t *perm,
                    const int32_t *offsets, const void *w1, const void *v1, float *h,
                    cudaStream_t st) {
    const int D = d.d_model, F = d.ffn_hidden, E = d.n_experts, K = d.top_k;
    const int S = T * K;
    const size_t smem = (size_t)NS * D * sizeof(float);
    auto kern = k_up_glu_gemv<TX, TW, NS>;
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    // per device: the largest dynamic shared memory configured so far and the
    // resulting residency
    static size_t configured_smem[64];
    static int blocks_per_sm[64];
    if (dev >= 64) return cudaErrorInvalidDevice;
    if (configured_smem[dev] < smem) {
        err = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (err != cudaSuccess) return err;
        configured_smem[dev] = smem;
    }
    err = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&blocks_per_sm[dev], kern, kThreads, smem);
    if (err != cudaSuccess) return err;
    const int bps = blocks_per_sm[dev] < 1 ? 1 : blocks_per_sm[dev];
    const int n_fb = (F + kRowsPerUnit - 1) / kRowsPerUnit;
    const long long max_units = (long long)(S / NS + E) * n_fb;
    const long long cap = (long long)device_info().sm_count * bps;
    const int grid = (int)(max_units < cap ? max_units : cap);
    if (grid <= 0) return cudaSuccess;
    LaunchScope ls("up_glu_gemv", st);
    kern<<<grid, kThreads, smem, st>>>(D, F, E, K, T, static_cast<const TX *>(x), perm, offsets,
                                      static_cast<const TW *>(w1), static_cast<const TW *>(v1), h,
                                      device_info().err);
    return cudaGetLastError();
}

template <typename TW, typename TO, typename TR>
cudaError_t down_impl(const moe_dims &d, int T, const float *h, const int32_t *perm,
                      const int32_t *offsets, const void *w2, const float *gate,
                      float *y_sorted, const void *residual, void *out, bool fused,
                      cudaStream_t st) {
    const int D = d.d_model, F = d.ffn_hidden, E = d.n_experts, K = d.top_k;
    const int grid = (D + kWarps - 1) / kWarps;
    if (fused) {
        LaunchScope ls("down_combine_gemv", st);
        k_down_gemv<TW, TO, TR, kDownSlots, true><<<grid, kThreads, 0, st>>>(
            D, F, E, K, T, h, perm, offsets, static_cast<const TW *>(w2), gate, nullptr,
            static_cast<const TR *>(residual), static_cast<TO *>(out), device_info().err);
    } else {
        LaunchScope ls("down_gemv", st);
        k_down_gemv<TW, float, float, kDownSlots, false><<<grid, kThreads, 0, st>>>(
            D, F, E, K, T, h, perm, offsets, static_cast<const TW *>(w2), gate, y_sorted,
            nullptr, nullptr, device_info().err);
    }
    return cudaGetLastError();
}

}  // namespace

cudaError_t launch_up_glu_gemv(const moe_dims &d, int T, const void *x, const int32_t *perm,
                               const int32_t *offsets, const void *w1, const void *v1,
                               float *h, cudaStream_t st) {
    // kUpSlots token vectors of D floats must fit in shared memory
    const bool wide = (size_t)kUpSlots * d.d_model * sizeof(float) > kUpSmemBudget;
    if (d.w_dtype == MOE_BF16)
        return wide ? up_impl<bf16, bf16, 1>(d, T, x, perm, offsets, w1, v1, h, st)
                    : up_impl<bf16, bf16, kUpSlots>(d, T, x, perm, offsets, w1, v1, h, st);
    return wide ? up_impl<float, float, 1>(d, T, x, perm, offsets, w1, v1, h, st)
                : up_impl<float, float, kUpSlots>(d, T, x, perm, offsets, w1, v1, h, st);
}

cudaError_t launch_down_gemv(const moe_dims &d, int T, const float *h, const int32_t *perm,
                             const int32_t *offsets, const void *w2, const float *gate,
                             float *y_sorted, const void *residual, void *out, bool fused,
                             cudaStream_t st) {
    const bool wb = d.w_dtype == MOE_BF16, ob = d.out_dtype == MOE_BF16;
    if (!fused) {
        if (wb) return down_impl<bf16, float, float>(d, T, h, perm, offsets, w2, gate, y_sorted,
                                                     nullptr, nullptr, false, st);
        return down_impl<float, float, float>(d, T, h, perm, offsets, w2, gate, y_sorted,
                                              nullptr, nullptr, false, st);
    }
    // the residual has the output's dtype
    if (wb && ob) return down_impl<bf16, bf16, bf16>(d, T, h, perm, offsets, w2, gate, nullptr, residual, out, true, st);
    if (wb) return down_impl<bf16, float, float>(d, T, h, perm, offsets, w2, gate, nullptr, residual, out, true, st);
    if (ob) return down_impl<float, bf16, bf16>(d, T, h, perm, offsets, w2, gate, nullptr, residual, out, true, st);
    return down_impl<float, float, float>(d, T, h, perm, offsets, w2, gate, nullptr, residual, out, true, st);
}

}  // namespace moe
