// Internal helpers shared by the CUDA translation units of libmoe.
// Nothing here is part of the C ABI (include/moe.h).
#pragma once

#include <algorithm>

#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "moe.h"

namespace moe {

typedef __nv_bfloat16 bf16;

// Device error word: the first error a kernel meets is stored here with an
// atomic compare-and-swap and read back by moe_get_last_error.
enum : unsigned { kErrNone = 0, kErrIndex = 1, kErrTimeout = 2 };

__device__ __forceinline__ void set_error(unsigned *err, unsigned code) {
    if (err) atomicCAS(err, 0u, code);
}

__device__ __forceinline__ float to_f(float v) { return v; }
__device__ __forceinline__ float to_f(bf16 v) { return __bfloat162float(v); }

template <typename T> __device__ __forceinline__ T from_f(float v);
template <> __device__ __forceinline__ float from_f<float>(float v) { return v; }
template <> __device__ __forceinline__ bf16 from_f<bf16>(float v) { return __float2bfloat16_rn(v); }

// Two bf16 packed in a 32-bit word -> two floats (exact).
__device__ __forceinline__ void unpack_bf16x2(uint32_t u, float &lo, float &hi) {
    lo = __uint_as_float(u << 16);
    hi = __uint_as_float(u & 0xffff0000u);
}

// 16-byte read-only load that does not allocate in L1 (weights are streamed
// once per call; keeping them out of L1 leaves it to the token vectors).
__device__ __forceinline__ uint4 ld_stream16(const void *p) {
    uint4 r;
    asm("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
        : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
        : "l"(p));
    return r;
}

// Eight consecutive weights (streamed) -> float[8].
__device__ __forceinline__ void stream8(const bf16 *p, float (&o)[8]) {
    uint4 u = ld_stream16(p);
    unpack_bf16x2(u.x, o[0], o[1]);
    unpack_bf16x2(u.y, o[2], o[3]);
    unpack_bf16x2(u.z, o[4], o[5]);
    unpack_bf16x2(u.w, o[6], o[7]);
}
__device__ __forceinline__ void stream8(const float *p, float (&o)[8]) {
    uint4 a = ld_stream16(p), b = ld_stream16(p + 4);
    o[0] = __uint_as_float(a.x); o[1] = __uint_as_float(a.y);
    o[2] = __uint_as_float(a.z); o[3] = __uint_as_float(a.w);
    o[4] = __uint_as_float(b.x); o[5] = __uint_as_float(b.y);
    o[6] = __uint_as_float(b.z); o[7] = __uint_as_float(b.w);
}

// Eight consecutive values through the normal cached path -> float[8].
__device__ __forceinline__ void load8(const bf16 *p, float (&o)[8]) {
    uint4 u = __ldg(reinterpret_cast<const uint4 *>(p));
    unpack_bf16x2(u.x, o[0], o[1]);
    unpack_bf16x2(u.y, o[2], o[3]);
    unpack_bf16x2(u.z, o[4], o[5]);
    unpack_bf16x2(u.w, o[6], o[7]);
}
__device__ __forceinline__ void load8(const float *p, float (&o)[8]) {
    float4 a = __ldg(reinterpret_cast<const float4 *>(p));
    float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
    o[0] = a.x; o[1] = a.y; o[2] = a.z; o[3] = a.w;
    o[4] = b.x; o[5] = b.y; o[6] = b.z; o[7] = b.w;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

__device__ __forceinline__ float silu(float a) { return a / (1.0f + expf(-a)); }

// An expert whose slot range is not inside [0, S] is recorded as an index
// error and given no work, so a corrupt offsets array cannot move an access
// out of bounds.
template <int NS>
__device__ __forceinline__ void chunk_prefix(const int32_t *offsets, int E, int S, int *prefix,
                             unsigned *err) {
    const int lane = threadIdx.x & 31;
    int run = 0;
    for (int base = 0; base < E; base += 32) {
        int e = base + lane;
        int c = 0;
        if (e < E) {
            const int lo = offsets[e], hi = offsets[e + 1];
            if (lo < 0 || hi < lo || hi > S) set_error(err, kErrIndex);
            else c = (hi - lo + NS - 1) / NS;
        }
        int incl = c;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int v = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += v;
        }
        if (e < E) prefix[e] = run + incl - c;
        run += __shfl_sync(0xffffffffu, incl, 31);
    }
    if (lane == 0) prefix[E] = run;
}


// Expert e of chunk q: the largest e with prefix[e] <= q (prefix from
// chunk_prefix; experts without chunks have prefix[e] == prefix[e+1]).
__device__ __forceinline__ int chunk_expert(const int *prefix, int E, int q) {
    int lo = 0, hi = E - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (prefix[mid] <= q) lo = mid; else hi = mid - 1;
    }
    return lo;
}

// Warp-level softmax + top-k of one token's logits l[0..E); writes
// topk_idx/topk_gate[t*K + k] (and sidx[k] if non-null).  A NaN logit (a
// token with a NaN or infinite component) ranks as -inf, so the K picks are
// always distinct experts in [0, E) (K <= E): the indices that address the
// dispatch arrays stay in range whatever the data; such a token's gates
// are NaN.
__device__ inline void select_topk(int E, int K, int t, const float *l, float *pk,
                            float *__restrict__ logits_opt, int32_t *__restrict__ topk_idx,
                            float *__restrict__ topk_gate, int *sidx) {
    const int lane = threadIdx.x & 31;
    if (logits_opt)
        for (int e = lane; e < E; e += 32) logits_opt[(size_t)t * E + e] = l[e];
    float m = -INFINITY;
    for (int e = lane; e < E; e += 32) m = fmaxf(m, l[e]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, o));
    float z = 0.f;
    for (int e = lane; e < E; e += 32) z += expf(l[e] - m);
    z = warp_sum(z);

    uint32_t taken = 0;  // bit i: expert lane + 32*i already selected
    float psel = 0.f;
    for (int k = 0; k < K; ++k) {
        float bv = -INFINITY;
        int bi = 0x7fffffff;
        for (int i = 0, e = lane; e < E; ++i, e += 32) {
            if ((taken >> i) & 1u) continue;
            const float v = isnan(l[e]) ? -INFINITY : l[e];
            if (v > bv || (v == bv && e < bi)) { bv = v; bi = e; }
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (ov > bv || (ov == bv && oi < bi)) { bv = ov; bi = oi; }
        }
        if ((bi & 31) == lane) taken |= 1u << (bi >> 5);
        const float p = expf(bv - m) / z;
        psel += p;
        if (lane == 0) {
            topk_idx[(size_t)t * K + k] = bi;
            pk[k] = p;
            if (sidx) sidx[k] = bi;
        }
    }
    __syncwarp();
    for (int k = lane; k < K; k += 32) topk_gate[(size_t)t * K + k] = pk[k] / psel;
}

// ---- host side -----------------------------------------------------------

struct DeviceInfo {
    int sm_count;
    unsigned *err;  // device address of the error word
};

// Per-device facts, looked up once per device (current device).
const DeviceInfo &device_info();

// Host-side fault injection for callers' error paths: MOE_INJECT_FAILURE
// "<entry point>:<status>" makes that entry return the status at once,
// before anything is validated or launched.  Read on every call (tests set
// it per process); nothing is injected when it is unset.
moe_status injected_failure(const char *entry);

#define MOE_INJECT(name)                                 \
    do {                                                 \
        moe_status inj_ = ::moe::injected_failure(name); \
        if (inj_ != MOE_OK) return inj_;                 \
    } while (0)

// Launch bookkeeping: counts every launch and, when profiling is on,
// brackets it with CUDA events on its stream.
struct LaunchScope {
    LaunchScope(const char *name, cudaStream_t stream);
    ~LaunchScope();
    const char *name;
    cudaStream_t stream;
    int slot;
};

// Workspace layout of moe_layer_forward / moe_expert_ffn for T tokens.
struct WsLayout {
    size_t idx, gate, counts, offsets, perm, inv_perm, h, xs, y, y_tail, ctr, total;
};
// Decode batches of up to this many tokens take the stream-K down projection
// (a second [T*K, D] fp32 output, added by the combine).
constexpr int kStreamKMaxTokens = 64;
WsLayout ws_layout(const moe_dims &d, int64_t T);

// Decode-path launchers (ffn_gemv.cu).
cudaError_t launch_up_glu_gemv(const moe_dims &d, int T, const void *x,
                               const int32_t *perm, const int32_t *offsets,
                               const void *w1, const void *v1, float *h,
                               cudaStream_t st);
cudaError_t launch_down_gemv(const moe_dims &d, int T, const float *h,
                             const int32_t *perm, const int32_t *offsets,
                             const void *w2, const float *gate, float *y_sorted,
                             const void *residual, void *out, bool fused,
                             cudaStream_t st);

// Launch with programmatic stream serialisation: the kernel may begin while
// the previous kernel in the stream finishes, and must execute
// griddepcontrol.wait before touching memory that kernel writes or reads.
inline cudaError_t launch_pdl(const void *func, dim3 grid, dim3 block, size_t smem,
                              cudaStream_t st, void **args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelExC(&cfg, func, args);
}

constexpr int kFusedCombineMaxTokens = 64;

// tcgen05 grouped GEMMs (ffn_tc.cu), bf16 only; h is bf16, y_sorted fp32.
bool tc_path_ok(const moe_dims &d);
cudaError_t launch_gather_rows(const moe_dims &d, int T, const void *x, const int32_t *perm,
                               void *x_sorted, cudaStream_t st, const int32_t *range = nullptr,
                               int n_range = 0);
cudaError_t launch_gemm_up_tc(const moe_dims &d, int T, const void *x_sorted,
                              const int32_t *offsets, const void *w1, const void *v1, void *h,
                              cudaStream_t st);
// One bf16 weight matrix w [Nw, Kdim] against T <= kRowsMaxTokens token rows
// x [T, Kdim]: y = x . w^T in fp32, weights as the MMA's M operand, the
// reduction split into `parts` (<= kRowsMaxParts) shares whose partial sums
// land in y + p*T*Nw for p < parts (the caller adds them in order).
// gemm_rows_parts: the split that keeps the SMs streaming for this shape.
constexpr int kRowsMaxTokens = 128;
constexpr int kRowsMaxParts = 4;
int gemm_rows_parts(int Kdim, int Nw);
cudaError_t launch_gemm_rows_tc(int T, int Kdim, int Nw, const void *x, const void *w, int parts,
                                float *y, cudaStream_t st, const char *name = nullptr);
// Causal attention of prefill tiles on the tensor cores (attn_tc.cu): every
// 128-token tile of the call whose tokens are positions p0..p0+127 of one
// sequence; tile_ok[i] = 1 for the tiles it handled (the others are left to
// the CUDA-core kernel).  q16 [T, Hq*128] bf16 queries (rotated, unscaled),
// caches [n_seq, Hkv, L, 128] bf16, head_dim 128.
constexpr int kAttnTcTile = 128;
bool attn_prefill_tc_ok();
cudaError_t launch_attn_prefill_tc(int T, int Hq, int Hkv, int n_seq, int L, const int32_t *seq,
                                   const int32_t *pos, const void *q16, const void *k_cache,
                                   const void *v_cache, void *ctx, int *tile_ok, cudaStream_t st);
// Decode attention on the tensor cores (attn_decode_tc.cu): every token of
// the call over positions 0..pos[t] of its sequence, in n_split (<= 8)
// position splits per (token, key/value head) that form a cluster and merge
// through distributed shared memory; ctx written.  Queries as above; query
// heads per key/value head <= 8.  attn_decode_tc_splits: the split count for
// one wave of CTAs.
bool attn_decode_tc_ok();
int attn_decode_tc_splits(int T, int Hkv, int max_len);
cudaError_t launch_attn_decode_tc(int T, int Hq, int Hkv, int n_seq, int L, int n_split,
                                  const int32_t *seq, const int32_t *pos, const void *q16,
                                  const void *k_cache, const void *v_cache, void *ctx,
                                  cudaStream_t st);

// name: the profiling name of the launch (default "gemm_down_tc").  y_tail
// (optional, [T*K, D]): the stream-K schedule's second output; the result is
// then y_sorted + y_tail.
cudaError_t launch_gemm_down_tc(const moe_dims &d, int T, const void *h, const int32_t *offsets,
                                const void *w2, float *y_sorted, cudaStream_t st,
                                const char *name = nullptr, float *y_tail = nullptr);

// Prefill forms of the two grouped GEMMs (ffn_tc_wm.cu): the expert weights
// as the MMA's M operand, the slots as a per-tile N; chosen by
// launch_gemm_up_tc / launch_gemm_down_tc when the batch is not a decode
// batch and gives the experts at least 128 slots each on average (fewer
// slots per weight tile stream the weights faster through the 128-slot
// tiles of ffn_tc.cu: 609 vs 641 us for the up projection at 128 tokens).
constexpr int kWmMinTokens = 65;
inline bool use_wm(const moe_dims &d, int T) {
    return T >= kWmMinTokens && (long long)T * d.top_k >= 128LL * d.n_experts;
}
cudaError_t launch_gemm_up_wm(const moe_dims &d, int T, const void *x_sorted,
                              const int32_t *offsets, const void *w1, const void *v1, void *h,
                              cudaStream_t st);
cudaError_t launch_gemm_down_wm(const moe_dims &d, int T, const void *h, const int32_t *offsets,
                                const void *w2, float *y_sorted, cudaStream_t st,
                                const char *name);

// Router logits of batches of 128 or more tokens on the tensor cores
// (route_tc.cu), E <= 16, bf16: partial logits of ksplit shares of d in
// `scratch` (route_tc_scratch_bytes), then top-k and gates as moe_route.
bool route_tc_ok(const moe_dims &d, int T);
size_t route_tc_scratch_bytes(const moe_dims &d, int T);
cudaError_t launch_route_tc(const moe_dims &d, int T, const void *x, const void *wr,
                            float *logits, int32_t *idx, float *gate, float *scratch,
                            cudaStream_t st);

// Bulk-copy pipelined decode kernels (ffn_stream.cu), bf16 only, up to
// kStreamMaxSlots slots; the GLU hidden vectors h are bf16.  Batches of at
// most kStreamMaxTokens tokens take them; larger ones take the tcgen05 GEMMs.
constexpr int kStreamMaxSlots = 64;
constexpr int kStreamMaxTokens = 1;
bool stream_path_ok(const moe_dims &d, int T);
// ctr (optional, one token only): a counter the routing kernel zeroed; the
// rows are then shared out as the SMs free their stages instead of in equal
// static shares.
cudaError_t launch_up_glu_stream(const moe_dims &d, int T, const void *x, const int32_t *perm,
                                 const int32_t *offsets, const void *w1, const void *v1, void *h,
                                 cudaStream_t st, int *ctr = nullptr);
cudaError_t launch_down_stream(const moe_dims &d, int T, const void *h, const int32_t *offsets,
                               const int32_t *inv_perm, const void *w2, const float *gate,
                               const void *residual, void *out, float *y_sorted, bool fused,
                               cudaStream_t st);

}  // namespace moe
