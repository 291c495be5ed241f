/*
 * moe.h -- C ABI of the GB300 (sm_103a) DBRX-style Mixture-of-Experts layer.
 *
 * The layer is the one of arxiv 2506.23635 (Sec. 2.1; Table 1 and its notes
 * (d),(e)): every token is routed to top_k of n_experts feed-forward experts,
 * each expert is a SiLU-GLU FFN with three matrices w1, v1, w2 of size
 * d_model x ffn_hidden, and the selected experts' outputs are combined by a
 * weighted sum (Table 2 caption; Sec. 4.2).  With all experts resident in one
 * GPU's memory the layer is five steps, each exported here:
 *
 *   moe_route        router product, softmax, top-k, renormalised gates
 *   moe_dispatch     histogram, prefix sum and stable permutation
 *   moe_expert_ffn   grouped SiLU-GLU expert FFN over sorted slots
 *   moe_combine      gated combine back to token order
 *   moe_layer_forward  all of the above, fused where it pays
 *
 * Formulas (the paper gives the structure; the router and GLU formula are
 * the standard DBRX readings):
 *   logits[t,e] = sum_d x[t,d] * w_router[d,e]
 *   p[t,:] = softmax(logits[t,:]);  idx[t,0..K) = K largest logits,
 *            descending, ties to the lower expert index
 *   gate[t,k] = p[t,idx[t,k]] / sum_j p[t,idx[t,j]]
 *   h = SiLU(x . w1[e]^T) * (x . v1[e]^T),  SiLU(z) = z * sigmoid(z)
 *   y = h . w2[e]^T;   out[t,:] = sum_k gate[t,k] * y[(t,k),:]
 *
 * Layouts (row-major, all experts of a tensor in one contiguous allocation):
 *   x [T, D]; w_router [D, E]; w1, v1 [E, F, D]; w2 [E, D, F];
 *   a slot is s = t*K + k; "sorted" arrays are indexed by the position of a
 *   slot in the dispatch order (by expert, then by s).
 *
 * Conventions shared by every entry point:
 *   - Tensor pointers are DEVICE pointers owned by the caller, 16-byte
 *     aligned.  The library allocates no device memory; scratch space is the
 *     caller's workspace (moe_workspace_size), which also holds the work
 *     counters the one-token kernels share out rows with: calls that run at
 *     the same time on the GPU need workspaces of their own.
 *   - Calls are asynchronous on `stream` and never synchronise with the host
 *     (except moe_get_last_error and moe_profile_read).
 *   - Arguments are validated before anything is launched; on a validation
 *     error nothing is written and the status says why.
 *   - T == 0 is valid and launches nothing (moe_dispatch still writes zero
 *     counts and offsets).
 *   - Limits: 1 <= top_k <= n_experts <= 256; d_model and ffn_hidden are
 *     multiples of 8, 8 <= d_model <= 49152, 8 <= ffn_hidden <= 65536;
 *     T <= 1048576 and T*top_k <= 16777216; w_dtype == x_dtype.
 *   - Errors found by kernels (an expert index out of range, a bounded wait
 *     that ran out) are recorded on the device and reported by
 *     moe_get_last_error.
 */
#ifndef MOE_H_
#define MOE_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same type as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st *moe_stream_t;

typedef enum {
    MOE_OK = 0,
    MOE_ERR_INVALID_ARG = 1,  /* null pointer, bad size, misaligned pointer */
    MOE_ERR_UNSUPPORTED = 2,  /* a dtype combination that is not built */
    MOE_ERR_WORKSPACE = 3,    /* workspace missing or too small */
    MOE_ERR_CUDA = 4,         /* a CUDA call or kernel launch failed */
    MOE_ERR_TIMEOUT = 5,      /* a bounded device-side wait gave up */
    MOE_ERR_DEVICE_INDEX = 6  /* a kernel met an index outside its range: an expert
                                 outside [0,E), or a cache sequence / position
                                 outside the cache (moe_sa_*) */
} moe_status;

typedef enum { MOE_F32 = 0, MOE_BF16 = 1 } moe_dtype;

typedef struct {
    int32_t d_model;    /* D, Table 1 "D_embed" (6144 for DBRX) */
    int32_t ffn_hidden; /* F, Table 1 "D_ffn" (10752 for DBRX) */
    int32_t n_experts;  /* E, Sec. 2.1 (16 for DBRX) */
    int32_t top_k;      /* K, Sec. 2.1 (4 for DBRX) */
    int32_t w_dtype;    /* moe_dtype of w_router, w1, v1, w2 */
    int32_t x_dtype;    /* moe_dtype of x */
    int32_t out_dtype;  /* moe_dtype of out and of a residual */
} moe_dims;

/* Bytes of workspace moe_layer_forward and moe_expert_ffn need for up to
 * max_tokens tokens (a multiple of 256).  Writes *bytes; MOE_ERR_INVALID_ARG
 * for bad dims or max_tokens < 0. */
moe_status moe_workspace_size(const moe_dims *dims, int32_t max_tokens,
                              size_t *bytes);

/* Step 1 -- router and gates (Sec. 2.1 "selects 4 out of 16"; Table 2
 * caption lists the router under "Misc").
 *   x          [T, D]  x_dtype
 *   w_router   [D, E]  w_dtype
 *   logits_opt [T, E]  float32, written if non-NULL
 *   topk_idx   [T, K]  int32 expert ids, descending logit, ties -> lower id
 *   topk_gate  [T, K]  float32 renormalised gates (sum over k is 1)
 * fp32 accumulation.  A NaN logit ranks below every number, so a token with
 * a NaN (or infinite) component still gets K distinct experts in [0, E);
 * its gates are NaN.  Errors: MOE_ERR_INVALID_ARG (nulls, sizes). */
moe_status moe_route(const moe_dims *dims, int32_t T, const void *x,
                     const void *w_router, float *logits_opt,
                     int32_t *topk_idx, float *topk_gate, moe_stream_t stream);

/* Step 2 -- dispatch of the T*K slots to experts (the fork of Sec. 3.1,
 * Fig. 2: tokens go to the nodes holding their selected experts).
 *   topk_idx [T, K]  int32 in [0, E)
 *   counts   [E]     int32, slots per expert
 *   offsets  [E+1]   int32, exclusive prefix sum of counts
 *   perm     [T*K]   int32, perm[j] = slot at sorted position j; slots of an
 *                    expert are in ascending slot order (stable)
 *   inv_perm [T*K]   int32, inv_perm[s] = sorted position of slot s
 * Deterministic and bit-exact.  An index outside [0,E) is recorded as
 * MOE_ERR_DEVICE_INDEX (read by moe_get_last_error) and that slot is left
 * out of the permutation. */
moe_status moe_dispatch(const moe_dims *dims, int32_t T,
                        const int32_t *topk_idx, int32_t *counts,
                        int32_t *offsets, int32_t *perm, int32_t *inv_perm,
                        moe_stream_t stream);

/* Step 3 -- grouped SiLU-GLU expert FFN (Table 1 notes (d),(e): w1, v1, w2),
 * ungated, over the sorted slots.
 *   x        [T, D]    x_dtype
 *   perm     [T*K], offsets [E+1]   from moe_dispatch
 *   w1, v1   [E, F, D] w_dtype;  w2 [E, D, F] w_dtype
 *   y_sorted [T*K, D]  float32: y_sorted[j] = expert(e_j)(x[perm[j] / K])
 *   ws       workspace of at least moe_workspace_size(dims, T) bytes
 * fp32 accumulation; the GLU hidden vector is kept in fp32 (small T) or
 * rounded to bf16 before the down projection (tensor-core path). */
moe_status moe_expert_ffn(const moe_dims *dims, int32_t T, const void *x,
                          const int32_t *perm, const int32_t *offsets,
                          const void *w1, const void *v1, const void *w2,
                          float *y_sorted, void *ws, size_t ws_bytes,
                          moe_stream_t stream);

/* Step 4 -- weighted combine (Sec. 4.2 "weighted sum"; Sec. 4.3).
 *   y_sorted     [T*K, D] float32;  inv_perm [T*K];  topk_gate [T, K]
 *   residual_opt [T, D]   out_dtype, added if non-NULL; may be `out` itself
 *   out          [T, D]   out_dtype
 *   out[t,:] = residual[t,:] + sum_{k=0..K-1} gate[t,k] * y_sorted[inv_perm[t*K+k],:]
 * summed in ascending k. */
moe_status moe_combine(const moe_dims *dims, int32_t T, const float *y_sorted,
                       const int32_t *inv_perm, const float *topk_gate,
                       const void *residual_opt, void *out,
                       moe_stream_t stream);

/* The whole layer: route, dispatch, expert FFN and combine, with the gate
 * and combine fused into the expert kernels where the token count allows.
 *   x [T,D], w_router [D,E], w1/v1 [E,F,D], w2 [E,D,F] as above;
 *   residual_opt [T,D] out_dtype or NULL (may be `out` itself: each
 *   residual element is read before the same output element is written);
 *   out [T,D] out_dtype;
 *   ws  workspace of at least moe_workspace_size(dims, T) bytes.
 * No host synchronisation; capturable in a CUDA graph. */
moe_status moe_layer_forward(const moe_dims *dims, int32_t T, const void *x,
                             const void *w_router, const void *w1,
                             const void *v1, const void *w2,
                             const void *residual_opt, void *out, void *ws,
                             size_t ws_bytes, moe_stream_t stream);

/* ---- busy full loading (comparison baseline) -----------------------------
 * Sec. 4.2 "Busy Full Loading": every expert computes every token and the
 * outputs of the experts the router did not select are zeroed in the
 * weighted sum.  The result equals moe_layer_forward's (within rounding);
 * the cost is all E experts' weights and E/K times the FLOPs.  Kept as the
 * baseline the paper's sparse strategies are measured against.
 * Same arguments as moe_layer_forward; bf16 weights only (else
 * MOE_ERR_UNSUPPORTED); workspace of moe_dense_workspace_size bytes. */
moe_status moe_dense_workspace_size(const moe_dims *dims, int32_t max_tokens,
                                    size_t *bytes);
moe_status moe_layer_forward_dense(const moe_dims *dims, int32_t T,
                                   const void *x, const void *w_router,
                                   const void *w1, const void *v1,
                                   const void *w2, const void *residual_opt,
                                   void *out, void *ws, size_t ws_bytes,
                                   moe_stream_t stream);

/* ---- one node's share of an expert-parallel layer ------------------------
 * Sec. 4.3 (Fig. 7), the paper's decentralised design: every node holds the
 * router and a disjoint range of the experts; it routes every token itself,
 * runs its own experts on the tokens that selected them, and the nodes' gated
 * outputs are summed by one all-reduce of a [T, D] partial per layer (the
 * exchange of expert outputs of Sec. 3.1, whose cost is the communication
 * term of Eq. 1).  moe_layer_forward_experts is one node's part:
 *   partial_out[t,:] = residual_opt[t,:]
 *       + sum over k with e_begin <= topk_idx[t,k] < e_end of
 *         gate[t,k] * y[(t,k),:]
 * where the routing (router over all E experts, softmax, top-k, gates,
 * dispatch) is the whole layer's, as in moe_layer_forward.
 *   0 <= e_begin < e_end <= E  (dims->n_experts is the whole layer's E);
 *   w_router [D, E]: the whole router;
 *   w1_local, v1_local [e_end - e_begin, F, D], w2_local [e_end - e_begin,
 *     D, F]: the weights of experts e_begin..e_end-1 only (a node's resident
 *     share; a caller holding every expert passes w1 + e_begin*F*D, ...);
 *   residual_opt [T, D] float32 or NULL (give it to one node only, so that
 *     the sum carries it once);
 *   partial_out [T, D] float32 whatever dims->out_dtype says; a token none of
 *     whose experts lies in the range gets its residual row (or zeros);
 *   ws: moe_workspace_size(dims, T) bytes.
 * The partials of disjoint ranges covering [0, E), summed, give
 * moe_layer_forward's output in fp32 (the k sum in another order).  The
 * sum itself (NCCL all-reduce between GPUs) is the caller's.  Errors: as
 * moe_layer_forward, plus MOE_ERR_INVALID_ARG for an empty or out-of-range
 * expert range. */
moe_status moe_layer_forward_experts(const moe_dims *dims, int32_t T,
                                     const void *x, const void *w_router,
                                     int32_t e_begin, int32_t e_end,
                                     const void *w1_local, const void *v1_local,
                                     const void *w2_local,
                                     const float *residual_opt,
                                     float *partial_out, void *ws,
                                     size_t ws_bytes, moe_stream_t stream);

/* ---- stack of layers (decode through consecutive MoE blocks) -------------
 * The paper runs DBRX's 40 decoder layers (Table 1); a stack of MoE blocks
 * needs the glue between them, which the paper does not print.  Reading
 * used here: a parameter-free RMS pre-norm and a residual add,
 *   x_{l+1} = x_l + MoE_l( RMSNorm0(x_l) ),
 *   RMSNorm0(r) = r / sqrt(mean(r^2) + eps),
 * with the residual stream in out_dtype (fp32 for the DBRX stack) and the
 * normalised layer input rounded to x_dtype.
 *
 * moe_prenorm: x_norm[t,:] = RMSNorm0(resid[t,:]).
 *   resid [T, D] out_dtype;  x_norm [T, D] x_dtype;  eps > 0.
 * moe_stack_workspace_size: bytes moe_stack_forward needs for max_tokens.
 * moe_stack_forward: applies n_layers layers in order to resid in place.
 *   w_router, w1, v1, w2: HOST arrays of n_layers DEVICE pointers, each
 *   laid out as for moe_layer_forward;  resid [T, D] out_dtype, in/out. */
moe_status moe_prenorm(const moe_dims *dims, int32_t T, const void *resid,
                       void *x_norm, float eps, moe_stream_t stream);
moe_status moe_stack_workspace_size(const moe_dims *dims, int32_t max_tokens,
                                    size_t *bytes);
moe_status moe_stack_forward(const moe_dims *dims, int32_t n_layers, int32_t T,
                             const void *const *w_router, const void *const *w1,
                             const void *const *v1, const void *const *w2,
                             void *resid, float eps, void *ws, size_t ws_bytes,
                             moe_stream_t stream);

/* ---- layer without a caller workspace ----------------------------------
 * The paper has no counterpart of this entry point; it serves callers that
 * cannot allocate device memory themselves (a framework that owns every
 * device buffer through its own pool, a plugin handed only its inputs and
 * outputs, a runtime that forbids allocation after start-up).
 *
 * Same arguments and result as moe_layer_forward, minus the workspace: the
 * scratch space is a fixed array of MOE_NOALLOC_SCRATCH_BYTES bytes in device
 * memory owned by the library.  Every GPU that loads this part of the
 * library holds that array until the process exits.
 *   - Limit: a call is accepted when moe_workspace_size(dims, T) is at most
 *     MOE_NOALLOC_SCRATCH_BYTES (24 MiB: the DBRX-shaped layer, D = 6144,
 *     F = 10752, E = 16, K = 4, fits at every T from 1 to 64, whose largest
 *     workspace is 20.25 MiB at T = 64); a larger workspace returns
 *     MOE_ERR_WORKSPACE and launches nothing.
 *   - The first call on a device looks up the array's device address (once
 *     per device, with that device current) and keeps it until the process
 *     exits; make that first call before any stream capture on the device.
 *     The kept address belongs to the device's context of that moment: after
 *     cudaDeviceReset (or a reset of the primary context) on a device, do not
 *     call this entry point on that device again in the same process.
 *   - Allocates nothing (no cudaMalloc, cudaFree or allocating library call).
 *   - Every call uses the same array, which keeps the last call's contents;
 *     nothing in it has to start at zero.  Calls whose executions overlap on
 *     the GPU (different streams, or different host threads on one device)
 *     race on the array: serialise them. */
#define MOE_NOALLOC_SCRATCH_BYTES (24u * 1024u * 1024u)

moe_status moe_layer_forward_noalloc(const moe_dims *dims, int32_t T,
                                     const void *x, const void *w_router,
                                     const void *w1, const void *v1,
                                     const void *w2, const void *residual_opt,
                                     void *out, moe_stream_t stream);

/* Human-readable name of a status. */
const char *moe_status_string(moe_status status);

/* Synchronises `stream`, then reports (and clears) the first error recorded
 * by a kernel since the last call, or MOE_ERR_CUDA for a failed launch or an
 * asynchronous CUDA fault. */
moe_status moe_get_last_error(moe_stream_t stream);

/* ---- failure detection ---------------------------------------------------
 * Every device-side wait in the pipelined kernels gives up after a wall-time
 * limit (2 s), records MOE_ERR_TIMEOUT and lets its kernel return, so a
 * broken pipeline ends instead of hanging the GPU.
 * moe_selftest_wait_timeout exercises exactly that path: one thread waits on
 * an mbarrier that nothing completes, with the given limit (<= 10 s); it
 * writes 1 to *gave_up (a DEVICE int) when the wait gave up, and the next
 * moe_get_last_error returns MOE_ERR_TIMEOUT.  The context stays usable.
 * Host-side fault injection: with MOE_INJECT_FAILURE="<entry>:<status>" in
 * the environment, the named entry point (moe_route, moe_dispatch,
 * moe_expert_ffn, moe_combine, moe_layer_forward, moe_layer_forward_dense,
 * moe_layer_forward_experts, moe_prenorm, moe_stack_forward,
 * moe_layer_forward_noalloc, moe_sa_qkv,
 * moe_sa_attend, moe_sa_forward, moe_decoder_forward) returns that status at
 * once without launching.
 * With MOE_WM_SINGLE_CTA=1 the prefill expert GEMMs (batches whose experts
 * hold 128 or more slots on average) run one CTA per tile, the form used on
 * devices that cannot keep CTA pairs resident, instead of CTA pairs. */
moe_status moe_selftest_wait_timeout(uint64_t limit_ns, int32_t *gave_up,
                                     moe_stream_t stream);

/* ---- launch accounting and per-kernel timing (benchmarks) ---------------
 * moe_launch_count: number of kernels this library has launched since load.
 * moe_profile_enable(1): every later kernel launch is bracketed by a pair of
 * CUDA events recorded on its own stream; moe_profile_read synchronises those
 * events and returns, per kernel name, the launches and the summed
 * event-measured milliseconds since the last moe_profile_reset. */
typedef struct {
    char name[48];
    int64_t launches;
    double total_ms;
} moe_kernel_stat;

int64_t moe_launch_count(void);
void moe_profile_enable(int on);
void moe_profile_reset(void);
int32_t moe_profile_read(moe_kernel_stat *stats, int32_t max_stats);

/* ---- self-attention block and whole decoder layers ---------------------
 * Table 1 (note (b)) sizes a DBRX layer's self-attention only by its
 * parameters, D_qkv_hidden x D_embed + D_embed^2 with D_qkv_hidden = 8,192,
 * and Table 2 books its time under "Misc." beside the router and the
 * weighted sum.  The paper prints nothing else about it; this library reads
 * it as the standard DBRX block:
 *   - grouped-query attention: n_heads query heads share n_kv_heads
 *     key/value heads of head_dim (48 + 2 x 8 heads of 128 give 8,192);
 *     query head h reads key/value head h / (n_heads / n_kv_heads);
 *   - rotary position embedding of queries and keys: in every head, dims i
 *     and i + head_dim/2 turn by the angle pos * rope_base^(-2i/head_dim);
 *   - causal softmax attention scaled by 1/sqrt(head_dim); no biases;
 *   - the pre-norm residual block  resid += w_o . Attn(RMSNorm0(resid)),
 *     RMSNorm0 as in moe_prenorm (no learned scale).
 * Storage: the normalised input, the rotated queries (as the attention
 * reads them), the cached keys and values and the attention output ctx are
 * bf16; projections accumulate in fp32; the residual stream is fp32.
 *
 * Layouts (row-major): w_qkv [(Hq + 2 Hkv) dh, D] bf16 -- the query rows,
 * then the key rows, then the value rows; w_o [D, Hq dh] bf16; k_cache and
 * v_cache [n_seq, Hkv, max_len, dh] bf16, owned by the caller; q [T, Hq, dh]
 * fp32; ctx [T, Hq dh] bf16; resid [T, D] fp32.
 *
 * Tokens: token t is position pos[t] of sequence seq[t] (device int32
 * arrays of T entries).  A call first writes every new token's key and value
 * at (seq[t], pos[t]) and then lets each token attend to positions
 * 0..pos[t] of its sequence: a prefill passes consecutive positions of one
 * sequence, a decode step one token per sequence.  The caller keeps the
 * (seq, pos) pairs of a call distinct and the positions below pos[t]
 * filled by earlier calls.  seq and pos are complete before the call in
 * stream order (written by a copy, or by a kernel that lets the next launch
 * start only when it ends: the decode attention reads them before it waits
 * for the kernel ahead of it).  A token whose seq or pos lies outside the cache
 * is recorded as MOE_ERR_DEVICE_INDEX, writes nothing to the cache and gets a
 * zero ctx.
 *
 * Limits: head_dim == 128; n_kv_heads divides n_heads and n_heads /
 * n_kv_heads <= 8; d_model a multiple of 8 in [8, 49152];
 * (n_heads + 2 n_kv_heads) * 128 <= 49152; n_seq >= 1, max_len >= 1;
 * rope_base > 1; T <= 65536.  bf16 only. */
typedef struct {
    int32_t d_model;     /* D */
    int32_t n_heads;     /* Hq: query heads */
    int32_t n_kv_heads;  /* Hkv: key/value heads */
    int32_t head_dim;    /* dh */
    float rope_base;     /* rotary base (DBRX: 500000) */
} moe_sa_dims;

/* moe_sa_workspace_size: bytes of scratch the moe_sa_* calls need for up to
 * max_tokens tokens. */
moe_status moe_sa_workspace_size(const moe_sa_dims *dims, int32_t max_tokens, size_t *bytes);

/* moe_sa_qkv: from the normalised input x_norm [T, D] (bf16): q = the
 * rotated queries (fp32 out), and the rotated keys and the values of the T
 * tokens written into k_cache / v_cache at (seq[t], pos[t]). */
moe_status moe_sa_qkv(const moe_sa_dims *dims, int32_t T, const void *x_norm,
                      const void *w_qkv, const int32_t *seq, const int32_t *pos,
                      int32_t n_seq, int32_t max_len, float *q, void *k_cache,
                      void *v_cache, void *ws, size_t ws_bytes, moe_stream_t stream);

/* moe_sa_attend: ctx[t, h dh .. (h+1) dh) = softmax over positions
 * 0..pos[t] of bf16(q[t,h]) . K / sqrt(dh), applied to V (bf16 out): the
 * queries are read rounded to bf16.  As in moe_sa_forward, every 128
 * consecutive tokens that are positions p0..p0+127 of one sequence (a
 * prefill chunk) are attended by the tensor-core flash attention, and the
 * tokens of a call without such a chunk (decode steps) by the tensor-core
 * decode attention; other tokens by the CUDA-core kernel.
 * MOE_ATTN_CUDA_CORES=1 in the environment keeps decode steps on the
 * CUDA-core kernel. */
moe_status moe_sa_attend(const moe_sa_dims *dims, int32_t T, const float *q,
                         const int32_t *seq, const int32_t *pos, int32_t n_seq,
                         int32_t max_len, const void *k_cache, const void *v_cache,
                         void *ctx, void *ws, size_t ws_bytes, moe_stream_t stream);

/* moe_sa_forward: the whole block in place on resid:
 * resid += w_o . Attn(RMSNorm0(resid)), caches updated as in moe_sa_qkv. */
moe_status moe_sa_forward(const moe_sa_dims *dims, int32_t T, const int32_t *seq,
                          const int32_t *pos, int32_t n_seq, int32_t max_len, float *resid,
                          const void *w_qkv, const void *w_o, void *k_cache, void *v_cache,
                          float eps, void *ws, size_t ws_bytes, moe_stream_t stream);

/* moe_decoder_workspace_size / moe_decoder_forward: n_layers decoder layers
 * in order, each  resid += w_o . Attn(RMSNorm0(resid));
 *                 resid += MoE(RMSNorm0(resid))  (as moe_stack_forward).
 * attn->d_model == moe->d_model; moe: bf16 weights and input, out_dtype F32
 * (the fp32 residual stream).  Per-layer tensors come as HOST arrays of
 * n_layers DEVICE pointers. */
moe_status moe_decoder_workspace_size(const moe_sa_dims *attn, const moe_dims *moe,
                                      int32_t max_tokens, size_t *bytes);
moe_status moe_decoder_forward(const moe_sa_dims *attn, const moe_dims *moe, int32_t n_layers,
                               int32_t T, const int32_t *seq, const int32_t *pos,
                               int32_t n_seq, int32_t max_len, float *resid,
                               const void *const *w_qkv, const void *const *w_o,
                               const void *const *w_router, const void *const *w1,
                               const void *const *v1, const void *const *w2,
                               void *const *k_cache, void *const *v_cache, float eps,
                               void *ws, size_t ws_bytes, moe_stream_t stream);

#ifdef __cplusplus
}
#endif
#endif /* MOE_H_ */
