"""Python binding of libmoe (``include/moe.h``): argument marshalling only.

Every step runs in the library's CUDA kernels; this module passes
``tensor.data_ptr()`` and the current CUDA stream through ctypes and raises
``MoeError`` on a non-zero status.  PyTorch is used for device memory and
streams only.  There is no fallback: if ``libmoe.so`` has not been built the
import of the library raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

from . import build as _build

F32, BF16 = 0, 1
_DT = {torch.float32: F32, torch.bfloat16: BF16}
_STATUS = {
    0: "MOE_OK", 1: "MOE_ERR_INVALID_ARG", 2: "MOE_ERR_UNSUPPORTED",
    3: "MOE_ERR_WORKSPACE", 4: "MOE_ERR_CUDA", 5: "MOE_ERR_TIMEOUT",
    6: "MOE_ERR_DEVICE_INDEX",
}

# Every function the header declares (checked by the CPU tests).
EXPORTS = (
    "moe_workspace_size", "moe_route", "moe_dispatch", "moe_expert_ffn",
    "moe_combine", "moe_layer_forward", "moe_layer_forward_noalloc",
    "moe_layer_forward_experts", "moe_status_string",
    "moe_prenorm", "moe_stack_workspace_size", "moe_stack_forward",
    "moe_selftest_wait_timeout", "moe_dense_workspace_size", "moe_layer_forward_dense",
    "moe_get_last_error", "moe_launch_count", "moe_profile_enable",
    "moe_profile_reset", "moe_profile_read",
    "moe_sa_workspace_size", "moe_sa_qkv", "moe_sa_attend", "moe_sa_forward",
    "moe_decoder_workspace_size", "moe_decoder_forward",
)


class MoeError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {_STATUS.get(status, status)}")


class Dims(ctypes.Structure):
    _fields_ = [("d_model", ctypes.c_int32), ("ffn_hidden", ctypes.c_int32),
                ("n_experts", ctypes.c_int32), ("top_k", ctypes.c_int32),
                ("w_dtype", ctypes.c_int32), ("x_dtype", ctypes.c_int32),
                ("out_dtype", ctypes.c_int32)]

    def __repr__(self):
        return (f"Dims(D={self.d_model}, F={self.ffn_hidden}, E={self.n_experts}, "
                f"K={self.top_k}, w={self.w_dtype}, x={self.x_dtype}, out={self.out_dtype})")


class SaDims(ctypes.Structure):
    """moe_sa_dims: the self-attention block's shape."""
    _fields_ = [("d_model", ctypes.c_int32), ("n_heads", ctypes.c_int32),
                ("n_kv_heads", ctypes.c_int32), ("head_dim", ctypes.c_int32),
                ("rope_base", ctypes.c_float)]

    def __repr__(self):
        return (f"SaDims(D={self.d_model}, Hq={self.n_heads}, Hkv={self.n_kv_heads}, "
                f"dh={self.head_dim}, base={self.rope_base})")


class KernelStat(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char * 48), ("launches", ctypes.c_int64),
                ("total_ms", ctypes.c_double)]


_lib = None


def library_path() -> str:
    return _build.LIB


def lib() -> ctypes.CDLL:
    """Load libmoe.so (built by ``__graft_entry__.build()``); raise if absent."""
    global _lib
    if _lib is not None:
        return _lib
    path = library_path()
    if not os.path.exists(path):
        raise RuntimeError(f"libmoe.so is not built ({path}); run __graft_entry__.build()")
    L = ctypes.CDLL(path)
    P, I32, SZ = ctypes.c_void_p, ctypes.c_int32, ctypes.c_size_t
    DP = ctypes.POINTER(Dims)
    SP = ctypes.POINTER(SaDims)
    sigs = {
        "moe_workspace_size": [DP, I32, ctypes.POINTER(SZ)],
        "moe_route": [DP, I32, P, P, P, P, P, P],
        "moe_dispatch": [DP, I32, P, P, P, P, P, P],
        "moe_expert_ffn": [DP, I32, P, P, P, P, P, P, P, P, SZ, P],
        "moe_combine": [DP, I32, P, P, P, P, P, P],
        "moe_layer_forward": [DP, I32, P, P, P, P, P, P, P, P, SZ, P],
        "moe_layer_forward_noalloc": [DP, I32, P, P, P, P, P, P, P, P],
        "moe_layer_forward_experts": [DP, I32, P, P, I32, I32, P, P, P, P, P, P, SZ, P],
        "moe_prenorm": [DP, I32, P, P, ctypes.c_float, P],
        "moe_selftest_wait_timeout": [ctypes.c_uint64, P, P],
        "moe_dense_workspace_size": [DP, I32, ctypes.POINTER(SZ)],
        "moe_layer_forward_dense": [DP, I32, P, P, P, P, P, P, P, P, SZ, P],
        "moe_stack_workspace_size": [DP, I32, ctypes.POINTER(SZ)],
        "moe_stack_forward": [DP, I32, I32, ctypes.POINTER(P), ctypes.POINTER(P),
                              ctypes.POINTER(P), ctypes.POINTER(P), P, ctypes.c_float, P, SZ, P],
        "moe_get_last_error": [P],
        "moe_status_string": [ctypes.c_int],
        "moe_profile_enable": [ctypes.c_int],
        "moe_profile_reset": [],
        "moe_profile_read": [ctypes.POINTER(KernelStat), I32],
        "moe_launch_count": [],
        "moe_sa_workspace_size": [SP, I32, ctypes.POINTER(SZ)],
        "moe_sa_qkv": [SP, I32, P, P, P, P, I32, I32, P, P, P, P, SZ, P],
        "moe_sa_attend": [SP, I32, P, P, P, I32, I32, P, P, P, P, SZ, P],
        "moe_sa_forward": [SP, I32, P, P, I32, I32, P, P, P, P, P, ctypes.c_float, P, SZ, P],
        "moe_decoder_workspace_size": [SP, DP, I32, ctypes.POINTER(SZ)],
        "moe_decoder_forward": [SP, DP, I32, I32, P, P, I32, I32, P] + [ctypes.POINTER(P)] * 8
                               + [ctypes.c_float, P, SZ, P],
    }
    for name, args in sigs.items():
        fn = getattr(L, name)
        fn.argtypes = args
        fn.restype = ctypes.c_int
    L.moe_status_string.restype = ctypes.c_char_p
    L.moe_launch_count.restype = ctypes.c_int64
    L.moe_profile_enable.restype = None
    L.moe_profile_reset.restype = None
    L.moe_profile_read.restype = I32
    _lib = L
    return L


def _check(status: int, where: str):
    if status != 0:
        raise MoeError(status, where)


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_contiguous():
        raise ValueError("tensors must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def dims(d_model: int, ffn_hidden: int, n_experts: int, top_k: int,
         w_dtype=torch.bfloat16, x_dtype=None, out_dtype=None) -> Dims:
    x_dtype = w_dtype if x_dtype is None else x_dtype
    out_dtype = x_dtype if out_dtype is None else out_dtype
    return Dims(d_model, ffn_hidden, n_experts, top_k, _DT[w_dtype], _DT[x_dtype],
                _DT[out_dtype])


def _tdt(code: int):
    return torch.bfloat16 if code == BF16 else torch.float32


def workspace_size(d: Dims, max_tokens: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().moe_workspace_size(ctypes.byref(d), max_tokens, ctypes.byref(n)),
           "moe_workspace_size")
    return int(n.value)


def alloc_workspace(d: Dims, max_tokens: int, device="cuda") -> torch.Tensor:
    return torch.empty(max(workspace_size(d, max_tokens), 256), dtype=torch.uint8, device=device)


def route(d: Dims, x: torch.Tensor, w_r: torch.Tensor, want_logits: bool = False,
          stream=None):
    """Step 1: returns (topk_idx int32 [T,K], topk_gate f32 [T,K], logits or None)."""
    T = x.shape[0]
    dev = x.device
    idx = torch.empty((T, d.top_k), dtype=torch.int32, device=dev)
    gate = torch.empty((T, d.top_k), dtype=torch.float32, device=dev)
    logits = torch.empty((T, d.n_experts), dtype=torch.float32, device=dev) if want_logits else None
    _check(lib().moe_route(ctypes.byref(d), T, _ptr(x), _ptr(w_r), _ptr(logits), _ptr(idx),
                           _ptr(gate), _stream(stream)), "moe_route")
    return idx, gate, logits


def dispatch(d: Dims, topk_idx: torch.Tensor, stream=None):
    """Step 2: returns (counts [E], offsets [E+1], perm [S], inv_perm [S]) int32."""
    T = topk_idx.shape[0]
    dev = topk_idx.device
    S = T * d.top_k
    counts = torch.empty(d.n_experts, dtype=torch.int32, device=dev)
    offsets = torch.empty(d.n_experts + 1, dtype=torch.int32, device=dev)
    perm = torch.empty(S, dtype=torch.int32, device=dev)
    inv = torch.empty(S, dtype=torch.int32, device=dev)
    _check(lib().moe_dispatch(ctypes.byref(d), T, _ptr(topk_idx), _ptr(counts), _ptr(offsets),
                              _ptr(perm), _ptr(inv), _stream(stream)), "moe_dispatch")
    return counts, offsets, perm, inv


def expert_ffn(d: Dims, x, perm, offsets, w1, v1, w2, ws=None, stream=None):
    """Step 3: returns y_sorted f32 [T*K, D] (ungated expert outputs)."""
    T = x.shape[0]
    ws = alloc_workspace(d, T, x.device) if ws is None else ws
    y = torch.empty((T * d.top_k, d.d_model), dtype=torch.float32, device=x.device)
    _check(lib().moe_expert_ffn(ctypes.byref(d), T, _ptr(x), _ptr(perm), _ptr(offsets),
                                _ptr(w1), _ptr(v1), _ptr(w2), _ptr(y), _ptr(ws),
                                ws.numel(), _stream(stream)), "moe_expert_ffn")
    return y


def combine(d: Dims, y_sorted, inv_perm, gate, residual=None, out=None, stream=None):
    """Step 4: returns out [T, D] (out_dtype)."""
    T = gate.shape[0]
    if out is None:
        out = torch.empty((T, d.d_model), dtype=_tdt(d.out_dtype), device=gate.device)
    _check(lib().moe_combine(ctypes.byref(d), T, _ptr(y_sorted), _ptr(inv_perm), _ptr(gate),
                             _ptr(residual), _ptr(out), _stream(stream)), "moe_combine")
    return out


def layer_forward(d: Dims, x, w_r, w1, v1, w2, residual=None, out=None, ws=None,
                  stream=None):
    """The whole layer; returns out [T, D] (out_dtype)."""
    T = x.shape[0]
    if out is None:
        out = torch.empty((T, d.d_model), dtype=_tdt(d.out_dtype), device=x.device)
    ws = alloc_workspace(d, T, x.device) if ws is None else ws
    _check(lib().moe_layer_forward(ctypes.byref(d), T, _ptr(x), _ptr(w_r), _ptr(w1), _ptr(v1),
                                   _ptr(w2), _ptr(residual), _ptr(out), _ptr(ws), ws.numel(),
                                   _stream(stream)), "moe_layer_forward")
    return out


def layer_forward_experts(d: Dims, x, w_r, e_begin: int, e_end: int, w1_local, v1_local,
                          w2_local, residual=None, out=None, ws=None, stream=None):
    """One node's share of an expert-parallel layer (Sec. 4.3): the whole
    routing, then only experts e_begin..e_end-1, whose weights are
    ``w1_local`` [n, F, D], ``v1_local`` [n, F, D], ``w2_local`` [n, D, F]
    (n = e_end - e_begin).  Returns the fp32 partial [T, D] (plus
    ``residual`` [T, D] fp32 when given)."""
    T = x.shape[0]
    if out is None:
        out = torch.empty((T, d.d_model), dtype=torch.float32, device=x.device)
    ws = alloc_workspace(d, T, x.device) if ws is None else ws
    _check(lib().moe_layer_forward_experts(ctypes.byref(d), T, _ptr(x), _ptr(w_r), e_begin,
                                           e_end, _ptr(w1_local), _ptr(v1_local),
                                           _ptr(w2_local), _ptr(residual), _ptr(out), _ptr(ws),
                                           ws.numel(), _stream(stream)),
           "moe_layer_forward_experts")
    return out


STACK_EPS = 1e-6  # RMS pre-norm epsilon of the stacked layers


def prenorm(d: Dims, resid, x_norm=None, eps: float = STACK_EPS, stream=None):
    """x_norm = RMSNorm0(resid) rounded to x_dtype (the glue between layers)."""
    T = resid.shape[0]
    if x_norm is None:
        x_norm = torch.empty((T, d.d_model), dtype=_tdt(d.x_dtype), device=resid.device)
    _check(lib().moe_prenorm(ctypes.byref(d), T, _ptr(resid), _ptr(x_norm), eps,
                             _stream(stream)), "moe_prenorm")
    return x_norm


def stack_workspace_size(d: Dims, max_tokens: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().moe_stack_workspace_size(ctypes.byref(d), max_tokens, ctypes.byref(n)),
           "moe_stack_workspace_size")
    return int(n.value)


class StackWeights:
    """Device pointers of every layer's W_r, W1, V1, W2 as C arrays (the
    tensors must outlive this object's use)."""

    def __init__(self, layers):
        n = len(layers)
        self.n = n
        self.tensors = layers
        arr = lambda i: (ctypes.c_void_p * n)(*[ctypes.c_void_p(l[i].data_ptr()) for l in layers])
        self.w_r, self.w1, self.v1, self.w2 = arr(0), arr(1), arr(2), arr(3)


def stack_forward(d: Dims, weights: StackWeights, resid, ws=None, eps: float = STACK_EPS,
                  stream=None):
    """resid <- resid + MoE_l(RMSNorm0(resid)) for every layer, in place."""
    T = resid.shape[0]
    if ws is None:
        ws = torch.empty(max(stack_workspace_size(d, T), 256), dtype=torch.uint8,
                         device=resid.device)
    _check(lib().moe_stack_forward(ctypes.byref(d), weights.n, T, weights.w_r, weights.w1,
                                   weights.v1, weights.w2, _ptr(resid), eps, _ptr(ws),
                                   ws.numel(), _stream(stream)), "moe_stack_forward")
    return resid


NOALLOC_SCRATCH_BYTES = 24 * 1024 * 1024  # MOE_NOALLOC_SCRATCH_BYTES


def layer_forward_noalloc(d: Dims, x, w_r, w1, v1, w2, residual=None, out=None, stream=None):
    """The whole layer with the library's fixed device scratch array instead
    of a workspace (for callers that cannot allocate; T limited so that the
    workspace fits in NOALLOC_SCRATCH_BYTES, 24 MiB).  Returns out [T, D]
    (out_dtype)."""
    T = x.shape[0]
    if out is None:
        out = torch.empty((T, d.d_model), dtype=_tdt(d.out_dtype), device=x.device)
    _check(lib().moe_layer_forward_noalloc(ctypes.byref(d), T, _ptr(x), _ptr(w_r), _ptr(w1),
                                           _ptr(v1), _ptr(w2), _ptr(residual), _ptr(out),
                                           _stream(stream)), "moe_layer_forward_noalloc")
    return out


def selftest_wait_timeout(limit_ns: int, stream=None) -> bool:
    """Run the bounded-wait self test; True if the wait gave up."""
    flag = torch.zeros(1, dtype=torch.int32, device="cuda")
    _check(lib().moe_selftest_wait_timeout(limit_ns, _ptr(flag), _stream(stream)),
           "moe_selftest_wait_timeout")
    return bool(flag.item())


def dense_workspace_size(d: Dims, max_tokens: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().moe_dense_workspace_size(ctypes.byref(d), max_tokens, ctypes.byref(n)),
           "moe_dense_workspace_size")
    return int(n.value)


def layer_forward_dense(d: Dims, x, w_r, w1, v1, w2, residual=None, out=None, ws=None,
                        stream=None):
    """Busy full loading (Sec. 4.2): all experts on all tokens, unselected
    gates zero.  Returns out [T, D] (out_dtype)."""
    T = x.shape[0]
    if out is None:
        out = torch.empty((T, d.d_model), dtype=_tdt(d.out_dtype), device=x.device)
    if ws is None:
        ws = torch.empty(max(dense_workspace_size(d, T), 256), dtype=torch.uint8, device=x.device)
    _check(lib().moe_layer_forward_dense(ctypes.byref(d), T, _ptr(x), _ptr(w_r), _ptr(w1),
                                         _ptr(v1), _ptr(w2), _ptr(residual), _ptr(out), _ptr(ws),
                                         ws.numel(), _stream(stream)), "moe_layer_forward_dense")
    return out


def get_last_error(stream=None) -> int:
    """Synchronise the stream and return the library's pending status code."""
    return int(lib().moe_get_last_error(_stream(stream)))


def check_device_errors(stream=None):
    _check(get_last_error(stream), "device")


def launch_count() -> int:
    return int(lib().moe_launch_count())


def profile_enable(on: bool = True):
    lib().moe_profile_enable(1 if on else 0)


def profile_reset():
    lib().moe_profile_reset()


def profile_read() -> dict:
    """{kernel name: (launches, total ms)} since the last reset."""
    buf = (KernelStat * 64)()
    n = lib().moe_profile_read(buf, 64)
    return {buf[i].name.decode(): (int(buf[i].launches), float(buf[i].total_ms))
            for i in range(min(n, 64))}


def status_string(code: int) -> str:
    return lib().moe_status_string(code).decode()


# ---- self-attention block and whole decoder layers --------------------------


def sa_dims(d_model: int, n_heads: int, n_kv_heads: int, head_dim: int = 128,
            rope_base: float = 500000.0) -> SaDims:
    return SaDims(d_model, n_heads, n_kv_heads, head_dim, rope_base)


def sa_workspace_size(a: SaDims, max_tokens: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().moe_sa_workspace_size(ctypes.byref(a), max_tokens, ctypes.byref(n)),
           "moe_sa_workspace_size")
    return int(n.value)


def _sa_ws(a: SaDims, T: int, device, ws):
    if ws is None:
        ws = torch.empty(max(sa_workspace_size(a, T), 256), dtype=torch.uint8, device=device)
    return ws


def sa_qkv(a: SaDims, x_norm, w_qkv, seq, pos, k_cache, v_cache, q=None, ws=None, stream=None):
    """Rotated queries q [T, Hq, dh] (fp32); the T tokens' keys and values
    written into the caches [n_seq, Hkv, max_len, dh] at (seq[t], pos[t])."""
    T = x_norm.shape[0]
    n_seq, _, max_len, _ = k_cache.shape
    if q is None:
        q = torch.empty((T, a.n_heads, a.head_dim), dtype=torch.float32, device=x_norm.device)
    ws = _sa_ws(a, T, x_norm.device, ws)
    _check(lib().moe_sa_qkv(ctypes.byref(a), T, _ptr(x_norm), _ptr(w_qkv), _ptr(seq), _ptr(pos),
                            n_seq, max_len, _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(ws),
                            ws.numel(), _stream(stream)), "moe_sa_qkv")
    return q


def sa_attend(a: SaDims, q, seq, pos, k_cache, v_cache, ctx=None, ws=None, stream=None):
    """ctx [T, Hq * dh] (bf16): causal attention of each token over positions
    0..pos[t] of its sequence."""
    T = q.shape[0]
    n_seq, _, max_len, _ = k_cache.shape
    if ctx is None:
        ctx = torch.empty((T, a.n_heads * a.head_dim), dtype=torch.bfloat16, device=q.device)
    ws = _sa_ws(a, T, q.device, ws)
    _check(lib().moe_sa_attend(ctypes.byref(a), T, _ptr(q), _ptr(seq), _ptr(pos), n_seq,
                               max_len, _ptr(k_cache), _ptr(v_cache), _ptr(ctx), _ptr(ws),
                               ws.numel(), _stream(stream)), "moe_sa_attend")
    return ctx


def sa_forward(a: SaDims, resid, w_qkv, w_o, seq, pos, k_cache, v_cache, eps: float = STACK_EPS,
               ws=None, stream=None):
    """resid <- resid + W_o . Attn(RMSNorm0(resid)) in place (fp32 [T, D])."""
    T = resid.shape[0]
    n_seq, _, max_len, _ = k_cache.shape
    ws = _sa_ws(a, T, resid.device, ws)
    _check(lib().moe_sa_forward(ctypes.byref(a), T, _ptr(seq), _ptr(pos), n_seq, max_len,
                                _ptr(resid), _ptr(w_qkv), _ptr(w_o), _ptr(k_cache),
                                _ptr(v_cache), eps, _ptr(ws), ws.numel(), _stream(stream)),
           "moe_sa_forward")
    return resid


def decoder_workspace_size(a: SaDims, d: Dims, max_tokens: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().moe_decoder_workspace_size(ctypes.byref(a), ctypes.byref(d), max_tokens,
                                            ctypes.byref(n)), "moe_decoder_workspace_size")
    return int(n.value)


class DecoderWeights:
    """Device pointers of every decoder layer's tensors as C arrays: per
    layer (w_qkv, w_o, w_r, w1, v1, w2, k_cache, v_cache).  The tensors must
    outlive this object's use."""

    def __init__(self, layers):
        n = len(layers)
        self.n = n
        self.tensors = layers
        arr = lambda i: (ctypes.c_void_p * n)(*[ctypes.c_void_p(l[i].data_ptr()) for l in layers])
        (self.w_qkv, self.w_o, self.w_r, self.w1, self.v1, self.w2, self.k_cache,
         self.v_cache) = (arr(i) for i in range(8))
        self.n_seq, _, self.max_len, _ = layers[0][6].shape


def decoder_forward(a: SaDims, d: Dims, weights: DecoderWeights, resid, seq, pos,
                    eps: float = STACK_EPS, ws=None, stream=None):
    """Every decoder layer in order, in place on resid (fp32 [T, D]):
    resid += W_o . Attn(RMSNorm0(resid)); resid += MoE(RMSNorm0(resid))."""
    T = resid.shape[0]
    if ws is None:
        ws = torch.empty(max(decoder_workspace_size(a, d, T), 256), dtype=torch.uint8,
                         device=resid.device)
    W = weights
    _check(lib().moe_decoder_forward(ctypes.byref(a), ctypes.byref(d), W.n, T, _ptr(seq),
                                     _ptr(pos), W.n_seq, W.max_len, _ptr(resid), W.w_qkv, W.w_o,
                                     W.w_r, W.w1, W.v1, W.w2, W.k_cache, W.v_cache, eps,
                                     _ptr(ws), ws.numel(), _stream(stream)),
           "moe_decoder_forward")
    return resid
