"""fp64 CPU oracle of the DBRX-style MoE layer (arxiv 2506.23635, Sec. 2.1,
Table 1 notes (d),(e), Sec. 4.2).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` are the only code allowed to import this
package.  It shares nothing with the CUDA path: the arithmetic lives in
``moe_oracle.c`` (plain C, fp64, OpenMP over output rows) and this module only
marshals numpy arrays into it.

Stored arrays use the numpy representation of ``paper_2506_23635_gb300.inputs``:
``"f32"`` = float32, ``"bf16"`` = uint16 bit patterns.  All functions return
float64 (values) or int32 (indices).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "moe_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libmoe_oracle.so")
_DT = {"f32": 0, "bf16": 1, "f64": 2}
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile ``moe_oracle.c`` with gcc (no -ffast-math) into ``_build/``."""
    os.makedirs(_BUILD, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    subprocess.check_call(["gcc", "-O2", "-fopenmp", "-fPIC", "-shared",
                           "-std=c11", "-o", tmp, _SRC, "-lm"])
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _bind(path: str) -> ctypes.CDLL:
    lib = ctypes.CDLL(path)
    P, I = ctypes.c_void_p, ctypes.c_int
    lib.orc_router_logits.argtypes = [I, I, I, P, I, P, I, P]
    lib.orc_topk_gates.argtypes = [I, I, I, P, P, P]
    lib.orc_dispatch.argtypes = [I, I, I, P, P, P, P, P]
    lib.orc_expert_ffn.argtypes = [I, I, P, P, P, P, I, P, P]
    lib.orc_layer_tokens.argtypes = [I, I, I, I, I, I, P, P, I, P, P, P, P, I,
                                     P, P, P, P]
    lib.orc_layer_tokens.restype = I
    lib.orc_layer_experts_tokens.argtypes = [I, I, I, I, I, I, I, I, P, P, I, P, P, P, P, I,
                                             P, P]
    lib.orc_layer_experts_tokens.restype = I
    lib.orc_layer_dense_masked.argtypes = [I, I, I, I, I, P, I, P, P, P, P, I, P]
    lib.orc_layer_dense_masked.restype = I
    lib.orc_num_threads.restype = I
    lib.orc_rmsnorm0.argtypes = [I, I, P, ctypes.c_double, P]
    lib.orc_round_bf16.argtypes = [ctypes.c_size_t, P, P]
    D_ = ctypes.c_double
    lib.orc_rope.argtypes = [I, I, I, D_, P, P]
    lib.orc_attention.argtypes = [I, I, I, I, I, I, P, P, P, P, P, P]
    lib.orc_attention.restype = I
    lib.orc_sa_forward.argtypes = [I, I, I, I, I, D_, D_, I, I, P, P, P, P, P, I, I, P, P]
    lib.orc_sa_forward.restype = I
    return lib


def _c(a: np.ndarray, dt=None) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dt) if dt is not None else np.ascontiguousarray(a)


def _p(a: np.ndarray):
    return ctypes.c_void_p(a.ctypes.data) if a is not None else None


def _storage(a: np.ndarray, dtype: str) -> np.ndarray:
    return _c(a, {"bf16": np.uint16, "f32": np.float32, "f64": np.float64}[dtype])


class OracleLib:
    """The oracle's functions bound to one compiled copy of ``moe_oracle.c``."""

    def __init__(self, path: str):
        self.path = path
        self.lib = _bind(path)

    def num_threads(self) -> int:
        """Threads the oracle's parallel loops use."""
        return int(self.lib.orc_num_threads())

    def router_logits(self, x, w_r, dtype: str, x_dtype: str = None) -> np.ndarray:
        """logits[t,e] = sum_d x[t,d] W_r[d,e] in fp64 (no bias)."""
        xdt = dtype if x_dtype is None else x_dtype
        x, w_r = _storage(x, xdt), _storage(w_r, dtype)
        T, D = x.shape
        E = w_r.shape[1]
        out = np.empty((T, E), np.float64)
        self.lib.orc_router_logits(T, D, E, _p(x), _DT[xdt], _p(w_r), _DT[dtype],
                                   _p(out))
        return out

    def topk_gates(self, logits: np.ndarray, k: int):
        """Softmax over all experts, K largest logits (descending, ties to the
        lower index), gates renormalised to sum to 1.  Returns (idx, gate)."""
        lg = _c(logits, np.float64)
        T, E = lg.shape
        idx = np.empty((T, k), np.int32)
        gate = np.empty((T, k), np.float64)
        self.lib.orc_topk_gates(T, E, k, _p(lg), _p(idx), _p(gate))
        return idx, gate

    def dispatch(self, topk_idx: np.ndarray, n_experts: int):
        """Stable dispatch by (expert, slot).  Returns counts [E], offsets
        [E+1], perm [S], inv_perm [S] (int32)."""
        idx = _c(topk_idx, np.int32)
        T, K = idx.shape
        if idx.size and (idx.min() < 0 or idx.max() >= n_experts):
            raise ValueError("expert index out of range")
        S = T * K
        counts = np.empty(n_experts, np.int32)
        offsets = np.empty(n_experts + 1, np.int32)
        perm = np.empty(S, np.int32)
        inv = np.empty(S, np.int32)
        self.lib.orc_dispatch(T, K, n_experts, _p(idx), _p(counts), _p(offsets),
                              _p(perm), _p(inv))
        return counts, offsets, perm, inv

    def expert_ffn(self, x_row64: np.ndarray, w1e, v1e, w2e, dtype: str):
        """One expert on one fp64 token vector: returns (h [F], y [D])."""
        xt = _c(x_row64, np.float64)
        w1e, v1e, w2e = (_storage(a, dtype) for a in (w1e, v1e, w2e))
        F, D = w1e.shape
        h = np.empty(F, np.float64)
        y = np.empty(D, np.float64)
        self.lib.orc_expert_ffn(D, F, _p(xt), _p(w1e), _p(v1e), _p(w2e), _DT[dtype],
                                _p(h), _p(y))
        return h, y

    def layer_tokens(self, x, w_r, w1, v1, w2, dtype: str, top_k: int,
                     tokens=None, residual=None, x_dtype: str = None):
        """The sparse MoE layer for the listed tokens (default: all).

        Returns (out [n,D] f64, idx [n,K] i32, gate [n,K] f64).  ``residual``
        ([T,D] float64) is added to each output row when given.  ``x_dtype``
        (default: ``dtype``) is the storage type of x, "f64" included.
        """
        xdt = dtype if x_dtype is None else x_dtype
        x = _storage(x, xdt)
        w_r, w1, v1, w2 = (_storage(a, dtype) for a in (w_r, w1, v1, w2))
        T, D = x.shape
        E, F, _ = w1.shape
        tok = _c(np.arange(T) if tokens is None else tokens, np.int32)
        n = tok.shape[0]
        out = np.empty((n, D), np.float64)
        idx = np.empty((n, top_k), np.int32)
        gate = np.empty((n, top_k), np.float64)
        res = None if residual is None else _c(residual, np.float64)
        rc = self.lib.orc_layer_tokens(T, D, F, E, top_k, n, _p(tok), _p(x),
                                       _DT[xdt], _p(w_r), _p(w1), _p(v1), _p(w2),
                                       _DT[dtype], _p(res), _p(out), _p(idx), _p(gate))
        if rc != 0:
            raise ValueError("token index out of range")
        return out, idx, gate

    def layer_experts_tokens(self, x, w_r, w1, v1, w2, dtype: str, top_k: int,
                             e_begin: int, e_end: int, tokens=None, residual=None):
        """One node's share of the expert-parallel layer (Sec. 4.3): the
        gated outputs of the selected experts in [e_begin, e_end) only, for
        the listed tokens (default: all), plus ``residual`` ([T,D] float64)
        when given.  w1, v1, w2 hold every expert.  Returns out [n,D] f64."""
        x = _storage(x, dtype)
        w_r, w1, v1, w2 = (_storage(a, dtype) for a in (w_r, w1, v1, w2))
        T, D = x.shape
        E, F, _ = w1.shape
        tok = _c(np.arange(T) if tokens is None else tokens, np.int32)
        out = np.empty((tok.shape[0], D), np.float64)
        res = None if residual is None else _c(residual, np.float64)
        rc = self.lib.orc_layer_experts_tokens(T, D, F, E, top_k, e_begin, e_end, tok.shape[0],
                                               _p(tok), _p(x), _DT[dtype], _p(w_r), _p(w1),
                                               _p(v1), _p(w2), _DT[dtype], _p(res), _p(out))
        if rc != 0:
            raise ValueError("token or expert range out of range")
        return out

    def rmsnorm0(self, x64: np.ndarray, eps: float) -> np.ndarray:
        """Parameter-free RMS pre-norm of each row (fp64)."""
        x = _c(x64, np.float64)
        T, D = x.shape
        out = np.empty_like(x)
        self.lib.orc_rmsnorm0(T, D, _p(x), float(eps), _p(out))
        return out

    def round_bf16(self, x64: np.ndarray) -> np.ndarray:
        """Nearest bfloat16 value of each element (ties to even), as fp64."""
        x = _c(x64, np.float64)
        out = np.empty_like(x)
        self.lib.orc_round_bf16(x.size, _p(x), _p(out))
        return out

    def stack_tokens(self, x0, layers, dtype: str, top_k: int, eps: float,
                     layer_callback=None):
        """Tokens through stacked layers: x_{l+1} = x_l + MoE_l(RMSNorm0(x_l)).

        x0: [n, D] token rows (storage ``dtype``, widened exactly); layers: a
        sequence of (w_r, w1, v1, w2) storage arrays, or a callable l -> that
        tuple (so a caller can bring one layer at a time to the host).
        Returns the fp64 residual stream after the last layer and an array
        [n_layers, n] of each token's gap between its K-th and (K+1)-th router
        logit divided by the RMS of its logits at that layer (how well
        conditioned the routing was; +inf when K = E)."""
        x = _to_f64(x0, dtype) if dtype != "f64" else _c(x0, np.float64)
        n_layers = len(layers) if not callable(layers) else None
        gaps = []
        l = 0
        while n_layers is None or l < n_layers:
            lw = layers(l) if callable(layers) else layers[l]
            if lw is None:
                break
            w_r, w1, v1, w2 = lw
            xn = self.rmsnorm0(x, eps)
            if dtype == "bf16":  # the layer input is stored in bf16 (reading C9)
                xn = self.round_bf16(xn)
            out, idx, _ = self.layer_tokens(xn, w_r, w1, v1, w2, dtype, top_k, residual=x,
                                            x_dtype="f64")
            logits = self.router_logits(xn, w_r, dtype, x_dtype="f64")
            if top_k >= logits.shape[1]:
                gaps.append(np.full(logits.shape[0], np.inf))
            else:
                srt = -np.sort(-logits, axis=1)
                rms = np.sqrt(np.mean(logits * logits, axis=1))
                gaps.append((srt[:, top_k - 1] - srt[:, top_k]) / rms)
            x = out
            l += 1
        return x, np.array(gaps)

    # ---- self-attention block of a decoder layer (readings in moe_oracle.c)

    def rope(self, u64: np.ndarray, pos, base: float) -> np.ndarray:
        """Rotary embedding of u [T, H, dh] (fp64) at positions pos [T]."""
        u = _c(u64, np.float64).copy()
        T, H, dh = u.shape
        pos = _c(pos, np.int32)
        self.lib.orc_rope(T, H, dh, base, _p(pos), _p(u))
        return u

    def attention(self, q64, k_cache64, v_cache64, seq, pos) -> np.ndarray:
        """Causal grouped-query attention of q [T, Hq, dh] over the caches
        [n_seq, Hkv, L, dh] (fp64 values); returns ctx [T, Hq, dh]."""
        q = _c(q64, np.float64)
        kc, vc = _c(k_cache64, np.float64), _c(v_cache64, np.float64)
        T, Hq, dh = q.shape
        n_seq, Hkv, L, _ = kc.shape
        seq, pos = _c(seq, np.int32), _c(pos, np.int32)
        ctx = np.empty_like(q)
        if self.lib.orc_attention(T, Hq, Hkv, dh, n_seq, L, _p(seq), _p(pos), _p(q), _p(kc),
                                  _p(vc), _p(ctx)) != 0:
            raise ValueError("sequence or position out of range")
        return ctx

    def sa_forward(self, x64, w_qkv, w_o, dtype: str, n_heads: int, n_kv_heads: int,
                   base: float, eps: float, seq, pos, k_cache64, v_cache64):
        """The self-attention block on the residual stream x [T, D] (fp64):
        returns (x + Wo ctx, k_cache, v_cache) with the new tokens' keys and
        values written into copies of the caches [n_seq, Hkv, L, dh]."""
        x = _c(x64, np.float64).copy()
        kc, vc = _c(k_cache64, np.float64).copy(), _c(v_cache64, np.float64).copy()
        T, D = x.shape
        n_seq, Hkv, L, dh = kc.shape
        assert Hkv == n_kv_heads
        wq, wo = _storage(w_qkv, dtype), _storage(w_o, dtype)
        seq, pos = _c(seq, np.int32), _c(pos, np.int32)
        rc = self.lib.orc_sa_forward(T, D, n_heads, n_kv_heads, dh, base, eps, n_seq, L,
                                     _p(seq), _p(pos), _p(x), _p(wq), _p(wo), _DT[dtype],
                                     1 if dtype == "bf16" else 0, _p(kc), _p(vc))
        if rc != 0:
            raise ValueError("sequence or position out of range")
        return x, kc, vc

    def decoder_layers(self, x0_64, layers, dtype: str, n_heads: int, n_kv_heads: int,
                       base: float, eps: float, top_k: int, seq, pos, caches):
        """Decoder layers x <- x + SA(x); x <- x + MoE(RMSNorm0(x)), in order.
        layers: sequence of (w_qkv, w_o, w_r, w1, v1, w2); caches: list of
        (k_cache, v_cache) fp64 per layer.  Returns the residual stream after
        the last layer, the updated caches and the routing gaps [n_layers, T]
        (as ``stack_tokens``)."""
        x = _c(x0_64, np.float64)
        out_caches, gaps = [], []
        for (w_qkv, w_o, w_r, w1, v1, w2), (kc, vc) in zip(layers, caches):
            x, kc, vc = self.sa_forward(x, w_qkv, w_o, dtype, n_heads, n_kv_heads, base, eps,
                                        seq, pos, kc, vc)
            x, g = self.moe_block(x, (w_r, w1, v1, w2), dtype, top_k, eps)
            out_caches.append((kc, vc))
            gaps.append(g)
        return x, out_caches, np.array(gaps)

    def moe_block(self, x64, layer, dtype: str, top_k: int, eps: float):
        """x + MoE(RMSNorm0(x)) on the fp64 residual stream x [T, D], the
        normalised input stored in bf16 when the weights are (reading C9).
        Returns the new stream and each token's routing gap (K-th minus
        (K+1)-th logit over the logit RMS; +inf when K = E)."""
        x = _c(x64, np.float64)
        xn = self.rmsnorm0(x, eps)
        if dtype == "bf16":
            xn = self.round_bf16(xn)
        w_r, w1, v1, w2 = layer
        out, _, _ = self.layer_tokens(xn, w_r, w1, v1, w2, dtype, top_k, residual=x,
                                      x_dtype="f64")
        logits = self.router_logits(xn, w_r, dtype, x_dtype="f64")
        if top_k >= logits.shape[1]:
            return out, np.full(logits.shape[0], np.inf)
        srt = -np.sort(-logits, axis=1)
        rms = np.sqrt(np.mean(logits * logits, axis=1))
        return out, (srt[:, top_k - 1] - srt[:, top_k]) / rms

    def layer_dense_masked(self, x, w_r, w1, v1, w2, dtype: str,
                           top_k: int) -> np.ndarray:
        """Busy full loading (Sec. 4.2): all experts on all tokens, unselected
        outputs zeroed in the weighted sum.  Returns out [T,D] f64."""
        x = _storage(x, dtype)
        w_r, w1, v1, w2 = (_storage(a, dtype) for a in (w_r, w1, v1, w2))
        T, D = x.shape
        E, F, _ = w1.shape
        out = np.empty((T, D), np.float64)
        self.lib.orc_layer_dense_masked(T, D, F, E, top_k, _p(x), _DT[dtype],
                                        _p(w_r), _p(w1), _p(v1), _p(w2), _DT[dtype],
                                        _p(out))
        return out

    def layer_steps(self, x, w_r, w1, v1, w2, dtype: str, top_k: int):
        """Every intermediate of the layer for all tokens, in the order of the
        method: logits, (idx, gate), dispatch, per-sorted-slot GLU hidden
        vectors and expert outputs (ungated), and the combined output."""
        logits = self.router_logits(x, w_r, dtype)
        idx, gate = self.topk_gates(logits, top_k)
        E = w1.shape[0]
        counts, offsets, perm, inv = self.dispatch(idx, E)
        x64 = _to_f64(x, dtype)
        S = perm.shape[0]
        T, D = x64.shape
        F = w1.shape[1]
        h_sorted = np.empty((S, F), np.float64)
        y_sorted = np.empty((S, D), np.float64)
        for j in range(S):
            t, k = divmod(int(perm[j]), top_k)
            e = int(idx[t, k])
            h_sorted[j], y_sorted[j] = self.expert_ffn(x64[t], w1[e], v1[e], w2[e], dtype)
        out = np.zeros((T, D), np.float64)
        for t in range(T):
            for k in range(top_k):
                out[t] += gate[t, k] * y_sorted[inv[t * top_k + k]]
        return dict(logits=logits, idx=idx, gate=gate, counts=counts,
                    offsets=offsets, perm=perm, inv_perm=inv, h_sorted=h_sorted,
                    y_sorted=y_sorted, out=out)


def default() -> OracleLib:
    """The oracle built from this directory's ``moe_oracle.c``."""
    global _lib
    with _lock:
        if _lib is None:
            _lib = OracleLib(build())
        return _lib


def num_threads():
    return default().num_threads()


def router_logits(*a, **k):
    return default().router_logits(*a, **k)


def topk_gates(*a, **k):
    return default().topk_gates(*a, **k)


def dispatch(*a, **k):
    return default().dispatch(*a, **k)


def expert_ffn(*a, **k):
    return default().expert_ffn(*a, **k)


def layer_tokens(*a, **k):
    return default().layer_tokens(*a, **k)


def layer_dense_masked(*a, **k):
    return default().layer_dense_masked(*a, **k)


def layer_experts_tokens(*a, **k):
    return default().layer_experts_tokens(*a, **k)


def layer_steps(*a, **k):
    return default().layer_steps(*a, **k)


def stack_tokens(*a, **k):
    return default().stack_tokens(*a, **k)


def rmsnorm0(*a, **k):
    return default().rmsnorm0(*a, **k)


def round_bf16(*a, **k):
    return default().round_bf16(*a, **k)


def rope(*a, **k):
    return default().rope(*a, **k)


def attention(*a, **k):
    return default().attention(*a, **k)


def sa_forward(*a, **k):
    return default().sa_forward(*a, **k)


def decoder_layers(*a, **k):
    return default().decoder_layers(*a, **k)


def moe_block(*a, **k):
    return default().moe_block(*a, **k)


def _to_f64(a, dtype):
    if dtype == "bf16":
        u = _c(a, np.uint16).astype(np.uint32) << 16
        return u.view(np.float32).astype(np.float64)
    return _c(a, np.float32).astype(np.float64)
