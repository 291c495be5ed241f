"""Seeded synthetic inputs for the DBRX-style MoE layer.

This module is shared by the CUDA path's tests and benchmark and by the
fp64 oracle's tests.  It holds none of the layer's arithmetic: it draws
normal numbers, rounds them to the storage type, and conditions the router so
that the top-k choice is well separated (every token has a gap of at least
``min_gap`` between its k-th and (k+1)-th router logit).  The gap check uses a
plain numpy fp64 matrix product of the stored bytes; it is input conditioning,
not a step of the method.

Two sources of randomness are used:

* host: ``numpy.random.Generator(PCG64)`` seeded from ``(seed, *tags)``, for
  every array that a test hands to the oracle directly;
* device: ``torch.Generator`` on a CUDA device, for the multi-GB expert weight
  tensors of the full-size layer.  Those bytes are copied back to the host
  whenever the oracle needs them, so the oracle always reads exactly the bytes
  the kernels read.

Storage types: ``"f32"`` (numpy float32) and ``"bf16"`` (numpy uint16 holding
the bfloat16 bit pattern, rounded to nearest even).
"""
from __future__ import annotations

import dataclasses
import hashlib
from typing import Optional, Sequence

import numpy as np

# --------------------------------------------------------------------------
# seeds and dtypes
# --------------------------------------------------------------------------


def stream_seed(seed: int, *tags) -> int:
    """A 63-bit seed derived from ``seed`` and any tags (ints or strings)."""
    h = hashlib.sha256(repr((int(seed),) + tuple(tags)).encode()).digest()
    return int.from_bytes(h[:8], "little") & ((1 << 63) - 1)


def host_rng(seed: int, *tags) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(stream_seed(seed, *tags)))


def f32_to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bfloat16 (nearest, ties to even); uint16 bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32).astype(np.uint64)
    u = u + 0x7FFF + ((u >> 16) & 1)
    return (u >> 16).astype(np.uint16)


def bf16_bits_to_f64(b: np.ndarray) -> np.ndarray:
    """Exact widening of bfloat16 bit patterns (uint16) to float64."""
    u = np.ascontiguousarray(b, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def to_f64(a: np.ndarray, dtype: str) -> np.ndarray:
    """Exact float64 view of a stored array (``dtype`` in {"f32","bf16"})."""
    if dtype == "bf16":
        return bf16_bits_to_f64(a)
    return np.asarray(a, dtype=np.float32).astype(np.float64)


def store(a64: np.ndarray, dtype: str) -> np.ndarray:
    """Round float64 values once to the storage type."""
    a32 = np.asarray(a64, dtype=np.float64).astype(np.float32)
    return f32_to_bf16_bits(a32) if dtype == "bf16" else a32


def host_normal(shape, std: float, dtype: str, seed: int, *tags) -> np.ndarray:
    """N(0, std^2) samples rounded to the storage type."""
    z = host_rng(seed, *tags).standard_normal(size=shape) * std
    return store(z, dtype)


# --------------------------------------------------------------------------
# layer configuration
# --------------------------------------------------------------------------


@dataclasses.dataclass(frozen=True)
class LayerShape:
    d_model: int
    ffn_hidden: int
    n_experts: int
    top_k: int
    dtype: str = "bf16"  # storage type of x and all weights

    @property
    def expert_params(self) -> int:
        return 3 * self.d_model * self.ffn_hidden


TINY = LayerShape(256, 512, 4, 2, "f32")
DBRX = LayerShape(6144, 10752, 16, 4, "bf16")

W_STD = 0.02  # weights ~ N(0, 0.02^2)
X_STD = 1.0  # tokens ~ N(0, 1)


# --------------------------------------------------------------------------
# router conditioning
# --------------------------------------------------------------------------


def topk_gaps(x: np.ndarray, w_r: np.ndarray, dtype: str, k: int) -> np.ndarray:
    """Per-token gap between the k-th and (k+1)-th largest realised logit.

    The logits are the fp64 product of the stored bytes.  With k == E there is
    no (k+1)-th logit and the gap is +inf.
    """
    lg = to_f64(x, dtype) @ to_f64(w_r, dtype)
    e = lg.shape[1]
    if k >= e:
        return np.full(lg.shape[0], np.inf)
    s = -np.sort(-lg, axis=1)
    return s[:, k - 1] - s[:, k]


def gap_condition_tokens(x: np.ndarray, w_r: np.ndarray, shape: LayerShape,
                         seed: int, min_gap: float = 1e-3,
                         max_tries: int = 64) -> np.ndarray:
    """Resample token rows whose top-k gap is below ``min_gap``.

    A failing row t is redrawn from the stream ``(seed, "x-retry", t, try)``;
    the result is deterministic for a given seed.
    """
    x = x.copy()
    for attempt in range(max_tries):
        bad = np.nonzero(topk_gaps(x, w_r, shape.dtype, shape.top_k) < min_gap)[0]
        if bad.size == 0:
            return x
        for t in bad:
            x[t] = host_normal((shape.d_model,), X_STD, shape.dtype, seed,
                               "x-retry", int(t), attempt)
    raise RuntimeError("could not separate the top-k logits")


def designed_router(x: np.ndarray, shape: LayerShape, skew: float, seed: int,
                    min_gap: float = 1e-3, max_tries: int = 64) -> np.ndarray:
    """Router weights whose logits follow a designed Zipf(skew) expert load.

    Target logits are ``log(pi_e) + Gumbel`` with ``pi_e ~ rank(e)^-skew`` over
    a seeded expert order, so the top-k of a token is a sample without
    replacement weighted by pi (skew 0 = uniform).  ``W_r`` is the minimum-norm
    solution of ``x W_r = L`` in fp64 (T <= D), rounded once to the storage
    type; the gaps are then re-checked on the realised logits and the Gumbel
    draws of failing tokens are redrawn.
    """
    T, D = x.shape
    E, K = shape.n_experts, shape.top_k
    if T > D:
        raise ValueError("designed router needs T <= d_model")
    rng = host_rng(seed, "router-order")
    order = rng.permutation(E)
    pi = np.empty(E)
    pi[order] = (np.arange(E) + 1.0) ** (-skew)
    pi /= pi.sum()
    x64 = to_f64(x, shape.dtype)
    gram = x64 @ x64.T
    gum = host_rng(seed, "gumbel").gumbel(size=(T, E))
    for attempt in range(max_tries):
        L = np.log(pi)[None, :] + gum
        w = x64.T @ np.linalg.solve(gram, L)
        w_r = store(w, shape.dtype)
        bad = np.nonzero(topk_gaps(x, w_r, shape.dtype, K) < min_gap)[0]
        if bad.size == 0:
            return w_r
        for t in bad:
            gum[t] = host_rng(seed, "gumbel-retry", int(t), attempt).gumbel(size=E)
    raise RuntimeError("could not separate the designed top-k logits")


# --------------------------------------------------------------------------
# whole-layer inputs on the host
# --------------------------------------------------------------------------


@dataclasses.dataclass
class HostLayer:
    shape: LayerShape
    x: np.ndarray  # [T, D]
    w_r: np.ndarray  # [D, E]
    w1: np.ndarray  # [E, F, D]
    v1: np.ndarray  # [E, F, D]
    w2: np.ndarray  # [E, D, F]


def host_router_and_tokens(shape: LayerShape, T: int, seed: int,
                           skew: Optional[float] = None,
                           min_gap: float = 1e-3):
    """Tokens x [T,D] and router W_r [D,E], gap-conditioned.

    ``skew=None``: random router W_r ~ N(0, 0.02^2) (experts exchangeable,
    uniform-random routing).  Otherwise the designed Zipf router.
    """
    D, E = shape.d_model, shape.n_experts
    x = host_normal((T, D), X_STD, shape.dtype, seed, "x")
    if skew is None:
        w_r = host_normal((D, E), W_STD, shape.dtype, seed, "w_r")
        x = gap_condition_tokens(x, w_r, shape, seed, min_gap)
    else:
        w_r = designed_router(x, shape, skew, seed, min_gap)
    return x, w_r


def host_expert_weights(shape: LayerShape, seed: int,
                        experts: Optional[Sequence[int]] = None):
    """W1, V1 [E,F,D] and W2 [E,D,F]; each expert is its own seeded stream.

    With ``experts`` given, only those experts are drawn (the rest are zero),
    which lets a host-only program build the experts a token selects.
    """
    D, F, E = shape.d_model, shape.ffn_hidden, shape.n_experts
    np_dt = np.uint16 if shape.dtype == "bf16" else np.float32
    w1 = np.zeros((E, F, D), np_dt)
    v1 = np.zeros((E, F, D), np_dt)
    w2 = np.zeros((E, D, F), np_dt)
    for e in (range(E) if experts is None else experts):
        w1[e] = host_normal((F, D), W_STD, shape.dtype, seed, "w1", int(e))
        v1[e] = host_normal((F, D), W_STD, shape.dtype, seed, "v1", int(e))
        w2[e] = host_normal((D, F), W_STD, shape.dtype, seed, "w2", int(e))
    return w1, v1, w2


def host_layer(shape: LayerShape, T: int, seed: int,
               skew: Optional[float] = None, min_gap: float = 1e-3) -> HostLayer:
    x, w_r = host_router_and_tokens(shape, T, seed, skew, min_gap)
    w1, v1, w2 = host_expert_weights(shape, seed)
    return HostLayer(shape, x, w_r, w1, v1, w2)


# --------------------------------------------------------------------------
# device-side weights (multi-GB); torch is imported lazily
# --------------------------------------------------------------------------


def device_normal_(out, std: float, seed: int, *tags, chunk_elems: int = 1 << 28):
    """Fill a CUDA tensor (bf16 or f32) with N(0, std^2), in place.

    Draws fp32 normals from a seeded ``torch.Generator`` on the tensor's
    device in chunks and rounds them to the tensor's dtype.
    """
    import torch

    g = torch.Generator(device=out.device)
    g.manual_seed(stream_seed(seed, *tags))
    flat = out.view(-1)
    n = flat.numel()
    for s in range(0, n, chunk_elems):
        m = min(chunk_elems, n - s)
        z = torch.randn(m, generator=g, device=out.device, dtype=torch.float32)
        flat[s:s + m].copy_(z.mul_(std))
    return out


def torch_dtype(dtype: str):
    import torch

    return {"bf16": torch.bfloat16, "f32": torch.float32}[dtype]


def host_to_torch(a: np.ndarray, dtype: str, device=None):
    """A numpy storage array as a torch tensor of the storage dtype."""
    import torch

    if dtype == "bf16":
        t = torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).view(torch.bfloat16)
    else:
        t = torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32))
    return t if device is None else t.to(device)


def torch_to_host(t, dtype: str) -> np.ndarray:
    """Bytes of a torch tensor back in the numpy storage representation."""
    import torch

    t = t.detach().contiguous().cpu()
    if dtype == "bf16":
        return t.view(torch.int16).numpy().view(np.uint16).copy()
    return t.numpy().astype(np.float32, copy=True)


def device_expert_weights(shape: LayerShape, seed: int, device, layer: int = 0):
    """W1, V1 [E,F,D] and W2 [E,D,F] drawn on ``device``, one stream per
    (layer, tensor, expert).  All experts of a tensor share one contiguous
    allocation, so an expert is a plain offset into it."""
    import torch

    D, F, E = shape.d_model, shape.ffn_hidden, shape.n_experts
    tdt = torch_dtype(shape.dtype)
    w1 = torch.empty((E, F, D), dtype=tdt, device=device)
    v1 = torch.empty((E, F, D), dtype=tdt, device=device)
    w2 = torch.empty((E, D, F), dtype=tdt, device=device)
    for e in range(E):
        device_normal_(w1[e], W_STD, seed, "dev-w1", layer, e)
        device_normal_(v1[e], W_STD, seed, "dev-v1", layer, e)
        device_normal_(w2[e], W_STD, seed, "dev-w2", layer, e)
    return w1, v1, w2


def stack_router(shape: LayerShape, seed: int, layer: int) -> np.ndarray:
    """Router W_r [D, E] of layer ``layer`` of a stack of MoE layers."""
    return host_normal((shape.d_model, shape.n_experts), W_STD, shape.dtype, seed, "stack-w_r",
                       layer)


def device_stack_layers(shape: LayerShape, n_layers: int, seed: int, device):
    """A stack of independently seeded layers on ``device``: per layer the
    tuple (W_r, W1, V1, W2), the experts drawn on the device."""
    layers = []
    for l in range(n_layers):
        w_r = host_to_torch(stack_router(shape, seed, l), shape.dtype, device)
        layers.append((w_r,) + device_expert_weights(shape, seed + 1 + l, device, layer=l))
    return layers


def stack_batch(shape: LayerShape, T: int, seed: int, step: int) -> np.ndarray:
    """The fresh tokens [T, D] of decode step ``step`` of a stack (reading
    C10: every step takes new seeded tokens)."""
    return host_normal((T, shape.d_model), X_STD, shape.dtype, seed, "stack-x", T, step)


# --------------------------------------------------------------------------
# self-attention block of a decoder layer
# --------------------------------------------------------------------------


@dataclasses.dataclass(frozen=True)
class AttnShape:
    """Grouped-query self-attention: n_heads query heads share n_kv_heads
    key/value heads of head_dim; (n_heads + 2 n_kv_heads) * head_dim is the
    width of the fused query/key/value projection (Table 1's D_qkv_hidden)."""
    d_model: int
    n_heads: int
    n_kv_heads: int
    head_dim: int
    rope_base: float = 500000.0
    dtype: str = "bf16"

    @property
    def qkv_rows(self) -> int:
        return (self.n_heads + 2 * self.n_kv_heads) * self.head_dim

    @property
    def ctx_width(self) -> int:
        return self.n_heads * self.head_dim


# 48 query heads and 8 key/value heads of 128: D_qkv_hidden = 8,192 (Table 1)
DBRX_ATTN = AttnShape(6144, 48, 8, 128)


def cache_std(shape: AttnShape) -> float:
    """Standard deviation of a projected key or value for unit-RMS input and
    N(0, W_STD^2) weights: the scale of the synthetic earlier cache entries."""
    return W_STD * float(np.sqrt(shape.d_model))


def host_attn_weights(shape: AttnShape, seed: int, layer: int = 0):
    """w_qkv [(Hq + 2 Hkv) dh, D] and w_o [D, Hq dh], N(0, W_STD^2)."""
    w_qkv = host_normal((shape.qkv_rows, shape.d_model), W_STD, shape.dtype, seed, "wqkv", layer)
    w_o = host_normal((shape.d_model, shape.ctx_width), W_STD, shape.dtype, seed, "wo", layer)
    return w_qkv, w_o


def host_kv_cache(shape: AttnShape, n_seq: int, max_len: int, seed: int, layer: int = 0):
    """Key and value caches [n_seq, Hkv, max_len, dh] filled with synthetic
    earlier entries (normal, at the scale a projection produces)."""
    dims = (n_seq, shape.n_kv_heads, max_len, shape.head_dim)
    k = host_normal(dims, cache_std(shape), shape.dtype, seed, "kcache", layer)
    v = host_normal(dims, cache_std(shape), shape.dtype, seed, "vcache", layer)
    return k, v


def device_attn_weights(shape: AttnShape, seed: int, device, layer: int = 0):
    import torch

    tdt = torch_dtype(shape.dtype)
    w_qkv = torch.empty((shape.qkv_rows, shape.d_model), dtype=tdt, device=device)
    w_o = torch.empty((shape.d_model, shape.ctx_width), dtype=tdt, device=device)
    device_normal_(w_qkv, W_STD, seed, "dev-wqkv", layer)
    device_normal_(w_o, W_STD, seed, "dev-wo", layer)
    return w_qkv, w_o


def device_kv_cache(shape: AttnShape, n_seq: int, max_len: int, seed: int, device,
                    layer: int = 0):
    import torch

    tdt = torch_dtype(shape.dtype)
    dims = (n_seq, shape.n_kv_heads, max_len, shape.head_dim)
    k = torch.empty(dims, dtype=tdt, device=device)
    v = torch.empty(dims, dtype=tdt, device=device)
    device_normal_(k, cache_std(shape), seed, "dev-kcache", layer)
    device_normal_(v, cache_std(shape), seed, "dev-vcache", layer)
    return k, v
