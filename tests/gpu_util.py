"""Helpers for the GPU parity tests: tolerance checks and device copies."""
from __future__ import annotations

import numpy as np
import pytest
import torch

from paper_2506_23635_gb300 import inputs as gen

# Layer-output bound for bf16 weights with fp32 accumulation: relative L2
# error <= 5e-3 and max abs error <= 2e-2 * RMS(reference output).
REL_L2 = 5e-3
MAX_ABS_OF_RMS = 2e-2
# fp32 weights and activations (the tiny layer): the same shape of bound,
# tightened to what fp32 accumulation over a few thousand terms reaches.
REL_L2_F32 = 1e-5
MAX_ABS_OF_RMS_F32 = 1e-4


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")


def bounds(dtype: str):
    return (REL_L2, MAX_ABS_OF_RMS) if dtype == "bf16" else (REL_L2_F32, MAX_ABS_OF_RMS_F32)


def assert_parity(got, want, dtype: str = "bf16", what: str = "", stored_bf16: bool = False,
                  extra=None):
    """rel L2 and max abs bounds of the path's dtype.  stored_bf16: the
    compared tensor is an intermediate that the path stores in bf16, so each
    element may also carry one bf16 rounding (2^-8 of its magnitude) beyond
    the max abs bound -- rows of very different magnitude (an attention
    output that is one value row next to one that averages thousands) make
    a bound on the RMS alone meaningless for them.  extra: a per-element
    allowance (same shape) for roundings upstream of the compared tensor
    that the oracle does not make, added to the max abs bound."""
    rel_l2, max_abs = bounds(dtype)
    g = np.asarray(got, np.float64)
    w = np.asarray(want, np.float64)
    assert g.shape == w.shape, f"{what}: shape {g.shape} vs {w.shape}"
    assert np.all(np.isfinite(g)), f"{what}: non-finite output"
    err = g - w
    nw = np.linalg.norm(w)
    rel = np.linalg.norm(err) / nw if nw > 0 else np.linalg.norm(err)
    rms = float(np.sqrt(np.mean(w * w))) if w.size else 0.0
    mx = float(np.max(np.abs(err))) if err.size else 0.0
    assert rel <= rel_l2, f"{what}: rel L2 {rel:.3e} > {rel_l2}"
    if stored_bf16 or extra is not None:
        lim = max_abs * rms + 1e-30
        if stored_bf16:
            lim = lim + 2.0 ** -8 * np.abs(w)
        if extra is not None:
            lim = lim + np.asarray(extra, np.float64)
        worst = float(np.max(np.abs(err) - lim)) if err.size else 0.0
        assert worst <= 0, (f"{what}: an element exceeds {max_abs}*RMS plus its rounding "
                            f"allowance by {worst:.3e}")
    else:
        assert mx <= max_abs * rms + 1e-30, f"{what}: max abs {mx:.3e} > {max_abs}*RMS ({rms:.3e})"
    return rel, mx / rms if rms else 0.0


def h_rounding_allowance(h_sorted, w2, offsets):
    """Per-element allowance for the GLU hidden vector's bf16 storage (the
    tensor-core and streaming paths, reading C7) in the ungated expert
    outputs y = h . W2[e]^T: each term h_f W2[e,d,f] moves by at most 2^-8 of
    itself, so the element by at most 2^-8 sum_f |h_f W2[e,d,f]| -- a bound
    that grows like sqrt(F) times the element for many terms of random sign,
    so it is capped at 3 * 2^-8 * sqrt(sum_f (h_f W2[e,d,f])^2), which is
    still the worst case up to 9 terms and five standard deviations of the
    sum of independent roundings beyond that."""
    h = np.asarray(h_sorted, np.float64)
    w = np.asarray(w2, np.float64)
    out = np.zeros((h.shape[0], w.shape[1]), np.float64)
    for e in range(w.shape[0]):
        j0, j1 = int(offsets[e]), int(offsets[e + 1])
        if j1 > j0:
            worst = np.abs(h[j0:j1]) @ np.abs(w[e]).T
            spread = np.sqrt((h[j0:j1] ** 2) @ (w[e] ** 2).T)
            out[j0:j1] = np.minimum(worst, 3.0 * spread)
    return 2.0 ** -8 * out


def to_numpy(t: torch.Tensor) -> np.ndarray:
    """Values of a device tensor as float64 (bf16 and f32 widen exactly)."""
    return t.detach().float().cpu().numpy().astype(np.float64)


def dev(a: np.ndarray, dtype: str):
    return gen.host_to_torch(a, dtype, "cuda")
