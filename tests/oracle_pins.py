"""Pins of the fp64 oracle against facts fixed outside the oracle itself.

Each ``pin_*`` takes an ``oracle.OracleLib`` and raises ``AssertionError`` if
the oracle disagrees with:

* exact integer arithmetic (router logits of small integers);
* brute force over every K-subset (top-k);
* a closed form of the gates that is not the oracle's formula (pairwise
  exponentials), the K=1 and K=E special cases (scipy softmax);
* Python's stable ``sorted`` (dispatch);
* closed forms of the SiLU-GLU expert on one-hot weights (sigma(ln 3) = 3/4),
  its linear regime (a library matmul) and the odd-part identity
  silu(z) - silu(-z) = z, which reduces the expert to a bilinear form;
* invariants of the layer: identical experts, K = 1, token permutation, expert
  relabelling, busy full loading (Sec. 4.2), linearity in W2 and V1.

The same pins are run against deliberately broken copies of the oracle in
``test_oracle_mutations.py``, so each plausible mistake is shown to fail one.
"""
from __future__ import annotations

import itertools
import math

import numpy as np

from paper_2506_23635_gb300 import inputs as gen

LN3 = math.log(3.0)


def _close(a, b, rtol, atol=0.0, msg=""):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    assert a.shape == b.shape, f"{msg}: shape {a.shape} vs {b.shape}"
    err = np.abs(a - b)
    lim = atol + rtol * np.abs(b)
    assert np.all(err <= lim), f"{msg}: max err {err.max()} (limit {lim.max()})"


# --------------------------------------------------------------------------
# router
# --------------------------------------------------------------------------


def pin_router_exact_integers(orc):
    """Small-integer x and W_r are exact in f32 and bf16; their dot products
    are exact integers, computed here with Python ints."""
    rng = np.random.default_rng(11)
    T, D, E = 3, 7, 5
    xi = rng.integers(-8, 9, size=(T, D))
    wi = rng.integers(-8, 9, size=(D, E))
    want = np.array([[sum(int(xi[t, d]) * int(wi[d, e]) for d in range(D))
                      for e in range(E)] for t in range(T)], np.float64)
    for dt in ("f32", "bf16"):
        got = orc.router_logits(gen.store(xi, dt), gen.store(wi, dt), dt)
        assert np.array_equal(got, want), f"router logits ({dt})"


# --------------------------------------------------------------------------
# softmax -> top-k -> renormalised gates
# --------------------------------------------------------------------------


def pin_topk_bruteforce(orc):
    rng = np.random.default_rng(12)
    for E in (2, 3, 5, 8):
        for K in range(1, E + 1):
            lg = rng.normal(size=(40, E)) * 2.0
            idx, _ = orc.topk_gates(lg, K)
            for t in range(lg.shape[0]):
                best = max(itertools.combinations(range(E), K),
                           key=lambda c: sum(lg[t, list(c)]))
                assert set(idx[t].tolist()) == set(best), "top-k set"
                vals = lg[t, idx[t]]
                assert np.all(vals[:-1] > vals[1:]), "top-k order"


def pin_topk_ties(orc):
    idx, _ = orc.topk_gates(np.array([[1.0, 3.0, 3.0, 2.0]]), 2)
    assert idx.tolist() == [[1, 2]], "tie keeps lower index first"
    idx, _ = orc.topk_gates(np.array([[5.0, 5.0, 5.0, 5.0]]), 3)
    assert idx.tolist() == [[0, 1, 2]], "all-equal logits"
    idx, _ = orc.topk_gates(np.array([[0.0, 7.0, 7.0, 7.0, 1.0]]), 4)
    assert idx.tolist() == [[1, 2, 3, 4]], "ties then smaller"


def pin_gates_closed_form(orc):
    """g_k = 1 / sum_j exp(l_j - l_k) over the selected j."""
    rng = np.random.default_rng(13)
    E, K = 16, 4
    lg = rng.normal(size=(64, E)) * 3.0
    idx, gate = orc.topk_gates(lg, K)
    for t in range(lg.shape[0]):
        sel = [lg[t, e] for e in idx[t]]
        want = [1.0 / sum(math.exp(lj - lk) for lj in sel) for lk in sel]
        _close(gate[t], want, 1e-13, msg="gate closed form")
    _close(gate.sum(axis=1), np.ones(lg.shape[0]), 1e-14, msg="sum of gates")


def pin_gates_special_cases(orc):
    from scipy.special import softmax

    rng = np.random.default_rng(14)
    lg = rng.normal(size=(32, 6)) * 4.0
    _, g1 = orc.topk_gates(lg, 1)
    assert np.all(g1 == 1.0), "K=1 gate is exactly 1"
    idx, gE = orc.topk_gates(lg, 6)
    want = np.take_along_axis(softmax(lg, axis=1), idx.astype(np.int64), axis=1)
    _close(gE, want, 1e-13, msg="K=E gates = softmax")


# --------------------------------------------------------------------------
# dispatch
# --------------------------------------------------------------------------


def pin_dispatch_stable_sort(orc):
    rng = np.random.default_rng(15)
    for (T, E, K) in ((1, 16, 4), (37, 16, 4), (64, 5, 2), (300, 7, 1), (9, 3, 3)):
        idx = np.stack([rng.permutation(E)[:K] for _ in range(T)]).astype(np.int32)
        flat = idx.reshape(-1)
        S = flat.size
        counts, offsets, perm, inv = orc.dispatch(idx, E)
        assert np.array_equal(counts, np.bincount(flat, minlength=E)), "counts"
        assert np.array_equal(offsets, np.concatenate([[0], np.cumsum(counts)])), "offsets"
        want = sorted(range(S), key=lambda s: (int(flat[s]), s))
        assert perm.tolist() == want, "perm = stable sort by expert"
        assert np.array_equal(inv[perm], np.arange(S)), "inv_perm inverts perm"


# --------------------------------------------------------------------------
# SiLU-GLU expert
# --------------------------------------------------------------------------


def _silu(z):
    return z / (1.0 + math.exp(-z))


def pin_expert_one_hot_closed_form(orc):
    """One-hot W1/V1 rows pick x entries; sigma(ln 3) = 3/4, sigma(-ln 3) = 1/4.

    D=5, F=3 so a transposed operand cannot pass."""
    D, F = 5, 3
    x = np.array([LN3, -LN3, 2.0, 0.5, 0.0])
    w1 = np.zeros((F, D)); v1 = np.zeros((F, D))
    for f, (d1, d2, c2) in enumerate(((0, 2, 1.0), (1, 3, 2.0), (4, 2, -1.0))):
        w1[f, d1] = 1.0
        v1[f, d2] = c2
    w2 = np.array([[1, 0, 0], [0, 1, 0], [1, 1, 0], [0, 0, 1], [2, 0, -1]], np.float64)
    x32 = x.astype(np.float32).astype(np.float64)
    h, y = orc.expert_ffn(x32, gen.store(w1, "f32"), gen.store(v1, "f32"),
                          gen.store(w2, "f32"), "f32")
    h_want = np.array([0.75 * LN3 * 2.0, -0.25 * LN3 * 1.0, 0.0])
    y_want = np.array([h_want[0], h_want[1], h_want[0] + h_want[1], h_want[2],
                       2.0 * h_want[0] - h_want[2]])
    _close(h, h_want, 1e-7, 1e-12, msg="GLU hidden, closed form")
    _close(y, y_want, 1e-7, 1e-12, msg="expert output, closed form")


def pin_expert_linear_regime(orc):
    """With b = 1 and a >= 50, SiLU(a) = a to 1e-21, so the expert is the
    plain product W2 (W1 x); with a <= -50 it is 0."""
    rng = np.random.default_rng(16)
    D, F = 16, 24
    x = rng.normal(size=D); x[0] = 1.0
    w1 = rng.normal(size=(F, D)) * 0.01; w1[:, 0] = 60.0
    v1 = np.zeros((F, D)); v1[:, 0] = 1.0
    w2 = rng.normal(size=(D, F))
    S = lambda a: gen.store(a, "f32")
    xs = S(x).astype(np.float64)
    w1s, v1s, w2s = (S(a).astype(np.float64) for a in (w1, v1, w2))
    _, y = orc.expert_ffn(xs, S(w1), S(v1), S(w2), "f32")
    _close(y, w2s @ (w1s @ xs), 1e-12, 1e-12, msg="linear regime")
    _, yneg = orc.expert_ffn(xs, S(-w1), S(v1), S(w2), "f32")
    assert np.max(np.abs(yneg)) < 1e-15, "negative regime is zero"


def pin_expert_odd_part(orc):
    """silu(z) - silu(-z) = z, so y(W1) - y(-W1) = W2 ((W1 x) * (V1 x))."""
    rng = np.random.default_rng(17)
    D, F = 24, 40
    for dt in ("f32", "bf16"):
        x = gen.store(rng.normal(size=D), dt)
        w1 = gen.store(rng.normal(size=(F, D)) * 0.3, dt)
        v1 = gen.store(rng.normal(size=(F, D)) * 0.3, dt)
        w2 = gen.store(rng.normal(size=(D, F)) * 0.3, dt)
        w1n = gen.store(-gen.to_f64(w1, dt), dt)  # exact negation
        x64 = gen.to_f64(x, dt)
        _, yp = orc.expert_ffn(x64, w1, v1, w2, dt)
        _, yn = orc.expert_ffn(x64, w1n, v1, w2, dt)
        W1, V1, W2 = (gen.to_f64(a, dt) for a in (w1, v1, w2))
        want = W2 @ ((W1 @ x64) * (V1 @ x64))
        _close(yp - yn, want, 1e-11, 1e-11, msg=f"odd part ({dt})")


# --------------------------------------------------------------------------
# whole-layer invariants
# --------------------------------------------------------------------------


def _small_layer(seed=21, T=12, E=5, K=2, D=32, F=48, dt="f32"):
    shape = gen.LayerShape(D, F, E, K, dt)
    L = gen.host_layer(shape, T, seed)
    # larger weights than the DBRX recipe so that every term is visible
    rng = np.random.default_rng(seed)
    L.w1 = gen.store(rng.normal(size=(E, F, D)) * 0.2, dt)
    L.v1 = gen.store(rng.normal(size=(E, F, D)) * 0.2, dt)
    L.w2 = gen.store(rng.normal(size=(E, D, F)) * 0.2, dt)
    L.w_r = gen.store(rng.normal(size=(D, E)) * 0.5, dt)
    L.x = gen.gap_condition_tokens(L.x, L.w_r, shape, seed, 1e-3)
    return L


def pin_layer_identical_experts(orc):
    """Identical experts: the layer is one expert, whatever the routing."""
    L = _small_layer()
    sh = L.shape
    for a in (L.w1, L.v1, L.w2):
        a[:] = a[0]
    out, _, gate = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    x64 = gen.to_f64(L.x, sh.dtype)
    for t in range(x64.shape[0]):
        _, y = orc.expert_ffn(x64[t], L.w1[0], L.v1[0], L.w2[0], sh.dtype)
        _close(out[t], y, 1e-12, 1e-12, msg="identical experts")


def pin_layer_k1_one_expert(orc):
    """K = 1: the output is exactly the arg-max expert's output."""
    L = _small_layer(K=1)
    sh = L.shape
    out, idx, gate = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, 1)
    lg = gen.to_f64(L.x, sh.dtype) @ gen.to_f64(L.w_r, sh.dtype)
    assert np.array_equal(idx[:, 0], np.argmax(lg, axis=1)), "K=1 expert"
    assert np.all(gate == 1.0)
    x64 = gen.to_f64(L.x, sh.dtype)
    for t in range(x64.shape[0]):
        e = int(idx[t, 0])
        _, y = orc.expert_ffn(x64[t], L.w1[e], L.v1[e], L.w2[e], sh.dtype)
        assert np.array_equal(out[t], y), "K=1 output"


def pin_layer_token_permutation(orc):
    L = _small_layer()
    sh = L.shape
    out, idx, _ = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    p = np.random.default_rng(5).permutation(L.x.shape[0])
    out_p, idx_p, _ = orc.layer_tokens(L.x[p], L.w_r, L.w1, L.v1, L.w2, sh.dtype,
                                       sh.top_k)
    _close(out_p, out[p], 1e-13, 1e-13, msg="token permutation")
    assert np.array_equal(idx_p, idx[p])


def pin_layer_expert_relabel(orc):
    L = _small_layer()
    sh = L.shape
    out, idx, _ = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    s = np.random.default_rng(6).permutation(sh.n_experts)
    out_s, idx_s, _ = orc.layer_tokens(L.x, L.w_r[:, s], L.w1[s], L.v1[s], L.w2[s],
                                       sh.dtype, sh.top_k)
    _close(out_s, out, 1e-13, 1e-13, msg="expert relabelling")
    assert np.array_equal(s[idx_s], idx)


def pin_layer_busy_full_loading(orc):
    """Sec. 4.2: computing all experts and zeroing the unselected ones in the
    weighted sum gives the same layer."""
    L = _small_layer()
    sh = L.shape
    out, _, _ = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    dense = orc.layer_dense_masked(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    _close(dense, out, 1e-13, 1e-13, msg="busy full loading")


def pin_layer_linear_in_w2_v1(orc):
    L = _small_layer()
    sh = L.shape
    out, _, _ = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    out2, _, _ = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2 * 2, sh.dtype, sh.top_k)
    out3, _, _ = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1 * 4, L.w2, sh.dtype, sh.top_k)
    assert np.array_equal(out2, 2 * out), "linear in W2"
    assert np.array_equal(out3, 4 * out), "linear in V1"


def pin_layer_steps_agree(orc):
    """The step-by-step route (dispatch, per-slot experts, combine) equals the
    per-token route."""
    L = _small_layer(T=9, E=4, K=3)
    sh = L.shape
    out, idx, gate = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    st = orc.layer_steps(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    assert np.array_equal(st["idx"], idx)
    _close(st["gate"], gate, 1e-15, msg="gates")
    _close(st["out"], out, 1e-13, 1e-13, msg="steps vs tokens")
    assert st["counts"].sum() == idx.size


def pin_experts_partition_sums_to_layer(orc):
    """Sec. 4.3: the all-reduce of the nodes' shares is the weighted sum.
    The share of [0, E) is the layer (same arithmetic, bit for bit); the
    shares of any partition of [0, E) into contiguous ranges add up to it;
    a residual is carried by the share it is given to."""
    L = _small_layer(E=7, K=3)
    sh = L.shape
    E = sh.n_experts
    out, _, _ = orc.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    whole = orc.layer_experts_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k, 0, E)
    assert np.array_equal(whole, out), "share of every expert"
    for cuts in ((0, 3, 7), (0, 1, 4, 6, 7), tuple(range(E + 1))):
        parts = [orc.layer_experts_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k,
                                          b, e) for b, e in zip(cuts[:-1], cuts[1:])]
        _close(np.sum(parts, axis=0), out, 1e-12, 1e-13, msg=f"partition {cuts}")
    res = np.random.default_rng(9).normal(size=out.shape)
    first = orc.layer_experts_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k, 0, 3,
                                     residual=res)
    rest = orc.layer_experts_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k, 3, E)
    _close(first + rest, out + res, 1e-12, 1e-13, msg="residual on one share")


def pin_experts_single_expert_k1(orc):
    """K = 1 and a one-expert share [e, e+1): a token whose arg-max logit
    (numpy) is e gets exactly that expert's output, every other token an
    exact zero row."""
    L = _small_layer(K=1)
    sh = L.shape
    x64 = gen.to_f64(L.x, sh.dtype)
    best = np.argmax(x64 @ gen.to_f64(L.w_r, sh.dtype), axis=1)
    for e in range(sh.n_experts):
        part = orc.layer_experts_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, 1, e, e + 1)
        for t in range(x64.shape[0]):
            if best[t] == e:
                _, y = orc.expert_ffn(x64[t], L.w1[e], L.v1[e], L.w2[e], sh.dtype)
                assert np.array_equal(part[t], y), "the selected expert's output"
            else:
                assert not np.any(part[t]), "another node's expert contributes nothing"


# --------------------------------------------------------------------------
# stack glue (reading C9): RMSNorm0 and the residual stream
# --------------------------------------------------------------------------


def pin_rmsnorm0_closed_form(orc):
    """[3, 4]: mean square 12.5, so the row becomes [3, 4] / sqrt(12.5 + eps);
    in general mean(out^2) = ms / (ms + eps) and the direction is kept."""
    eps = 1e-6
    out = orc.rmsnorm0(np.array([[3.0, 4.0]]), eps)
    _close(out[0], np.array([3.0, 4.0]) / math.sqrt(12.5 + eps), 1e-15, msg="rmsnorm [3,4]")
    x = np.random.default_rng(31).normal(size=(5, 24)) * 7.0
    y = orc.rmsnorm0(x, eps)
    ms = (x * x).mean(axis=1)
    _close((y * y).mean(axis=1), ms / (ms + eps), 1e-13, msg="mean square")
    ratio = y / x
    _close(ratio, np.broadcast_to(ratio[:, :1], ratio.shape), 1e-13, msg="direction kept")


def pin_round_bf16_cases(orc):
    """bf16 keeps 8 significant bits: spacing 2^-7 on [1, 2).  Exact cases:
    1 + 2^-8 is a tie and goes to the even 1; 1 + 3*2^-8 is a tie and goes to
    the even 1 + 2^-6; 1 + 0.75*2^-7 rounds up; values already on the grid
    stay; and every float32 goes where the integer round-half-even of its bit
    pattern sends it."""
    cases = {1.0 + 2.0 ** -8: 1.0, 1.0 + 3 * 2.0 ** -8: 1.0 + 2.0 ** -6,
             1.0 + 0.75 * 2.0 ** -7: 1.0 + 2.0 ** -7, -(1.0 + 2.0 ** -8): -1.0,
             3.0: 3.0, 0.0: 0.0, 2.0 ** -20 * (1 + 2.0 ** -8): 2.0 ** -20}
    got = orc.round_bf16(np.array(list(cases)))
    assert np.array_equal(got, np.array(list(cases.values()))), "bf16 rounding cases"
    x32 = np.random.default_rng(38).normal(size=512).astype(np.float32) * 100
    want = gen.bf16_bits_to_f64(gen.f32_to_bf16_bits(x32))
    assert np.array_equal(orc.round_bf16(x32.astype(np.float64)), want), "vs bit rounding"


def _stack_layers(seed, n_layers, D=32, F=48, E=5, K=2, dt="f32"):
    rng = np.random.default_rng(seed)
    layers = []
    for _ in range(n_layers):
        layers.append((gen.store(rng.normal(size=(D, E)) * 0.5, dt),
                       gen.store(rng.normal(size=(E, F, D)) * 0.2, dt),
                       gen.store(rng.normal(size=(E, F, D)) * 0.2, dt),
                       gen.store(rng.normal(size=(E, D, F)) * 0.2, dt)))
    return layers


def pin_stack_zero_w2_is_identity(orc):
    """Zero down projections make every MoE block zero: the stack returns its
    input exactly."""
    layers = [(w_r, w1, v1, np.zeros_like(w2)) for (w_r, w1, v1, w2) in _stack_layers(32, 3)]
    x0 = gen.store(np.random.default_rng(33).normal(size=(4, 32)), "f32")
    out, _ = orc.stack_tokens(x0, layers, "f32", 2, 1e-6)
    assert np.array_equal(out, gen.to_f64(x0, "f32")), "zero MoE blocks"


def pin_stack_prenorm_scale_invariance(orc):
    """The pre-norm makes a block's input independent of the residual's scale,
    so one block adds the same vector to x and to c*x: f(c x) - c x = f(x) - x."""
    layers = _stack_layers(34, 1)
    x0 = np.random.default_rng(35).normal(size=(4, 32))
    a, _ = orc.stack_tokens(x0, layers, "f64", 2, 1e-12)
    b, _ = orc.stack_tokens(3.0 * x0, layers, "f64", 2, 1e-12)
    _close(b - 3.0 * x0, a - x0, 1e-9, 1e-12, msg="pre-norm scale invariance")


def pin_stack_residual_composition(orc):
    """Two stacked blocks = block 1 applied to the output of block 0, and each
    block adds its MoE output to the residual (checked against the single
    layer with the residual passed in)."""
    layers = _stack_layers(36, 2)
    x0 = np.random.default_rng(37).normal(size=(3, 32))
    two, _ = orc.stack_tokens(x0, layers, "f64", 2, 1e-6)
    one, _ = orc.stack_tokens(x0, layers[:1], "f64", 2, 1e-6)
    w_r, w1, v1, w2 = layers[1]
    xn = orc.rmsnorm0(one, 1e-6)
    moe, _, _ = orc.layer_tokens(xn, w_r, w1, v1, w2, "f32", 2, x_dtype="f64")
    _close(two, one + moe, 1e-13, 1e-13, msg="residual composition")


# --------------------------------------------------------------------------
# self-attention block of a decoder layer (readings in moe_oracle.c)
# --------------------------------------------------------------------------


def _rope_generator(dh, base):
    """Skew-symmetric generator of the rotary embedding: the plane of dims
    (i, i + dh/2) turns at angular rate base^(-2i/dh)."""
    G = np.zeros((dh, dh))
    h = dh // 2
    for i in range(h):
        w = base ** (-2.0 * i / dh)
        G[i + h, i] = w
        G[i, i + h] = -w
    return G


def pin_rope_matrix_exponential(orc):
    """rope(u, p) = expm(p G) u for the generator G (scipy's matrix
    exponential, not the oracle's cos/sin); position 0 is the identity and
    every head keeps its norm."""
    from scipy.linalg import expm
    rng = np.random.default_rng(41)
    for dh, base in ((8, 10000.0), (16, 500000.0), (2, 7.0)):
        u = rng.normal(size=(4, 3, dh))
        pos = np.array([0, 1, 17, 250], np.int32)
        got = orc.rope(u, pos, base)
        G = _rope_generator(dh, base)
        for t in range(4):
            R = expm(pos[t] * G)
            _close(got[t], u[t] @ R.T, 1e-10, 1e-12, f"rope dh={dh} pos={pos[t]}")
        assert np.array_equal(got[0], u[0]), "rope at position 0"
        _close(np.linalg.norm(got, axis=-1), np.linalg.norm(u, axis=-1), 1e-12, 0, "rope norm")


def _sdpa(q, k, v, causal):
    """torch's scaled_dot_product_attention in fp64 on the CPU; q [Hq, n, dh],
    k, v [Hkv, m, dh]; grouped queries by repeating each key/value head."""
    import torch
    g = q.shape[0] // k.shape[0]
    tq = torch.from_numpy(q)[None]
    tk = torch.from_numpy(k).repeat_interleave(g, dim=0)[None]
    tv = torch.from_numpy(v).repeat_interleave(g, dim=0)[None]
    out = torch.nn.functional.scaled_dot_product_attention(tq, tk, tv, is_causal=causal)
    return out[0].numpy()


def pin_attention_against_sdpa(orc):
    """Prefill of one sequence (positions 0..n-1, causal) and decode tokens of
    several sequences at scattered positions, against torch's attention."""
    rng = np.random.default_rng(43)
    Hq, Hkv, dh, L = 6, 2, 16, 40
    # prefill: tokens 0..n-1 of sequence 1
    n = 23
    kc = rng.normal(size=(3, Hkv, L, dh))
    vc = rng.normal(size=(3, Hkv, L, dh))
    q = rng.normal(size=(n, Hq, dh)) * 2.0
    seq = np.full(n, 1, np.int32)
    pos = np.arange(n, dtype=np.int32)
    got = orc.attention(q, kc, vc, seq, pos)
    want = _sdpa(q.transpose(1, 0, 2), kc[1, :, :n], vc[1, :, :n], True).transpose(1, 0, 2)
    _close(got, want, 1e-10, 1e-12, "attention prefill vs sdpa")
    # decode: one token per sequence, each at its own position
    seq = np.array([2, 0, 1], np.int32)
    pos = np.array([39, 0, 11], np.int32)
    q = rng.normal(size=(3, Hq, dh)) * 2.0
    got = orc.attention(q, kc, vc, seq, pos)
    for t in range(3):
        s, p = seq[t], pos[t]
        want = _sdpa(q[t][:, None, :], kc[s, :, :p + 1], vc[s, :, :p + 1], False)[:, 0, :]
        _close(got[t], want, 1e-10, 1e-12, f"attention decode token {t}")
    assert np.array_equal(got[1], np.repeat(vc[0, :, 0], Hq // Hkv, axis=0)), \
        "one cached position: ctx is that value row, for every head of the group"


def _sa_case(rng, D=24, Hq=4, Hkv=2, dh=8, n_seq=2, L=12, dt="f32"):
    nr = (Hq + 2 * Hkv) * dh
    w_qkv = gen.store(rng.normal(size=(nr, D)) * 0.2, dt)
    w_o = gen.store(rng.normal(size=(D, Hq * dh)) * 0.2, dt)
    kc = gen.to_f64(gen.store(rng.normal(size=(n_seq, Hkv, L, dh)), dt), dt)
    vc = gen.to_f64(gen.store(rng.normal(size=(n_seq, Hkv, L, dh)), dt), dt)
    return w_qkv, w_o, kc, vc


def pin_sa_block_composition(orc):
    """The block is rmsnorm0 -> projection (numpy matmul) -> rotary (matrix
    exponential) -> cache write -> torch attention -> output projection ->
    residual add; D differs from Hq*dh so an operand read the wrong way
    round cannot fit."""
    from scipy.linalg import expm
    rng = np.random.default_rng(47)
    D, Hq, Hkv, dh, base, eps = 24, 4, 2, 8, 1000.0, 1e-6
    w_qkv, w_o, kc, vc = _sa_case(rng, D, Hq, Hkv, dh)
    x = rng.normal(size=(5, D)) * 3.0
    seq = np.array([0, 0, 0, 1, 1], np.int32)
    pos = np.array([4, 5, 6, 0, 1], np.int32)
    got, gk, gv = orc.sa_forward(x, w_qkv, w_o, "f32", Hq, Hkv, base, eps, seq, pos, kc, vc)
    xn = x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + eps)
    qkv = xn @ gen.to_f64(w_qkv, "f32").T
    q = qkv[:, :Hq * dh].reshape(5, Hq, dh)
    k = qkv[:, Hq * dh:(Hq + Hkv) * dh].reshape(5, Hkv, dh)
    v = qkv[:, (Hq + Hkv) * dh:].reshape(5, Hkv, dh)
    G = _rope_generator(dh, base)
    R = [expm(p * G) for p in pos]
    q = np.stack([q[t] @ R[t].T for t in range(5)])
    k = np.stack([k[t] @ R[t].T for t in range(5)])
    wk, wv = kc.copy(), vc.copy()
    for t in range(5):
        wk[seq[t], :, pos[t]] = k[t]
        wv[seq[t], :, pos[t]] = v[t]
    _close(gk, wk, 1e-10, 1e-12, "cached keys")
    _close(gv, wv, 1e-10, 1e-12, "cached values")
    ctx = np.stack([_sdpa(q[t][:, None, :], wk[seq[t], :, :pos[t] + 1],
                          wv[seq[t], :, :pos[t] + 1], False)[:, 0, :] for t in range(5)])
    want = x + ctx.reshape(5, Hq * dh) @ gen.to_f64(w_o, "f32").T
    _close(got, want, 1e-9, 1e-11, "self-attention block")


def pin_sa_incremental_equals_prefill(orc):
    """Prefilling a sequence in one call equals feeding its tokens one per
    call (the cache carries the earlier keys and values); a second sequence
    in the same call does not disturb the first."""
    rng = np.random.default_rng(53)
    D, Hq, Hkv, dh, base, eps = 24, 4, 2, 8, 1000.0, 1e-6
    w_qkv, w_o, kc, vc = _sa_case(rng, D, Hq, Hkv, dh)
    n = 6
    x = rng.normal(size=(n, D))
    seq = np.zeros(n, np.int32)
    pos = np.arange(n, dtype=np.int32)
    full, fk, fv = orc.sa_forward(x, w_qkv, w_o, "f32", Hq, Hkv, base, eps, seq, pos, kc, vc)
    k1, v1 = kc, vc
    for t in range(n):
        o, k1, v1 = orc.sa_forward(x[t:t + 1], w_qkv, w_o, "f32", Hq, Hkv, base, eps,
                                   seq[t:t + 1], pos[t:t + 1], k1, v1)
        _close(o[0], full[t], 1e-10, 1e-12, f"incremental token {t}")
    _close(k1, fk, 0, 1e-14, "incremental caches")
    x2 = rng.normal(size=(1, D))
    both, _, _ = orc.sa_forward(np.vstack([x, x2]), w_qkv, w_o, "f32", Hq, Hkv, base, eps,
                                np.append(seq, 1).astype(np.int32),
                                np.append(pos, 3).astype(np.int32), kc, vc)
    _close(both[:n], full, 1e-10, 1e-12, "another sequence in the same call")


def pin_sa_causality(orc):
    """Changing a later token of a prefill leaves every earlier token's
    output unchanged and changes the later one."""
    rng = np.random.default_rng(59)
    D, Hq, Hkv, dh = 24, 4, 2, 8
    w_qkv, w_o, kc, vc = _sa_case(rng, D, Hq, Hkv, dh)
    n = 5
    x = rng.normal(size=(n, D))
    seq = np.zeros(n, np.int32)
    pos = np.arange(n, dtype=np.int32)
    a, _, _ = orc.sa_forward(x, w_qkv, w_o, "f32", Hq, Hkv, 1000.0, 1e-6, seq, pos, kc, vc)
    x[3] += 1.0
    b, _, _ = orc.sa_forward(x, w_qkv, w_o, "f32", Hq, Hkv, 1000.0, 1e-6, seq, pos, kc, vc)
    assert np.array_equal(a[:3], b[:3]), "earlier tokens saw a later one"
    assert not np.allclose(a[3:], b[3:]), "later tokens did not change"


def pin_sa_bf16_storage(orc):
    """With bf16 storage the cached keys and values are bf16 values (the
    rounding of the f32-storage result); a zero output projection leaves
    the residual unchanged."""
    rng = np.random.default_rng(61)
    D, Hq, Hkv, dh = 24, 4, 2, 8
    w_qkv, w_o, kc, vc = _sa_case(rng, D, Hq, Hkv, dh, dt="bf16")
    x = rng.normal(size=(3, D))
    seq = np.array([0, 1, 1], np.int32)
    pos = np.array([2, 7, 8], np.int32)
    zero_o = gen.store(np.zeros((D, Hq * dh)), "bf16")
    out, k, v = orc.sa_forward(x, w_qkv, zero_o, "bf16", Hq, Hkv, 1000.0, 1e-6, seq, pos, kc, vc)
    assert np.array_equal(out, x), "zero output projection"
    for c in (k, v):
        assert np.array_equal(gen.to_f64(gen.store(c, "bf16"), "bf16"), c), "cache not bf16"


def pin_sa_bf16_block_composition(orc):
    """With bf16 storage the block is the composition of pin_sa_block_-
    composition with every stored activation rounded to bf16 by numpy's bit
    rounding (independent of the oracle's): the normalised input, the rotated
    queries and keys, the values, and ctx."""
    from scipy.linalg import expm

    def r16(a):
        return gen.to_f64(gen.store(a, "bf16"), "bf16")

    rng = np.random.default_rng(71)
    D, Hq, Hkv, dh, base, eps = 24, 4, 2, 8, 1000.0, 1e-6
    w_qkv, w_o, kc, vc = _sa_case(rng, D, Hq, Hkv, dh, dt="bf16")
    n = 5
    x = rng.normal(size=(n, D)) * 3.0
    seq = np.array([0, 0, 1, 1, 1], np.int32)
    pos = np.array([3, 4, 0, 1, 2], np.int32)
    got, _, _ = orc.sa_forward(x, w_qkv, w_o, "bf16", Hq, Hkv, base, eps, seq, pos, kc, vc)
    xn = r16(x / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + eps))
    qkv = xn @ gen.to_f64(w_qkv, "bf16").T
    q = qkv[:, :Hq * dh].reshape(n, Hq, dh)
    k = qkv[:, Hq * dh:(Hq + Hkv) * dh].reshape(n, Hkv, dh)
    v = r16(qkv[:, (Hq + Hkv) * dh:].reshape(n, Hkv, dh))
    G = _rope_generator(dh, base)
    R = [expm(p * G) for p in pos]
    q = r16(np.stack([q[t] @ R[t].T for t in range(n)]))
    k = r16(np.stack([k[t] @ R[t].T for t in range(n)]))
    wk, wv = kc.copy(), vc.copy()
    for t in range(n):
        wk[seq[t], :, pos[t]] = k[t]
        wv[seq[t], :, pos[t]] = v[t]
    ctx = r16(np.stack([_sdpa(q[t][:, None, :], wk[seq[t], :, :pos[t] + 1],
                              wv[seq[t], :, :pos[t] + 1], False)[:, 0, :] for t in range(n)]))
    want = x + ctx.reshape(n, Hq * dh) @ gen.to_f64(w_o, "bf16").T
    _close(got, want, 1e-9, 1e-11, "self-attention block, bf16 storage")


def pin_decoder_layer_composition(orc):
    """A decoder layer whose output projection is zero is the MoE stack
    layer alone (pinned above); with it, the layer is the self-attention
    block followed by that stack layer."""
    rng = np.random.default_rng(67)
    D, Hq, Hkv, dh = 32, 4, 2, 8
    w_qkv, w_o, kc, vc = _sa_case(rng, D, Hq, Hkv, dh)
    (w_r, w1, v1, w2), = _stack_layers(69, 1, D=D)
    x0 = gen.store(rng.normal(size=(3, D)), "f32")
    seq = np.array([0, 1, 1], np.int32)
    pos = np.array([3, 5, 6], np.int32)
    zero_o = gen.store(np.zeros((D, Hq * dh)), "f32")
    got, _, gaps = orc.decoder_layers(gen.to_f64(x0, "f32"), [(w_qkv, zero_o, w_r, w1, v1, w2)],
                                      "f32", Hq, Hkv, 1000.0, 1e-6, 2, seq, pos, [(kc, vc)])
    want, wgaps = orc.stack_tokens(x0, [(w_r, w1, v1, w2)], "f32", 2, 1e-6)
    _close(got, want, 1e-12, 1e-14, "decoder layer with zero output projection")
    _close(gaps, wgaps, 1e-12, 0, "routing gaps")
    got, _, _ = orc.decoder_layers(gen.to_f64(x0, "f32"), [(w_qkv, w_o, w_r, w1, v1, w2)],
                                   "f32", Hq, Hkv, 1000.0, 1e-6, 2, seq, pos, [(kc, vc)])
    mid, _, _ = orc.sa_forward(gen.to_f64(x0, "f32"), w_qkv, w_o, "f32", Hq, Hkv, 1000.0, 1e-6,
                               seq, pos, kc, vc)
    want, _ = orc.stack_tokens(mid, [(w_r, w1, v1, w2)], "f64", 2, 1e-6)
    _close(got, want, 1e-12, 1e-14, "decoder layer = attention block then stack layer")


ALL_PINS = [v for k, v in sorted(globals().items()) if k.startswith("pin_")]
