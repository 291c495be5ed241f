"""CUDA path vs the fp64 oracle, step by step and for the whole layer, on
seeded inputs that span several tiles and ragged tails.

Bars: expert indices, counts, offsets and permutations bit-exact; values
within rel L2 5e-3 and max abs 2e-2 * RMS (bf16), tighter for fp32."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_23635_gb300 import inputs as gen
from tests.gpu_util import assert_parity, h_rounding_allowance, dev, need_gpu, to_numpy

pytestmark = pytest.mark.gpu


def moe():
    need_gpu()
    from paper_2506_23635_gb300 import moe as m
    return m


# (D, F, E, K, T, dtype): tiny layer, ragged widths, K = E, E = 1,
# E = 256, minimum widths, token counts on both sides of the fused combine
# limit (64), a prefill-like batch whose experts hold 2-3 slot tiles (ragged
# reduction and output widths), and a decode batch with more down-projection
# tiles than SMs (the stream-K schedule splits tiles into heads and tails).
SMALL = [
    (256, 512, 4, 2, 8, "f32"),
    (64, 96, 8, 2, 1, "bf16"),
    (72, 40, 5, 3, 17, "bf16"),
    (128, 136, 16, 4, 65, "bf16"),
    (256, 264, 7, 7, 33, "f32"),
    (40, 24, 1, 1, 5, "bf16"),
    (512, 256, 256, 8, 130, "bf16"),
    (8, 8, 3, 2, 300, "f32"),
    (264, 520, 16, 4, 64, "bf16"),
    (200, 264, 3, 2, 400, "bf16"),
    (4096, 256, 16, 4, 16, "bf16"),  # ~250 down-projection tiles: stream-K heads and tails
]


def _random_cases(n=16, seed=77):
    """Seeded layer shapes over the validated ranges (D, F multiples of 8 up
    to 768, E up to 32, K up to min(E, 8), T from 1 to 600, a quarter fp32):
    every kernel path of the layer (one-token streaming, decode-batch
    tiles, prefill CTA pairs, CUDA-core GEMV) on shapes no table lists."""
    rng = np.random.default_rng(seed)
    out = []
    for _ in range(n):
        D = 8 * int(rng.integers(1, 97))
        F = 8 * int(rng.integers(1, 97))
        E = int(rng.integers(1, 33))
        K = int(rng.integers(1, min(E, 8) + 1))
        T = int(rng.choice([int(rng.integers(1, 17)), int(rng.integers(17, 81)),
                            int(rng.integers(81, 601))]))
        out.append((D, F, E, K, T, "f32" if rng.random() < 0.25 else "bf16"))
    return out


RANDOM = _random_cases()


def _host(case, seed=3, skew=None):
    D, F, E, K, T, dt = case
    shape = gen.LayerShape(D, F, E, K, dt)
    return gen.host_layer(shape, T, seed, skew)


def _dims(m, shape, out_dtype=None):
    tdt = gen.torch_dtype(shape.dtype)
    return m.dims(shape.d_model, shape.ffn_hidden, shape.n_experts, shape.top_k, tdt, tdt,
                  out_dtype or tdt)


def _devlayer(L):
    dt = L.shape.dtype
    return [dev(a, dt) for a in (L.x, L.w_r, L.w1, L.v1, L.w2)]


@pytest.mark.parametrize("case", SMALL + RANDOM, ids=lambda c: "D{}F{}E{}K{}T{}{}".format(*c))
def test_steps_and_layer(case):
    m = moe()
    L = _host(case)
    sh = L.shape
    d = _dims(m, sh)
    ref = oracle.layer_steps(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    x, w_r, w1, v1, w2 = _devlayer(L)

    idx, gate, logits = m.route(d, x, w_r, want_logits=True)
    assert np.array_equal(idx.cpu().numpy(), ref["idx"]), "top-k indices"
    np.testing.assert_allclose(to_numpy(gate), ref["gate"], rtol=0, atol=2e-6)
    scale = np.abs(gen.to_f64(L.x, sh.dtype)) @ np.abs(gen.to_f64(L.w_r, sh.dtype))
    assert np.all(np.abs(to_numpy(logits) - ref["logits"]) <= 1e-5 * scale + 1e-7)

    counts, offsets, perm, inv = m.dispatch(d, idx)
    assert np.array_equal(counts.cpu().numpy(), ref["counts"])
    assert np.array_equal(offsets.cpu().numpy(), ref["offsets"])
    assert np.array_equal(perm.cpu().numpy(), ref["perm"])
    assert np.array_equal(inv.cpu().numpy(), ref["inv_perm"])

    # bf16: the expert outputs come from the GLU hidden vector stored in bf16
    # (reading C7): where few terms are summed (small F) an element far above
    # the RMS can carry more of that rounding than the RMS bound, so each
    # element gets the rounding's bound (tests/gpu_util.py) as an allowance,
    # gated into the layer output, which also carries its own bf16 storage
    # rounding (reading C22)
    extra_y = extra_out = None
    stored = sh.dtype == "bf16"
    if stored:
        extra_y = h_rounding_allowance(ref["h_sorted"], gen.to_f64(L.w2, "bf16"),
                                       ref["offsets"])
        slots = ref["inv_perm"].reshape(-1, sh.top_k)
        extra_out = sum(ref["gate"][:, k, None] * extra_y[slots[:, k]]
                        for k in range(sh.top_k))
    y = m.expert_ffn(d, x, perm, offsets, w1, v1, w2)
    assert_parity(to_numpy(y), ref["y_sorted"], sh.dtype, "expert_ffn y_sorted", extra=extra_y)

    out = m.combine(d, y, inv, gate)
    assert_parity(to_numpy(out), ref["out"], sh.dtype, "combine", stored, extra=extra_out)

    out2 = m.layer_forward(d, x, w_r, w1, v1, w2)
    assert_parity(to_numpy(out2), ref["out"], sh.dtype, "layer_forward", stored,
                  extra=extra_out)
    assert m.get_last_error() == 0


@pytest.mark.parametrize("T", [1, 8, 64, 65, 200])
def test_layer_residual_and_bf16_out(T):
    """out = residual + MoE(x), written in bf16; both the fused (T <= 64) and
    the unfused combine."""
    m = moe()
    L = _host((136, 200, 6, 2, T, "bf16"), seed=7)
    sh = L.shape
    d = _dims(m, sh)
    res = gen.host_normal((T, sh.d_model), 1.0, "bf16", 7, "residual")
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k,
                                     residual=gen.to_f64(res, "bf16"))
    x, w_r, w1, v1, w2 = _devlayer(L)
    out = m.layer_forward(d, x, w_r, w1, v1, w2, residual=dev(res, "bf16"))
    assert out.dtype == torch.bfloat16
    assert_parity(to_numpy(out), want, "bf16", "layer + residual")
    d32 = _dims(m, sh, out_dtype=torch.float32)
    # the residual has the output's dtype
    out32 = m.layer_forward(d32, x, w_r, w1, v1, w2, residual=dev(res, "bf16").float())
    assert out32.dtype == torch.float32
    assert_parity(to_numpy(out32), want, "bf16", "layer + residual, f32 out")


@pytest.mark.parametrize("skew", [0.0, 0.6, 1.2])
def test_designed_router_skew(skew):
    """Zipf-skewed expert loads (few experts carry most slots)."""
    m = moe()
    L = _host((192, 128, 16, 4, 64, "bf16"), seed=11, skew=skew)
    sh = L.shape
    d = _dims(m, sh)
    ref = oracle.layer_steps(L.x, L.w_r, L.w1, L.v1, L.w2, sh.dtype, sh.top_k)
    x, w_r, w1, v1, w2 = _devlayer(L)
    idx, gate, _ = m.route(d, x, w_r)
    assert np.array_equal(idx.cpu().numpy(), ref["idx"])
    out = m.layer_forward(d, x, w_r, w1, v1, w2)
    assert_parity(to_numpy(out), ref["out"], "bf16", f"skew {skew}")


def test_all_tokens_one_expert():
    """A router that sends every token to the same top-1 expert: one expert
    holds all slots, the others none."""
    m = moe()
    D, F, E, K, T = 64, 80, 8, 1, 77
    shape = gen.LayerShape(D, F, E, K, "bf16")
    x = gen.host_normal((T, D), 1.0, "bf16", 5, "x")
    w_r = np.zeros((D, E), np.float64)
    x64 = gen.to_f64(x, "bf16")
    # W_r column 3 = sign(sum of x) direction: every token's logit 3 is large
    w_r[:, 3] = np.sign(x64.sum(0)) * 0.5
    w_r = gen.store(w_r, "bf16")
    lg = x64 @ gen.to_f64(w_r, "bf16")
    keep = lg[:, 3] > 0.1  # the other logits are exactly 0
    x = x[keep]
    T = x.shape[0]
    assert T > 10
    w1, v1, w2 = gen.host_expert_weights(shape, 5)
    d = _dims(m, shape)
    want, idx, _ = oracle.layer_tokens(x, w_r, w1, v1, w2, "bf16", K)
    assert np.all(idx == 3)
    X, WR, W1, V1, W2 = (dev(a, "bf16") for a in (x, w_r, w1, v1, w2))
    gi, _, _ = m.route(d, X, WR)
    counts, offsets, perm, inv = m.dispatch(d, gi)
    c = counts.cpu().numpy()
    assert c[3] == T and c.sum() == T
    out = m.layer_forward(d, X, WR, W1, V1, W2)
    assert_parity(to_numpy(out), want, "bf16", "one expert")


@pytest.mark.parametrize("T", [256, 257, 513])
def test_one_expert_slot_runs(T):
    """Every token to the same top-1 expert with exactly T slots: the prefill
    GEMMs cut an expert into runs of at most 256 slots (256 -> one full run,
    257 -> 128 + 129, 513 -> 171 + 171 + 171); ragged F and D; the other
    expert holds none."""
    m = moe()
    D, F, E, K = 136, 200, 2, 1
    shape = gen.LayerShape(D, F, E, K, "bf16")
    x = gen.host_normal((4 * T, D), 1.0, "bf16", 29, "x")
    x64 = gen.to_f64(x, "bf16")
    col = np.zeros(D)
    col[: D // 2] = 0.25
    w_r = np.zeros((D, E), np.float64)
    w_r[:, 1] = col
    w_r = gen.store(w_r, "bf16")
    proj = x64 @ gen.to_f64(w_r, "bf16")[:, 1]
    xs = np.where((proj < 0)[:, None], -x64, x64)  # sign flips are exact in bf16
    keep = np.abs(proj) > 0.1
    xs = xs[keep][:T]
    assert xs.shape[0] == T
    xb = gen.store(xs, "bf16")
    w1, v1, w2 = gen.host_expert_weights(shape, 29)
    d = _dims(m, shape)
    want, idx, _ = oracle.layer_tokens(xb, w_r, w1, v1, w2, "bf16", K)
    assert np.all(idx == 1)
    X, WR, W1, V1, W2 = (dev(a, "bf16") for a in (xb, w_r, w1, v1, w2))
    counts, _, _, _ = m.dispatch(d, m.route(d, X, WR)[0])
    assert counts.cpu().numpy()[1] == T
    out = m.layer_forward(d, X, WR, W1, V1, W2)
    assert m.get_last_error() == 0
    assert_parity(to_numpy(out), want, "bf16", f"one expert, {T} slots")


@pytest.mark.parametrize("layout", ["w1_first", "v1_first", "same_tensor"])
def test_prefill_weight_layouts(layout):
    """The prefill up projection reads a tile of W1 and V1 rows as one copy
    over both tensors when V1 lies a whole tensor or more after W1 or before
    it, else as two copies (here: W1 and V1 the same tensor)."""
    m = moe()
    D, F, E, K, T = 136, 200, 2, 2, 160
    L = _host((D, F, E, K, T, "bf16"), seed=31)
    sh = L.shape
    d = _dims(m, sh)
    v1_host = L.w1 if layout == "same_tensor" else L.v1
    want, idx, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, v1_host, L.w2, "bf16", K)
    x, w_r, w1, v1, w2 = _devlayer(L)
    if layout == "v1_first":
        both = torch.empty((2,) + tuple(w1.shape), dtype=w1.dtype, device=w1.device)
        both[0].copy_(v1)
        both[1].copy_(w1)
        v1, w1 = both[0], both[1]
    elif layout == "w1_first":
        both = torch.stack([w1, v1])
        w1, v1 = both[0], both[1]
    else:
        v1 = w1
    out = m.layer_forward(d, x, w_r, w1, v1, w2)
    assert m.get_last_error() == 0
    assert_parity(to_numpy(out), want, "bf16", f"prefill, {layout}")


@pytest.mark.parametrize("E,K", [(2, 1), (4, 4), (5, 3), (8, 2), (16, 4), (16, 16), (17, 4)])
def test_one_token_layer(E, K):
    """One token: the fused routing kernel and the two streaming kernels,
    over expert counts and top-k widths (K = 1, K = E, E not a multiple of
    8)."""
    m = moe()
    L = _host((136, 200, E, K, 1, "bf16"), seed=37)
    sh = L.shape
    d = _dims(m, sh)
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, "bf16", K)
    x, w_r, w1, v1, w2 = _devlayer(L)
    m.layer_forward(d, x, w_r, w1, v1, w2)
    torch.cuda.synchronize()
    n0 = m.launch_count()
    out = m.layer_forward(d, x, w_r, w1, v1, w2)
    torch.cuda.synchronize()
    assert m.launch_count() - n0 == 3
    assert m.get_last_error() == 0
    assert_parity(to_numpy(out), want, "bf16", f"one token, E={E}, K={K}")


@pytest.mark.parametrize("T", [1, 3, 70, 600])
def test_nan_token_stays_contained(T):
    """A token whose row is NaN (its logits are NaN) is routed to valid
    experts, raises no device error and spoils only its own output row: the
    other tokens match the oracle (one-token, cluster, large-batch and
    prefill paths)."""
    m = moe()
    D, F, E, K = 136, 200, 8, 2
    L = _host((D, F, E, K, T, "bf16"), seed=41)
    sh = L.shape
    d = _dims(m, sh)
    x = gen.to_f64(L.x, "bf16").copy()
    bad = T // 2
    x[bad, :] = np.nan
    xb = gen.store(x, "bf16")
    X, WR, W1, V1, W2 = (dev(a, "bf16") for a in (xb, L.w_r, L.w1, L.v1, L.w2))
    idx, _, _ = m.route(d, X, WR)
    ii = idx.cpu().numpy()
    assert ii.min() >= 0 and ii.max() < E
    assert all(len(set(r)) == K for r in ii.tolist())
    out = to_numpy(m.layer_forward(d, X, WR, W1, V1, W2))
    assert m.get_last_error() == 0
    assert not np.isfinite(out[bad]).any()
    others = np.array([t for t in range(T) if t != bad], dtype=np.int32)
    if others.size:
        want, _, _ = oracle.layer_tokens(xb, L.w_r, L.w1, L.v1, L.w2, "bf16", K, tokens=others)
        assert_parity(out[others], want, "bf16", f"tokens beside a NaN token, T={T}")


@pytest.mark.parametrize("case", [(200, 264, 3, 2, 400), (136, 200, 2, 1, 513)],
                         ids=lambda c: "D{}F{}E{}K{}T{}".format(*c))
def test_prefill_single_cta_form(case, monkeypatch):
    """The prefill GEMMs' one-CTA-per-tile form (MOE_WM_SINGLE_CTA=1) against
    the oracle and against the CTA-pair form."""
    m = moe()
    D, F, E, K, T = case
    L = _host((D, F, E, K, T, "bf16"), seed=43)
    d = _dims(m, L.shape)
    x, w_r, w1, v1, w2 = _devlayer(L)
    pair = to_numpy(m.layer_forward(d, x, w_r, w1, v1, w2))
    monkeypatch.setenv("MOE_WM_SINGLE_CTA", "1")
    single = to_numpy(m.layer_forward(d, x, w_r, w1, v1, w2))
    monkeypatch.delenv("MOE_WM_SINGLE_CTA")
    assert m.get_last_error() == 0
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, "bf16", K)
    assert_parity(single, want, "bf16", "single-CTA prefill GEMMs")
    assert_parity(single, pair, "bf16", "single-CTA vs CTA-pair prefill GEMMs")


def test_empty_batch_is_a_no_op():
    m = moe()
    d = m.dims(64, 64, 4, 2)
    x = torch.zeros((0, 64), dtype=torch.bfloat16, device="cuda")
    w = torch.zeros((64, 4), dtype=torch.bfloat16, device="cuda")
    idx, gate, _ = m.route(d, x, w)
    assert idx.shape == (0, 2)
    counts, offsets, perm, inv = m.dispatch(d, idx)
    assert counts.cpu().tolist() == [0, 0, 0, 0]
    assert offsets.cpu().tolist() == [0, 0, 0, 0, 0]
    w1 = torch.zeros((4, 64, 64), dtype=torch.bfloat16, device="cuda")
    out = m.layer_forward(d, x, w, w1, w1, w1)
    assert out.shape == (0, 64)
    assert m.get_last_error() == 0


def test_dispatch_reports_bad_index():
    m = moe()
    d = m.dims(64, 64, 4, 2)
    idx = torch.tensor([[0, 1], [2, 9]], dtype=torch.int32, device="cuda")
    m.dispatch(d, idx)
    assert m.get_last_error() == 6  # MOE_ERR_DEVICE_INDEX
    assert m.get_last_error() == 0  # cleared by the read


def test_bad_arguments_with_real_tensors():
    m = moe()
    d = m.dims(64, 64, 4, 2)
    x = torch.zeros((4, 64), dtype=torch.bfloat16, device="cuda")
    w = torch.zeros((64, 4), dtype=torch.bfloat16, device="cuda")
    w1 = torch.zeros((4, 64, 64), dtype=torch.bfloat16, device="cuda")
    small = torch.empty(16, dtype=torch.uint8, device="cuda")
    with pytest.raises(m.MoeError) as ei:
        m.layer_forward(d, x, w, w1, w1, w1, ws=small)
    assert ei.value.status == 3
    xm = torch.zeros(4 * 64 + 1, dtype=torch.bfloat16, device="cuda")[1:].view(4, 64)
    with pytest.raises(m.MoeError) as ei:
        m.layer_forward(d, xm, w, w1, w1, w1)
    assert ei.value.status == 1
    bad = m.dims(64, 64, 4, 5)
    with pytest.raises(m.MoeError):
        m.route(bad, x, w)


@pytest.mark.parametrize("T,kernels", [
    (1, {"route_dispatch_small", "up_glu_stream", "down_combine_stream"}),
    (3, {"route_dispatch_cluster", "gather_rows", "gemm_up_glu_tc", "gemm_down_tc", "combine"}),
    (64, {"route_dispatch_cluster", "gather_rows", "gemm_up_glu_tc", "gemm_down_tc", "combine"}),
    (70, {"route", "dispatch", "gather_rows", "gemm_up_glu_tc", "gemm_down_tc", "combine"}),
])
def test_launch_count_and_profile(T, kernels):
    """One token: fused routing + the two streaming kernels; 2..64 tokens: the
    cluster routing kernel and the tensor-core path; more: separate routing
    and dispatch.  Every launch is counted and event-timed."""
    m = moe()
    L = _host((64, 64, 4, 2, T, "bf16"))
    d = _dims(m, L.shape)
    x, w_r, w1, v1, w2 = _devlayer(L)
    m.layer_forward(d, x, w_r, w1, v1, w2)
    torch.cuda.synchronize()
    n0 = m.launch_count()
    m.profile_reset()
    m.profile_enable(True)
    m.layer_forward(d, x, w_r, w1, v1, w2)
    m.profile_enable(False)
    stats = {k: v for k, v in m.profile_read().items() if v[0] > 0}
    assert m.launch_count() - n0 == sum(v[0] for v in stats.values()) == len(kernels)
    assert set(stats) == kernels
    assert all(v[1] > 0 for v in stats.values())


@pytest.mark.parametrize("case", [(64, 96, 8, 2, 1), (128, 136, 16, 4, 9), (72, 40, 5, 3, 33)],
                         ids=lambda c: "D{}F{}E{}K{}T{}".format(*c))
def test_busy_full_loading_equals_sparse(case):
    """Sec. 4.2 busy full loading (all experts, unselected gates zero) gives
    the same layer as the sparse path: against the oracle's busy-full-loading
    route and against the sparse CUDA path."""
    m = moe()
    D, F, E, K, T = case
    L = _host((D, F, E, K, T, "bf16"), seed=19)
    d = _dims(m, L.shape)
    want = oracle.layer_dense_masked(L.x, L.w_r, L.w1, L.v1, L.w2, "bf16", K)
    x, w_r, w1, v1, w2 = _devlayer(L)
    dense = m.layer_forward_dense(d, x, w_r, w1, v1, w2)
    assert m.get_last_error() == 0
    assert_parity(to_numpy(dense), want, "bf16", "busy full loading vs oracle")
    sparse = m.layer_forward(d, x, w_r, w1, v1, w2)
    assert_parity(to_numpy(dense), to_numpy(sparse), "bf16", "busy full loading vs sparse")


@pytest.mark.parametrize("case", [
    (16384, 256, 4, 2, 1, "bf16"),     # wide token rows: too wide for the streaming kernels
    (256, 16384, 4, 2, 3, "bf16"),     # wide hidden layer
    (128, 192, 8, 2, 2048, "bf16"),    # many slot tiles per expert
    (256, 512, 4, 2, 1, "f32"),        # one token on the fp32 path
], ids=lambda c: "D{}F{}E{}K{}T{}{}".format(*c))
def test_size_extremes(case):
    m = moe()
    D, F, E, K, T, dt = case
    L = _host(case, seed=23)
    sh = L.shape
    d = _dims(m, sh)
    x, w_r, w1, v1, w2 = _devlayer(L)
    out = m.layer_forward(d, x, w_r, w1, v1, w2)
    assert m.get_last_error() == 0
    toks = np.unique(np.linspace(0, T - 1, min(T, 24)).astype(np.int32))
    want, idx, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, dt, K, tokens=toks)
    gi, _, _ = m.route(d, x, w_r)
    assert np.array_equal(gi.cpu().numpy()[toks], idx)
    assert_parity(to_numpy(out)[toks], want, dt, f"extremes {case}")
