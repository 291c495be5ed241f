"""The self-attention block of a decoder layer and whole decoder layers on
the GPU against the fp64 oracle.

Bars: cache entries the call does not write stay bit-identical; values
within rel L2 5e-3 and max abs 2e-2 * RMS.  Step by step: the rotated
queries and the new cache entries against the oracle's rotary embedding of
the projection (numpy's matmul of the stored bytes), ctx against the
oracle's attention over the GPU's own queries and caches, then the whole
block, and whole decoder layers (attention + MoE) with the routing-gap
filter of the stacked MoE tests."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_23635_gb300 import inputs as gen
from tests.gpu_util import assert_parity, dev, need_gpu, to_numpy

pytestmark = pytest.mark.gpu

EPS = 1e-6
WELL_CONDITIONED = 0.02


def moe():
    need_gpu()
    from paper_2506_23635_gb300 import moe as m
    return m


def _tokens(kind, n_seq, L, rng):
    """(seq, pos) of a call: a decode step (one token per sequence), a
    prefill (consecutive positions of one sequence from 0 or from an offset)
    or a mix of both."""
    if kind == "decode1":
        return np.array([n_seq - 1], np.int32), np.array([L - 1], np.int32)
    if kind == "decode":
        seq = np.arange(n_seq, dtype=np.int32)
        pos = rng.integers(0, L, size=n_seq).astype(np.int32)
        pos[0] = 0
        pos[-1] = L - 1
        return seq, pos
    if kind == "prefill":
        n = min(L, 70)
        return np.zeros(n, np.int32), np.arange(n, dtype=np.int32)
    if kind == "chunk300":  # positions 37..336 of sequence 1: two full 128-token tiles + 44
        return np.ones(300, np.int32), np.arange(37, 337, dtype=np.int32)
    # a chunk of sequence 0 after 10 cached positions, plus decode tokens
    seq = np.concatenate([np.zeros(20, np.int32), np.arange(1, n_seq, dtype=np.int32)])
    pos = np.concatenate([np.arange(10, 30, dtype=np.int32),
                          rng.integers(0, L, size=n_seq - 1).astype(np.int32)])
    return seq, pos


# (D, Hq, Hkv, n_seq, max_len, tokens): groups of 2, 6, 1, 8 and 3 query
# heads per key/value head; one token and batches of up to 128 tokens (the
# tensor-core kernel with the weights as the M operand), beyond 128 the
# grouped tensor-core GEMM (DBRX test below); position splits with ragged
# ends, and a single split.
CASES = [
    (256, 4, 2, 3, 64, "decode1"),
    (256, 4, 2, 6, 300, "decode"),
    (768, 6, 1, 2, 96, "prefill"),
    (512, 4, 4, 5, 200, "mixed"),
    (1024, 8, 1, 4, 2500, "decode"),
    (384, 3, 1, 1, 1100, "decode1"),
    (512, 8, 4, 1, 100, "prefill"),  # one position split per token: ctx written directly
    (256, 4, 2, 2, 400, "chunk300"),  # tensor-core prefill tiles + a CUDA-core tail
]


def _case(case, seed=5):
    D, Hq, Hkv, n_seq, L, kind = case
    shape = gen.AttnShape(D, Hq, Hkv, 128, 10000.0, "bf16")
    rng = np.random.default_rng(seed)
    w_qkv, w_o = gen.host_attn_weights(shape, seed)
    kc, vc = gen.host_kv_cache(shape, n_seq, L, seed)
    seq, pos = _tokens(kind, n_seq, L, rng)
    return shape, w_qkv, w_o, kc, vc, seq, pos


def _ids(c):
    return "D{}Hq{}Hkv{}S{}L{}-{}".format(*c)


def _sa(m, shape):
    return m.sa_dims(shape.d_model, shape.n_heads, shape.n_kv_heads, shape.head_dim,
                     shape.rope_base)


def _written(kc_shape, seq, pos):
    mask = np.zeros(kc_shape[:3], bool)
    mask[seq, :, pos] = True
    return mask


@pytest.mark.parametrize("case", CASES, ids=_ids)
def test_qkv_attend_and_block(case):
    m = moe()
    shape, w_qkv, w_o, kc, vc, seq, pos = _case(case)
    a = _sa(m, shape)
    T, D, Hq, Hkv, dh = len(seq), shape.d_model, shape.n_heads, shape.n_kv_heads, 128
    nq, nkv = Hq * dh, Hkv * dh
    rng = np.random.default_rng(9)
    xn = gen.store(rng.normal(size=(T, D)), "bf16")
    d_seq, d_pos = torch.from_numpy(seq).cuda(), torch.from_numpy(pos).cuda()

    # step 1: projection, rotary embedding, cache writes
    gk, gv = dev(kc, "bf16"), dev(vc, "bf16")
    q = m.sa_qkv(a, dev(xn, "bf16"), dev(w_qkv, "bf16"), d_seq, d_pos, gk, gv)
    assert m.get_last_error() == 0
    proj = gen.to_f64(xn, "bf16") @ gen.to_f64(w_qkv, "bf16").T
    q_ref = oracle.rope(proj[:, :nq].reshape(T, Hq, dh), pos, shape.rope_base)
    k_ref = oracle.round_bf16(oracle.rope(proj[:, nq:nq + nkv].reshape(T, Hkv, dh), pos,
                                          shape.rope_base))
    v_ref = oracle.round_bf16(proj[:, nq + nkv:].reshape(T, Hkv, dh))
    assert_parity(to_numpy(q), q_ref, "bf16", "rotated queries")  # fp32: no storage rounding
    hk, hv = gk.cpu().view(torch.int16).numpy().view(np.uint16), \
        gv.cpu().view(torch.int16).numpy().view(np.uint16)
    keep = ~_written(kc.shape, seq, pos)
    assert np.array_equal(hk[keep], kc[keep]) and np.array_equal(hv[keep], vc[keep]), \
        "cache entries outside the new tokens changed"
    assert_parity(gen.to_f64(hk, "bf16")[seq, :, pos], k_ref, "bf16", "cached keys", True)
    assert_parity(gen.to_f64(hv, "bf16")[seq, :, pos], v_ref, "bf16", "cached values", True)

    # step 2: attention over the GPU's own queries and caches
    ctx = m.sa_attend(a, q, d_seq, d_pos, gk, gv)
    assert m.get_last_error() == 0
    # the attention reads the queries rounded to bf16 (reading C20)
    want = oracle.attention(oracle.round_bf16(to_numpy(q)), gen.to_f64(hk, "bf16"),
                            gen.to_f64(hv, "bf16"), seq, pos)
    assert_parity(to_numpy(ctx), want.reshape(T, nq), "bf16", "attention ctx", True)

    # the whole block on an fp32 residual stream, from the original caches
    x = rng.normal(size=(T, D)).astype(np.float32) * 2.0
    resid = torch.from_numpy(x).cuda()
    gk, gv = dev(kc, "bf16"), dev(vc, "bf16")
    m.sa_forward(a, resid, dev(w_qkv, "bf16"), dev(w_o, "bf16"), d_seq, d_pos, gk, gv, eps=EPS)
    assert m.get_last_error() == 0
    out, wk, wv = oracle.sa_forward(x.astype(np.float64), w_qkv, w_o, "bf16", Hq, Hkv,
                                    shape.rope_base, EPS, seq, pos, gen.to_f64(kc, "bf16"),
                                    gen.to_f64(vc, "bf16"))
    got = to_numpy(resid)
    assert_parity(got - x, out - x, "bf16", "attention block update")
    assert_parity(to_numpy(gk)[seq, :, pos], wk[seq, :, pos], "bf16", "block cached keys", True)


def test_out_of_range_token_is_reported_and_writes_nothing():
    m = moe()
    shape, w_qkv, w_o, kc, vc, _, _ = _case((256, 4, 2, 3, 64, "decode"))
    a = _sa(m, shape)
    seq = torch.tensor([0, 3, 1], dtype=torch.int32, device="cuda")   # sequence 3 does not exist
    pos = torch.tensor([5, 2, 64], dtype=torch.int32, device="cuda")  # position 64 is past the end
    gk, gv = dev(kc, "bf16"), dev(vc, "bf16")
    xn = dev(gen.store(np.ones((3, 256)), "bf16"), "bf16")
    q = m.sa_qkv(a, xn, dev(w_qkv, "bf16"), seq, pos, gk, gv)
    ctx = m.sa_attend(a, q, seq, pos, gk, gv)
    assert m.get_last_error() == 6  # MOE_ERR_DEVICE_INDEX
    assert m.get_last_error() == 0
    hk = gk.cpu().view(torch.int16).numpy().view(np.uint16)
    mask = np.ones(kc.shape[:3], bool)
    mask[0, :, 5] = False
    assert np.array_equal(hk[mask], kc[mask])
    assert torch.all(ctx[1:] == 0)
    assert torch.all(torch.isfinite(ctx[0].float()))


def test_empty_call_and_bad_arguments():
    m = moe()
    a = m.sa_dims(256, 4, 2)
    z = torch.zeros(0, dtype=torch.int32, device="cuda")
    cache = torch.zeros((1, 2, 4, 128), dtype=torch.bfloat16, device="cuda")
    resid = torch.zeros((0, 256), dtype=torch.float32, device="cuda")
    w = torch.zeros((1024, 256), dtype=torch.bfloat16, device="cuda")
    m.sa_forward(a, resid, w, w, z, z, cache, cache)  # T = 0: nothing launched
    with pytest.raises(m.MoeError):  # 4 query heads cannot share 3 key/value heads
        m.sa_forward(m.sa_dims(256, 4, 3), resid, w, w, z, z, cache, cache)
    with pytest.raises(m.MoeError):
        m.sa_forward(m.sa_dims(256, 4, 2, head_dim=64), resid, w, w, z, z, cache, cache)


def _decoder_layers(shape_a, shape_m, n_layers, n_seq, L, seed):
    layers, caches = [], []
    for l in range(n_layers):
        w_qkv, w_o = gen.host_attn_weights(shape_a, seed, l)
        w_r = gen.host_normal((shape_m.d_model, shape_m.n_experts), gen.W_STD, "bf16", seed,
                              "dec-w_r", l)
        w1, v1, w2 = gen.host_expert_weights(shape_m, seed + 100 * (l + 1))
        layers.append((w_qkv, w_o, w_r, w1, v1, w2))
        caches.append(gen.host_kv_cache(shape_a, n_seq, L, seed, l))
    return layers, caches


@pytest.mark.parametrize("kind", ["decode1", "decode", "prefill"])
def test_decoder_layers(kind):
    """Three decoder layers (attention + MoE) on the fp32 residual stream;
    tokens whose routing gap falls under 2% of the logit RMS at some layer
    are ill-conditioned and left out (reading C15), the bound is compounded
    over the layers (reading C14)."""
    m = moe()
    n_layers, n_seq, L = 3, 4, 80
    sa_shape = gen.AttnShape(256, 4, 2, 128, 10000.0, "bf16")
    moe_shape = gen.LayerShape(256, 512, 8, 2, "bf16")
    layers, caches = _decoder_layers(sa_shape, moe_shape, n_layers, n_seq, L, 17)
    rng = np.random.default_rng(3)
    seq, pos = _tokens(kind, n_seq, L, rng)
    T = len(seq)
    x = rng.normal(size=(T, 256)).astype(np.float32)
    want, _, gaps = oracle.decoder_layers(
        x.astype(np.float64), layers, "bf16", 4, 2, sa_shape.rope_base, EPS, 2, seq, pos,
        [(gen.to_f64(k, "bf16"), gen.to_f64(v, "bf16")) for k, v in caches])
    a = _sa(m, sa_shape)
    d = m.dims(256, 512, 8, 2, torch.bfloat16, torch.bfloat16, torch.float32)
    dl = [tuple(dev(t, "bf16") for t in lw) + (dev(k, "bf16"), dev(v, "bf16"))
          for lw, (k, v) in zip(layers, caches)]
    W = m.DecoderWeights(dl)
    resid = torch.from_numpy(x).cuda()
    m.decoder_forward(a, d, W, resid, torch.from_numpy(seq).cuda(), torch.from_numpy(pos).cuda(),
                      eps=EPS)
    assert m.get_last_error() == 0
    got = to_numpy(resid)
    ok = np.all(gaps >= WELL_CONDITIONED, axis=0)
    assert ok.sum() >= max(1, (3 * T) // 4), f"only {ok.sum()} of {T} tokens well conditioned"
    err = got[ok] - want[ok]
    rel = np.linalg.norm(err) / np.linalg.norm(want[ok] - x[ok])
    assert rel <= 5e-3 * np.sqrt(n_layers), f"decoder layers: rel L2 of the update {rel:.3e}"


def test_prefill_ignores_cache_rows_past_the_chunk():
    """Positions 37..336 of sequence 1 (two tensor-core tiles whose last
    key/value tile runs past their last query, and a CUDA-core tail) with NaN
    in every cache row the chunk does not reach: the result equals the
    oracle's, which reads only positions up to each token's own."""
    m = moe()
    shape, w_qkv, w_o, kc, vc, seq, pos = _case((256, 4, 2, 2, 400, "chunk300"), seed=13)
    nan = gen.store(np.full(1, np.nan), "bf16")[0]
    kc = kc.copy()
    vc = vc.copy()
    kc[1, :, 337:, :] = nan
    vc[1, :, 337:, :] = nan
    T = seq.size
    x = np.random.default_rng(17).normal(size=(T, shape.d_model)).astype(np.float32)
    want, _, _ = oracle.sa_forward(x.astype(np.float64), w_qkv, w_o, "bf16", shape.n_heads,
                                   shape.n_kv_heads, shape.rope_base, EPS, seq, pos,
                                   gen.to_f64(kc, "bf16"), gen.to_f64(vc, "bf16"))
    resid = torch.from_numpy(x).cuda()
    m.sa_forward(_sa(m, shape), resid, dev(w_qkv, "bf16"), dev(w_o, "bf16"),
                 torch.from_numpy(seq).cuda(), torch.from_numpy(pos).cuda(), dev(kc, "bf16"),
                 dev(vc, "bf16"), eps=EPS)
    assert m.get_last_error() == 0
    got = to_numpy(resid)
    assert np.isfinite(got).all()
    assert_parity(got - x, want - x, "bf16", "prefill chunk beside NaN cache rows")


@pytest.mark.parametrize("T,ctx_len", [(1, 2048), (8, 2048), (256, 256), (2048, 2048)])
def test_dbrx_attention_block(T, ctx_len):
    """DBRX's attention dims (D = 6144, 48 query and 8 key/value heads of
    128, D_qkv = 8,192): decode steps of 1 and 8 sequences at context 2048,
    a 256-token prefill and the benchmarked 2048-token prefill (sixteen
    128-token tiles of the tensor-core flash attention), the whole block
    against the oracle on every token."""
    m = moe()
    shape = gen.DBRX_ATTN
    n_seq = max(T, 1) if T <= 8 else 1
    L = ctx_len
    w_qkv, w_o = gen.host_attn_weights(shape, 29)
    kc, vc = gen.host_kv_cache(shape, n_seq, L, 29)
    if T <= 8:
        seq = np.arange(T, dtype=np.int32)
        pos = np.full(T, L - 1, np.int32)
    else:
        seq = np.zeros(T, np.int32)
        pos = np.arange(T, dtype=np.int32)
    x = np.random.default_rng(31).normal(size=(T, shape.d_model)).astype(np.float32)
    want, _, _ = oracle.sa_forward(x.astype(np.float64), w_qkv, w_o, "bf16", 48, 8,
                                   shape.rope_base, EPS, seq, pos, gen.to_f64(kc, "bf16"),
                                   gen.to_f64(vc, "bf16"))
    a = _sa(m, shape)
    resid = torch.from_numpy(x).cuda()
    m.sa_forward(a, resid, dev(w_qkv, "bf16"), dev(w_o, "bf16"), torch.from_numpy(seq).cuda(),
                 torch.from_numpy(pos).cuda(), dev(kc, "bf16"), dev(vc, "bf16"), eps=EPS)
    assert m.get_last_error() == 0
    assert_parity(to_numpy(resid) - x, want - x, "bf16", f"DBRX attention block T={T}")


def _plateau_case(levels, T, L=600, seed=41):
    """Queries u (one bf16-exact unit vector for every token and head) and
    keys c(pos) * u * sqrt(128) / log2(e) plus N(0,1) noise, so the scaled
    score of position pos is c(pos) in base-2 units (+ ~0.13 noise): the
    running row maximum steps as `levels` says.  Sequence 1, positions
    0..T-1; values N(0,1)."""
    rng = np.random.default_rng(seed)
    Hq, Hkv, dh = 4, 2, 128
    u = rng.normal(size=dh)
    u = gen.to_f64(gen.store(u / np.linalg.norm(u), "bf16"), "bf16")
    q = np.tile(u, (T, Hq)).astype(np.float32)
    c = np.zeros(L)
    for lo, hi, lv in levels:
        c[lo:hi] = lv
    k = np.empty((2, Hkv, L, dh))
    k[:] = rng.normal(size=(2, Hkv, L, dh))
    k[1] += (c[:, None] * u[None, :] * np.sqrt(dh) / np.log2(np.e))[None]
    kc = gen.store(k, "bf16")
    vc = gen.store(rng.normal(size=(2, Hkv, L, dh)), "bf16")
    seq = np.ones(T, np.int32)
    pos = np.arange(T, dtype=np.int32)
    return gen.AttnShape(512, Hq, Hkv, dh, 10000.0, "bf16"), q, kc, vc, seq, pos


# (levels as (first, end, base-2 score), tokens): the exponent base moves in
# the first tile, stays while the maximum rises by 4.5 (probabilities up to
# 2^4.5), moves by 9 in the third tile and again inside the diagonal tile of
# the fourth, then the scores drop by 20; a ragged CUDA-core tail after four
# tensor-core tiles.  Then a maximum of 40 in the first tile that nothing
# later approaches (every later probability ~2^-40).
PLATEAUS = [
    ([(100, 230, 8.5), (230, 300, 13.0), (300, 420, 22.0), (420, 470, 31.0),
      (470, 600, 11.0)], 571),
    ([(0, 12, 40.0)], 512),
]


@pytest.mark.parametrize("levels,T", PLATEAUS, ids=["rising", "first-tile-max"])
def test_prefill_running_max_rescales(levels, T):
    """The prefill tensor-core attention keeps the exponent base of a row
    until the row maximum passes it by more than 8 (base 2) and then
    rescales the output accumulated in tensor memory: scores built to step
    across that threshold (and below it) give the oracle's attention."""
    m = moe()
    shape, q, kc, vc, seq, pos = _plateau_case(levels, T)
    a = _sa(m, shape)
    m.profile_reset()
    m.profile_enable(True)
    ctx = m.sa_attend(a, torch.from_numpy(q).cuda(), torch.from_numpy(seq).cuda(),
                      torch.from_numpy(pos).cuda(), dev(kc, "bf16"), dev(vc, "bf16"))
    assert m.get_last_error() == 0
    m.profile_enable(False)
    assert m.profile_read().get("attention_tc", (0,))[0] == 1, "tensor-core attention did not run"
    want = oracle.attention(q.reshape(T, shape.n_heads, 128).astype(np.float64),
                            gen.to_f64(kc, "bf16"), gen.to_f64(vc, "bf16"), seq, pos)
    assert_parity(to_numpy(ctx), want.reshape(T, -1), "bf16", "attention across rescales", True)


@pytest.mark.parametrize("Hq,Hkv", [(5, 5), (6, 2), (5, 1), (8, 1), (4, 2)],
                         ids=["G1", "G3", "G5", "G8", "G2"])
def test_prefill_head_groups(Hq, Hkv):
    """The tensor-core prefill attention pairs the query heads of a
    key/value head two to a CTA; with 1, 3 or 5 heads per group the last head
    of each group is alone in its CTA.  Two full 128-token tiles at positions
    7..262 of sequence 0 and a 3-token tail, random queries and caches,
    against the oracle (and the kernel must have run)."""
    m = moe()
    rng = np.random.default_rng(50 + Hq * 8 + Hkv)
    dh, L, T = 128, 300, 259
    q = rng.normal(size=(T, Hq * dh)).astype(np.float32)
    q = gen.to_f64(gen.store(q, "bf16"), "bf16").astype(np.float32)  # bf16-exact
    kc = gen.store(rng.normal(size=(1, Hkv, L, dh)), "bf16")
    vc = gen.store(rng.normal(size=(1, Hkv, L, dh)), "bf16")
    seq = np.zeros(T, np.int32)
    pos = np.arange(7, 7 + T, dtype=np.int32)
    a = _sa(m, gen.AttnShape(512, Hq, Hkv, dh, 10000.0, "bf16"))
    m.profile_reset()
    m.profile_enable(True)
    ctx = m.sa_attend(a, torch.from_numpy(q).cuda(), torch.from_numpy(seq).cuda(),
                      torch.from_numpy(pos).cuda(), dev(kc, "bf16"), dev(vc, "bf16"))
    assert m.get_last_error() == 0
    m.profile_enable(False)
    assert m.profile_read().get("attention_tc", (0,))[0] == 1, "tensor-core attention did not run"
    want = oracle.attention(q.reshape(T, Hq, dh).astype(np.float64), gen.to_f64(kc, "bf16"),
                            gen.to_f64(vc, "bf16"), seq, pos)
    assert_parity(to_numpy(ctx), want.reshape(T, -1), "bf16", f"prefill Hq={Hq} Hkv={Hkv}", True)


def _decode_path_child():
    """(run in a child process) A DBRX decode step, 8 sequences at context
    2048, through moe_sa_forward: which attention kernel ran, and the block
    against the oracle."""
    import os
    m = moe()
    shape = gen.DBRX_ATTN
    T, L = 8, 2048
    w_qkv, w_o = gen.host_attn_weights(shape, 37)
    kc, vc = gen.host_kv_cache(shape, T, L, 37)
    seq = np.arange(T, dtype=np.int32)
    pos = np.full(T, L - 1, np.int32)
    pos[0] = 700  # a shorter context: a partial last tile, an empty split
    x = np.random.default_rng(41).normal(size=(T, shape.d_model)).astype(np.float32)
    want, _, _ = oracle.sa_forward(x.astype(np.float64), w_qkv, w_o, "bf16", 48, 8,
                                   shape.rope_base, EPS, seq, pos, gen.to_f64(kc, "bf16"),
                                   gen.to_f64(vc, "bf16"))
    resid = torch.from_numpy(x).cuda()
    m.profile_reset()
    m.profile_enable(True)
    m.sa_forward(_sa(m, shape), resid, dev(w_qkv, "bf16"), dev(w_o, "bf16"),
                 torch.from_numpy(seq).cuda(), torch.from_numpy(pos).cuda(), dev(kc, "bf16"),
                 dev(vc, "bf16"), eps=EPS)
    assert m.get_last_error() == 0
    m.profile_enable(False)
    ran = {k for k, v in m.profile_read().items() if v[0] > 0}
    expect = "attention" if os.environ.get("MOE_ATTN_CUDA_CORES") == "1" else "attention_decode_tc"
    assert expect in ran, f"{expect} did not run: {sorted(ran)}"
    assert_parity(to_numpy(resid) - x, want - x, "bf16", f"decode block on {expect}")
    print("decode path ok:", expect)


@pytest.mark.parametrize("cuda_cores", [False, True], ids=["tensor_cores", "cuda_cores"])
def test_dbrx_decode_on_both_attention_kernels(cuda_cores):
    """Decode steps attend on the tensor-core decode kernel by default and on
    the CUDA-core kernel with MOE_ATTN_CUDA_CORES=1; both meet the block
    bound (a fresh process each: the switch is read once)."""
    need_gpu()
    import os
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ)
    env.pop("MOE_ATTN_CUDA_CORES", None)
    if cuda_cores:
        env["MOE_ATTN_CUDA_CORES"] = "1"
    p = subprocess.run([sys.executable, "-c",
                        "import tests.test_gpu_attention as t; t._decode_path_child()"],
                       cwd=root, env=env, capture_output=True, text=True, timeout=600)
    assert p.returncode == 0, (p.stdout + p.stderr)[-3000:]
    assert "decode path ok" in p.stdout


# (Hq, Hkv, sequences = decode tokens, max_len): the tensor-core decode
# kernel's position tiles shared between the splits of one (token, key/value
# head): one split that takes all its tiles after the first three (192 pairs),
# three splits over up to 20 tiles (50 pairs), eight splits over up to 40
# tiles (2 pairs), and short sequences whose splits have fewer than three
# tiles or none; positions random, with 0 and max_len - 1 present.
SHARED_TILES = [(16, 8, 24, 1000), (6, 1, 50, 2500), (8, 1, 2, 5000), (6, 2, 9, 300)]


@pytest.mark.parametrize("Hq,Hkv,n_seq,L", SHARED_TILES,
                         ids=["one-split", "three-splits", "eight-splits", "short"])
def test_decode_splits_share_position_tiles(Hq, Hkv, n_seq, L):
    m = moe()
    rng = np.random.default_rng(11)
    shape = gen.AttnShape(Hq * 128, Hq, Hkv, 128, 10000.0, "bf16")
    kc, vc = gen.host_kv_cache(shape, n_seq, L, 11)
    seq = np.arange(n_seq, dtype=np.int32)
    pos = rng.integers(0, L, size=n_seq).astype(np.int32)
    pos[0], pos[-1] = 0, L - 1
    q = rng.normal(size=(n_seq, Hq, 128)).astype(np.float32)
    a = m.sa_dims(shape.d_model, Hq, Hkv, 128, shape.rope_base)
    m.profile_enable(True)
    m.profile_reset()
    ctx = m.sa_attend(a, torch.from_numpy(q).cuda(), torch.from_numpy(seq).cuda(),
                      torch.from_numpy(pos).cuda(), dev(kc, "bf16"), dev(vc, "bf16"))
    torch.cuda.synchronize()
    ran = {k for k, v in m.profile_read().items() if v[0] > 0}
    m.profile_enable(False)
    assert m.get_last_error() == 0
    assert "attention_decode_tc" in ran, sorted(ran)
    want = oracle.attention(oracle.round_bf16(q.astype(np.float64)), gen.to_f64(kc, "bf16"),
                            gen.to_f64(vc, "bf16"), seq, pos)
    assert_parity(to_numpy(ctx), want.reshape(n_seq, Hq * 128), "bf16", "attention ctx", True)


def _random_decode_configs(n=12, seed=2024):
    """Seeded decode calls over the tensor-core kernel's launch shapes: head
    groups of 1-8, one to eight position splits per (token, key/value head)
    (SMs / pairs, at most the cache's tiles), caches of 1-40 tiles with
    ragged ends, and tokens at random positions (some at 0, some at the last
    cache row)."""
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n):
        G = int(rng.integers(1, 9))
        Hkv = int(rng.choice([1, 2, 4, 8]))
        n_seq = int(rng.integers(1, 25))
        L = int(rng.integers(1, 5121))
        n_seq = max(1, min(n_seq, 120_000 // (Hkv * L)))  # caches of at most ~30 MB
        out.append((G * Hkv, Hkv, n_seq, L, int(rng.integers(0, 1 << 30))))
    return out


@pytest.mark.parametrize("Hq,Hkv,n_seq,L,s", _random_decode_configs())
def test_decode_random_launch_shapes(Hq, Hkv, n_seq, L, s):
    m = moe()
    rng = np.random.default_rng(s)
    shape = gen.AttnShape(Hq * 128, Hq, Hkv, 128, 10000.0, "bf16")
    kc, vc = gen.host_kv_cache(shape, n_seq, L, s % 1000)
    seq = rng.permutation(n_seq).astype(np.int32)
    pos = rng.integers(0, L, size=n_seq).astype(np.int32)
    pos[rng.random(n_seq) < 0.15] = 0
    pos[rng.random(n_seq) < 0.15] = L - 1
    q = rng.normal(size=(n_seq, Hq, 128)).astype(np.float32)
    a = m.sa_dims(shape.d_model, Hq, Hkv, 128, shape.rope_base)
    ctx = m.sa_attend(a, torch.from_numpy(q).cuda(), torch.from_numpy(seq).cuda(),
                      torch.from_numpy(pos).cuda(), dev(kc, "bf16"), dev(vc, "bf16"))
    torch.cuda.synchronize()
    assert m.get_last_error() == 0
    want = oracle.attention(oracle.round_bf16(q.astype(np.float64)), gen.to_f64(kc, "bf16"),
                            gen.to_f64(vc, "bf16"), seq, pos)
    assert_parity(to_numpy(ctx), want.reshape(n_seq, Hq * 128), "bf16", "attention ctx", True)
