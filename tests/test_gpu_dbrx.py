"""DBRX-shaped layer (D=6144, F=10752, E=16, K=4, bf16; Table 1 and Sec. 2.1)
at full size, in the launch configuration the benchmark times.

Routing (indices, counts, offsets, permutations) is compared bit-exactly on
every token.  Layer outputs are compared on every token of every decode
batch (1..64 tokens) and, in the 2048-token prefill, on a stratified sample
of at least 256 tokens that holds, for every expert, the tokens of the first
and last slot of every slot run the CTA-pair GEMMs cut the expert into (so
every run boundary and every expert's ragged tail is checked) and of every
128-slot tile, plus seeded random tokens.  The fp64 oracle rows are computed
one by one from the same bytes copied back to the host."""
import numpy as np
import pytest
import torch

import oracle
from paper_2506_23635_gb300 import inputs as gen
from tests.gpu_util import assert_parity, dev, need_gpu, to_numpy

pytestmark = pytest.mark.gpu

SEED = 2025


@pytest.fixture(scope="module")
def layer():
    need_gpu()
    from paper_2506_23635_gb300 import moe
    sh = gen.DBRX
    w1, v1, w2 = gen.device_expert_weights(sh, SEED, "cuda")
    host = [gen.torch_to_host(t, "bf16") for t in (w1, v1, w2)]
    d = moe.dims(sh.d_model, sh.ffn_hidden, sh.n_experts, sh.top_k)
    d32 = moe.dims(sh.d_model, sh.ffn_hidden, sh.n_experts, sh.top_k, torch.bfloat16,
                   torch.bfloat16, torch.float32)
    ws = moe.alloc_workspace(d, 2048)
    yield dict(moe=moe, d=d, d32=d32, dev=(w1, v1, w2), host=host, ws=ws, shape=sh)
    del w1, v1, w2
    torch.cuda.empty_cache()


def _check(layer, T, skew, n_sample, seed):
    m, d, sh = layer["moe"], layer["d"], layer["shape"]
    w1, v1, w2 = layer["dev"]
    h1, hv, h2 = layer["host"]
    x, w_r = gen.host_router_and_tokens(sh, T, seed, skew)
    X, WR = dev(x, "bf16"), dev(w_r, "bf16")

    # routing on every token, bit-exact
    lg = oracle.router_logits(x, w_r, "bf16")
    ref_idx, ref_gate = oracle.topk_gates(lg, sh.top_k)
    idx, gate, _ = m.route(d, X, WR)
    assert np.array_equal(idx.cpu().numpy(), ref_idx), "top-k indices"
    np.testing.assert_allclose(to_numpy(gate), ref_gate, rtol=0, atol=2e-6)
    counts, offsets, perm, inv = m.dispatch(d, idx)
    rc, ro, rp, ri = oracle.dispatch(ref_idx, sh.n_experts)
    assert np.array_equal(counts.cpu().numpy(), rc)
    assert np.array_equal(offsets.cpu().numpy(), ro)
    assert np.array_equal(perm.cpu().numpy(), rp)
    assert np.array_equal(inv.cpu().numpy(), ri)

    # the fused layer: every token, or the stratified sample.  Written in
    # fp32, the output meets the layer bound; written in bf16 (the
    # benchmarked form), each element also carries its one storage rounding
    # (reading C24)
    toks = np.arange(T) if n_sample is None else _stratified_tokens(rp, ro, sh.top_k, T,
                                                                    n_sample, seed)
    want, _, _ = oracle.layer_tokens(x, w_r, h1, hv, h2, "bf16", sh.top_k, tokens=toks)
    out32 = m.layer_forward(layer["d32"], X, WR, w1, v1, w2, ws=layer["ws"])
    out = m.layer_forward(d, X, WR, w1, v1, w2, ws=layer["ws"])
    assert m.get_last_error() == 0
    what = f"T={T} skew={skew} ({toks.size} tokens)"
    r = assert_parity(to_numpy(out32)[toks], want, "bf16", what + ", fp32 out")
    assert_parity(to_numpy(out)[toks], want, "bf16", what + ", bf16 out", stored_bf16=True)
    return r


RUN_MAX = 256   # slots per run of the CTA-pair GEMMs (the MMA's largest N)
SLOT_TILE = 128  # slots per tile of the single-CTA GEMMs


def _stratified_tokens(perm, offsets, K, T, n_min, seed):
    """Token 0, token T-1, and for every expert the tokens holding the first
    and last sorted slot of each slot run (an expert of n_e slots is cut into
    ceil(n_e / 256) runs [floor(i n_e / r), floor((i+1) n_e / r))) and of
    each 128-slot tile; then seeded random tokens up to n_min."""
    pick = {0, T - 1}
    for e in range(offsets.size - 1):
        lo, n_e = int(offsets[e]), int(offsets[e + 1] - offsets[e])
        if n_e == 0:
            continue
        r = -(-n_e // RUN_MAX)
        for i in range(r):
            a, b = i * n_e // r, (i + 1) * n_e // r
            pick.update((int(perm[lo + a]) // K, int(perm[lo + b - 1]) // K))
        for a in range(0, n_e, SLOT_TILE):
            b = min(n_e, a + SLOT_TILE)
            pick.update((int(perm[lo + a]) // K, int(perm[lo + b - 1]) // K))
    rng = np.random.default_rng(seed)
    while len(pick) < n_min:
        pick.add(int(rng.integers(0, T)))
    return np.array(sorted(pick), np.int32)


def test_decode_one_token(layer):
    """One DBRX-shaped layer, decode of a single token."""
    _check(layer, 1, None, None, 101)


@pytest.mark.parametrize("T", [1, 2, 4, 8, 16, 32, 64])
@pytest.mark.parametrize("skew", [0.0, 0.6, 1.2])
def test_decode_sweep(layer, T, skew):
    """Decode batch sweep with designed routing from uniform to Zipf(1.2);
    every token of the batch."""
    _check(layer, T, skew, None, 200 + T)


def test_prefill_2048(layer):
    """2048-token prefill with uniform-random routing: at least 256 tokens,
    every slot-run boundary of every expert among them."""
    _check(layer, 2048, None, 256, 303)


@pytest.mark.parametrize("T,cuts", [(1, (0, 8, 16)), (8, (0, 4, 8, 12, 16)),
                                    (512, (0, 8, 16))])
def test_expert_parallel_shares(layer, T, cuts):
    """Sec. 4.3: the shares of 2 and 4 nodes (8 or 4 experts each, their
    weights as views of the resident tensors) summed equal the layer: every
    token for decode, 48 tokens of the 512-token batch."""
    m, d, sh = layer["moe"], layer["d"], layer["shape"]
    w1, v1, w2 = layer["dev"]
    h1, hv, h2 = layer["host"]
    x, w_r = gen.host_router_and_tokens(sh, T, 400 + T, None)
    X, WR = dev(x, "bf16"), dev(w_r, "bf16")
    toks = np.arange(T) if T <= 64 else np.unique(np.concatenate(
        [[0, T - 1], np.random.default_rng(T).integers(0, T, size=46)])).astype(np.int32)
    total = np.zeros((toks.size, sh.d_model))
    for b, e in zip(cuts[:-1], cuts[1:]):
        part = m.layer_forward_experts(d, X, WR, b, e, w1[b:e], v1[b:e], w2[b:e],
                                       ws=layer["ws"])
        assert m.get_last_error() == 0
        got = to_numpy(part)[toks]
        ref = oracle.layer_experts_tokens(x, w_r, h1, hv, h2, "bf16", sh.top_k, b, e,
                                          tokens=toks)
        assert_parity(got, ref, "bf16", f"T={T} share [{b},{e})")
        total += got
    want, _, _ = oracle.layer_tokens(x, w_r, h1, hv, h2, "bf16", sh.top_k, tokens=toks)
    assert_parity(total, want, "bf16", f"T={T}: sum of {len(cuts) - 1} shares")
