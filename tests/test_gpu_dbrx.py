"""DBRX-shaped layer (D=6144, F=10752, E=16, K=4, bf16; Table 1 and Sec. 2.1)
at full size, in the launch configuration the benchmark times.

Routing (indices, counts, offsets, permutations) is compared bit-exactly on
every token; layer outputs are compared on sampled tokens, whose fp64 oracle
rows are computed one by one from the same bytes copied back to the host."""
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
    ws = moe.alloc_workspace(d, 2048)
    yield dict(moe=moe, d=d, dev=(w1, v1, w2), host=host, ws=ws, shape=sh)
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

    # the fused layer, sampled rows
    out = m.layer_forward(d, X, WR, w1, v1, w2, ws=layer["ws"])
    assert m.get_last_error() == 0
    rng = np.random.default_rng(seed)
    toks = np.unique(np.concatenate([[0, T - 1], rng.integers(0, T, size=n_sample)]))
    want, _, _ = oracle.layer_tokens(x, w_r, h1, hv, h2, "bf16", sh.top_k, tokens=toks)
    got = to_numpy(out)[toks]
    return assert_parity(got, want, "bf16", f"T={T} skew={skew}")


def test_decode_one_token(layer):
    """One DBRX-shaped layer, decode of a single token."""
    _check(layer, 1, None, 0, 101)


@pytest.mark.parametrize("T", [1, 2, 4, 8, 16, 32, 64])
@pytest.mark.parametrize("skew", [0.0, 0.6, 1.2])
def test_decode_sweep(layer, T, skew):
    """Decode batch sweep with designed routing from uniform to Zipf(1.2)."""
    _check(layer, T, skew, 3, 200 + T)


def test_prefill_2048(layer):
    """2048-token prefill with uniform-random routing."""
    _check(layer, 2048, None, 6, 303)
