"""One node's share of the expert-parallel layer (Sec. 4.3, Fig. 7) through
the C ABI (moe_layer_forward_experts) against the fp64 oracle.

Every share routes over all experts and computes only its own; each share
is compared with the oracle's share of the same range, and the shares of a
partition of [0, E), summed (the all-reduce), with the oracle's whole
layer.  Cases cover every kernel path of the share: one token (the
row-streaming kernels), decode batches (the 128-slot-tile tensor-core GEMMs,
stream-K tails), a prefill batch (the CTA-pair GEMMs), fp32 weights (the
CUDA-core kernels, fused and unfused combine), and a residual given to one
share.  A two-process gloo group on the one GPU runs the product's
expert_parallel.layer_forward, all-reducing the shares through the host."""
import os
import socket
import sys

import numpy as np
import pytest
import torch

import oracle
from paper_2506_23635_gb300 import inputs as gen
from tests.gpu_util import assert_parity, dev, h_rounding_allowance, need_gpu, to_numpy

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def moe():
    need_gpu()
    from paper_2506_23635_gb300 import moe as m
    return m


def _dims(m, sh):
    tdt = gen.torch_dtype(sh.dtype)
    return m.dims(sh.d_model, sh.ffn_hidden, sh.n_experts, sh.top_k, tdt, tdt, tdt)


# (D, F, E, K, T, dtype, partition of [0, E))
CASES = [
    (512, 1024, 8, 2, 1, "bf16", (0, 4, 8)),
    (512, 1024, 8, 2, 1, "bf16", (0, 1, 3, 6, 8)),
    (264, 520, 16, 4, 24, "bf16", (0, 8, 16)),
    (264, 520, 16, 4, 64, "bf16", (0, 5, 6, 16)),
    (4096, 256, 16, 4, 16, "bf16", (0, 4, 8, 12, 16)),  # stream-K heads and tails
    (200, 264, 8, 2, 600, "bf16", (0, 3, 8)),            # CTA-pair GEMMs, ragged runs
    (256, 512, 4, 2, 8, "f32", (0, 2, 4)),               # CUDA-core GEMV, fused combine
    (72, 40, 5, 3, 70, "f32", (0, 1, 5)),                # unfused combine
]


@pytest.mark.parametrize("case", CASES, ids=lambda c: "D{}F{}E{}K{}T{}{}-{}".format(
    *c[:6], "-".join(map(str, c[6]))))
def test_shares_sum_to_the_layer(case):
    m = moe()
    D, F, E, K, T, dt, cuts = case
    sh = gen.LayerShape(D, F, E, K, dt)
    L = gen.host_layer(sh, T, 17)
    d = _dims(m, sh)
    x, w_r, w1, v1, w2 = [dev(a, dt) for a in (L.x, L.w_r, L.w1, L.v1, L.w2)]
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, dt, K)
    # bf16: each slot's expert output carries the GLU hidden vector's bf16
    # storage (reading C7); its worst case, gated, is each element's
    # allowance in a share (fp32 output: no storage rounding of its own)
    slot_allow = None
    if dt == "bf16":
        st = oracle.layer_steps(L.x, L.w_r, L.w1, L.v1, L.w2, dt, K)
        y_allow = h_rounding_allowance(st["h_sorted"], gen.to_f64(L.w2, dt), st["offsets"])
        slots = st["inv_perm"].reshape(T, K)
        slot_allow = [(st["idx"][:, k], st["gate"][:, k, None] * y_allow[slots[:, k]])
                      for k in range(K)]
    total = np.zeros((T, D))
    for b, e in zip(cuts[:-1], cuts[1:]):
        part = m.layer_forward_experts(d, x, w_r, b, e, w1[b:e], v1[b:e], w2[b:e])
        assert part.dtype == torch.float32
        assert m.get_last_error() == 0
        got = to_numpy(part)
        ref = oracle.layer_experts_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, dt, K, b, e)
        # the bound on the rows of the tokens the share serves (the others,
        # zero, would only shrink the RMS the bound scales with); rows of
        # tokens that selected none of the share's experts are zero
        served = np.any(ref, axis=1)
        extra = None
        if slot_allow is not None:
            extra = sum(np.where(((ix >= b) & (ix < e))[:, None], a, 0.0) for ix, a in slot_allow)
        if np.any(served):
            assert_parity(got[served], ref[served], dt, f"share [{b},{e})",
                          extra=None if extra is None else extra[served])
        assert not np.any(got[~served]), f"share [{b},{e}): foreign rows"
        total += got
    full = None if slot_allow is None else sum(a for _, a in slot_allow)
    assert_parity(total, want, dt, "sum of the shares", extra=full)


@pytest.mark.parametrize("T", [1, 40, 300])
def test_residual_on_one_share_and_whole_range(T):
    """The residual given to one share is carried once; the share of
    [0, E) is the whole layer (fp32 out)."""
    m = moe()
    sh = gen.LayerShape(320, 448, 6, 2, "bf16")
    L = gen.host_layer(sh, T, 23)
    d = _dims(m, sh)
    x, w_r, w1, v1, w2 = [dev(a, "bf16") for a in (L.x, L.w_r, L.w1, L.v1, L.w2)]
    res = gen.host_normal((T, sh.d_model), 1.0, "f32", 23, "residual")
    res64 = gen.to_f64(res, "f32")
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, "bf16", 2, residual=res64)
    a = m.layer_forward_experts(d, x, w_r, 0, 2, w1[0:2], v1[0:2], w2[0:2],
                                residual=dev(res, "f32"))
    b = m.layer_forward_experts(d, x, w_r, 2, 6, w1[2:6], v1[2:6], w2[2:6])
    assert_parity(to_numpy(a) + to_numpy(b), want, "bf16", "residual on one share")
    whole = m.layer_forward_experts(d, x, w_r, 0, 6, w1, v1, w2, residual=dev(res, "f32"))
    assert_parity(to_numpy(whole), want, "bf16", "share of every expert")
    assert m.get_last_error() == 0


def test_expert_range_validation():
    m = moe()
    sh = gen.LayerShape(64, 64, 4, 2, "bf16")
    L = gen.host_layer(sh, 4, 29)
    d = _dims(m, sh)
    x, w_r, w1, v1, w2 = [dev(a, "bf16") for a in (L.x, L.w_r, L.w1, L.v1, L.w2)]
    for b, e in ((2, 2), (3, 1), (-1, 2), (0, 5)):
        with pytest.raises(m.MoeError) as ex:
            m.layer_forward_experts(d, x, w_r, b, e, w1, v1, w2)
        assert ex.value.status == 1


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _ep_rank(rank, world, port, case, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    from paper_2506_23635_gb300 import expert_parallel as ep
    from paper_2506_23635_gb300 import inputs as g
    from paper_2506_23635_gb300 import moe as m

    D, F, E, K, T = case
    sh = g.LayerShape(D, F, E, K, "bf16")
    L = g.host_layer(sh, T, 31)
    torch.cuda.set_device(0)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    t = [g.host_to_torch(a, "bf16", "cuda") for a in (L.x, L.w_r, L.w1, L.v1, L.w2)]
    res = g.host_to_torch(g.host_normal((T, D), 1.0, "f32", 31, "residual"), "f32", "cuda")
    shard = ep.ExpertShard.from_full(t[1], t[2], t[3], t[4], world, rank)
    d = m.dims(D, F, E, K, torch.bfloat16)
    y = ep.layer_forward(d, t[0], shard, residual=res)
    torch.cuda.synchronize()
    out[rank] = y.cpu().numpy().astype(np.float64)
    dist.destroy_process_group()


@pytest.mark.parametrize("case", [(256, 384, 8, 2, 1), (256, 384, 8, 2, 200)])
def test_two_ranks_gloo_on_one_gpu(case):
    """Two ranks, each holding half of the experts, run their shares on the
    one GPU (no kernel of one rank waits on the other's) and sum them with a
    gloo all-reduce; both ranks end with the whole layer plus the residual."""
    need_gpu()
    import torch.multiprocessing as mp

    D, F, E, K, T = case
    sh = gen.LayerShape(D, F, E, K, "bf16")
    L = gen.host_layer(sh, T, 31)
    res = gen.to_f64(gen.host_normal((T, D), 1.0, "f32", 31, "residual"), "f32")
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, "bf16", K, residual=res)
    # the shared dict's manager process is spawned too: nothing is forked
    # after this process has initialised CUDA
    out = mp.get_context("spawn").Manager().dict()
    mp.start_processes(_ep_rank, args=(2, _free_port(), case, out), nprocs=2, join=True,
                       start_method="spawn")
    for r in range(2):
        assert_parity(out[r], want, "bf16", f"rank {r}")
    assert np.array_equal(out[0], out[1])
