"""Host side of the expert-parallel layer (Sec. 4.3) on CPU: the expert
ranges, the shard views, and the all-reduce of the shares over a gloo group
of two ranks, with the fp64 oracle computing each rank's share (the kernels
need a GPU).  The summed shares must equal the oracle's whole layer."""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

import oracle
from paper_2506_23635_gb300 import expert_parallel as ep
from paper_2506_23635_gb300 import inputs as gen

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.mark.parametrize("E,W", [(16, 1), (16, 2), (16, 3), (16, 4), (16, 16), (7, 3), (5, 2)])
def test_expert_ranges_partition(E, W):
    ranges = [ep.expert_range(E, W, r) for r in range(W)]
    assert ranges[0][0] == 0 and ranges[-1][1] == E
    for (b0, e0), (b1, e1) in zip(ranges[:-1], ranges[1:]):
        assert e0 == b1  # contiguous and disjoint
    sizes = [e - b for b, e in ranges]
    assert min(sizes) >= 1 and max(sizes) - min(sizes) <= 1
    assert sizes == sorted(sizes, reverse=True)


def test_expert_range_rejects_bad_groups():
    with pytest.raises(ValueError):
        ep.expert_range(3, 4, 0)
    with pytest.raises(ValueError):
        ep.expert_range(16, 2, 2)


def test_shard_views_hold_the_rank_experts():
    E, F, D = 6, 4, 8
    w1 = torch.arange(E * F * D, dtype=torch.float32).reshape(E, F, D)
    w2 = torch.arange(E * D * F, dtype=torch.float32).reshape(E, D, F)
    s = ep.ExpertShard.from_full(None, w1, w1, w2, 4, 1)
    assert (s.e_begin, s.e_end) == (2, 4)
    assert torch.equal(s.w1, w1[2:4]) and torch.equal(s.w2, w2[2:4])
    assert s.w1.data_ptr() == w1[2].data_ptr()  # a view, no copy


def test_all_reduce_without_a_group_is_identity():
    p = torch.ones(3, 5)
    assert ep.all_reduce_partials(p) is p and torch.equal(p, torch.ones(3, 5))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import oracle as orc
    from paper_2506_23635_gb300 import expert_parallel as e
    from paper_2506_23635_gb300 import inputs as g

    dist.init_process_group("gloo", rank=rank, world_size=world)
    sh = g.LayerShape(48, 40, 6, 2, "f32")
    L = g.host_layer(sh, 11, 5)
    b, en = e.expert_range(sh.n_experts, world, rank)
    res = np.random.default_rng(3).normal(size=(11, 48)) if rank == 0 else None
    share = orc.layer_experts_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, "f32", sh.top_k, b, en,
                                     residual=res)
    p = torch.from_numpy(share)
    e.all_reduce_partials(p)
    out[rank] = p.numpy().copy()
    dist.destroy_process_group()


def test_two_rank_all_reduce_of_shares_gloo():
    world = 2
    out = mp.Manager().dict()
    mp.spawn(_rank, args=(world, _free_port(), out), nprocs=world, join=True)
    sh = gen.LayerShape(48, 40, 6, 2, "f32")
    L = gen.host_layer(sh, 11, 5)
    res = np.random.default_rng(3).normal(size=(11, 48))
    want, _, _ = oracle.layer_tokens(L.x, L.w_r, L.w1, L.v1, L.w2, "f32", sh.top_k,
                                     residual=res)
    for r in range(world):
        np.testing.assert_allclose(out[r], want, rtol=1e-12, atol=1e-12)
