"""Expert parallelism across GPUs: the paper's decentralised design.

Sec. 4.3 (Fig. 7) of arxiv 2506.23635: every node holds the router (and,
in the paper, the attention layers) and a disjoint share of the experts.
Each node routes every token itself, runs its own experts on the tokens
that selected them, and one all-reduce of the [T, D] partial outputs per
layer sums the nodes' gated outputs (the exchange of expert outputs of
Sec. 3.1; its cost is the communication term of Eq. 1).

Here a node is a GPU rank of ``torch.distributed``.  The compute of a share
is the C ABI's ``moe_layer_forward_experts`` (every step in the library's
kernels); this module chooses the shares and sums the partials with one
all-reduce (NCCL between GPUs; over gloo, CUDA partials take a host copy).
"""
from __future__ import annotations

from dataclasses import dataclass


def expert_range(n_experts: int, world_size: int, rank: int) -> tuple:
    """The contiguous range [e_begin, e_end) of experts rank ``rank`` holds:
    an even split (Sec. 3.1: 16 experts, 4 on each of 4 nodes, 8 on each of
    2), where the first ``n_experts % world_size`` ranks take one expert more
    than the others when the count does not divide.  (The paper's 3-node
    system loads some experts on more than one node, Sec. 5.3; a disjoint
    partition is what the all-reduce of partials needs.)"""
    if world_size < 1 or not 0 <= rank < world_size:
        raise ValueError("rank outside the group")
    if n_experts < world_size:
        raise ValueError("every rank needs at least one expert")
    base, extra = divmod(n_experts, world_size)
    begin = rank * base + min(rank, extra)
    return begin, begin + base + (1 if rank < extra else 0)


def all_reduce_partials(partial, group=None, stream=None):
    """Sum a rank's partial output [T, D] (fp32) over the group, in place;
    returns it.  One collective per layer, ordered after the work on
    ``stream`` (default: torch's current stream) that wrote the partial;
    without an initialised process group (one node) the partial is already
    the sum."""
    import contextlib

    import torch
    import torch.distributed as dist

    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size(group) == 1:
        return partial
    on = torch.cuda.stream(stream) if (partial.is_cuda and stream is not None) \
        else contextlib.nullcontext()
    with on:
        if partial.is_cuda and dist.get_backend(group) == "gloo":
            host = partial.cpu()
            dist.all_reduce(host, op=dist.ReduceOp.SUM, group=group)
            partial.copy_(host)
            return partial
        dist.all_reduce(partial, op=dist.ReduceOp.SUM, group=group)
    return partial


@dataclass
class ExpertShard:
    """A rank's resident share of one layer: the whole router and the
    weights of experts [e_begin, e_end) as [n, F, D] / [n, D, F] tensors."""
    w_router: object
    e_begin: int
    e_end: int
    w1: object
    v1: object
    w2: object

    @staticmethod
    def from_full(w_router, w1, v1, w2, world_size: int, rank: int) -> "ExpertShard":
        """This rank's share cut from tensors that hold every expert (views,
        no copy; a deployment loads only its share)."""
        b, e = expert_range(w1.shape[0], world_size, rank)
        return ExpertShard(w_router, b, e, w1[b:e], v1[b:e], w2[b:e])


def layer_forward(d, x, shard: ExpertShard, residual=None, group=None, ws=None, stream=None,
                  add_residual: bool = None):
    """The whole expert-parallel layer on this rank: its share through
    ``moe_layer_forward_experts``, then the all-reduce.  The residual [T, D]
    fp32 is added once, by rank 0 of the group (``add_residual`` overrides).
    Returns the layer output [T, D] fp32 on every rank."""
    import torch.distributed as dist

    from . import moe

    if add_residual is None:
        add_residual = (not (dist.is_available() and dist.is_initialized())
                        or dist.get_rank(group) == 0)
    partial = moe.layer_forward_experts(d, x, shard.w_router, shard.e_begin, shard.e_end,
                                        shard.w1, shard.v1, shard.w2,
                                        residual=residual if add_residual else None, ws=ws,
                                        stream=stream)
    return all_reduce_partials(partial, group, stream)
