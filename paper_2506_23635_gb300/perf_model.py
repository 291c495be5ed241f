"""The paper's performance model (Eq. 1), and its refit for one GB300.

Eq. 1 of arxiv 2506.23635 bounds the time per generated token of the
expert-parallel DBRX deployment from below by

    max(GPU load, GPU compute) + communication latency x layers
                               + communication data / bandwidth,

where GPU load = (attention parameter bytes + expert parameter bytes x
E[executed experts per node per layer]) / memory bandwidth and GPU compute
is the same with FLOPs over the bf16 rate.  The sizes come from Table 1's
notes (a)-(e).  ``eq1`` reproduces Table 5 (pinned by tests/golden).

On one GB300 there is no communication and only the MoE block is in scope,
so the refit (``gb300_moe_layer_time``) is one layer's
max(expert bytes of the U distinct selected experts / HBM bandwidth,
expert FLOPs of the T*K slots / bf16 rate).
"""
from __future__ import annotations

import dataclasses


@dataclasses.dataclass(frozen=True)
class DbrxSizes:
    """Table 1 model variables."""
    layers: int = 40
    precision_bytes: int = 2
    d_embed: int = 6144
    d_qkv_hidden: int = 8192
    d_ffn: int = 10752

    @property
    def params_sa_bytes(self) -> float:  # note (b)
        return (self.d_qkv_hidden * self.d_embed + self.d_embed ** 2) * self.layers * \
            self.precision_bytes

    @property
    def flops_sa(self) -> float:  # note (c)
        return 2.0 * self.params_sa_bytes

    @property
    def params_expert_bytes(self) -> float:  # note (d)
        return self.d_embed * self.d_ffn * 3 * self.layers * self.precision_bytes

    @property
    def flops_expert(self) -> float:  # note (e)
        return 2.0 * self.d_embed * self.d_ffn * 3 * self.layers

    @property
    def comm_data_bytes(self) -> float:  # note (a)
        return self.d_embed * 4 * self.layers * self.precision_bytes


@dataclasses.dataclass(frozen=True)
class Node:
    bf16_flops: float = 54e12          # M2 Ultra GPU, Table 1
    memory_bandwidth: float = 800e9    # bytes/s, Table 1
    comm_bandwidth: float = 1.25e9     # bytes/s, 10 GbE, Table 1
    comm_latency: float = 1e-3         # s, measured, Table 1


def eq1(exec_experts: float, node: Node = Node(), m: DbrxSizes = DbrxSizes()) -> dict:
    """Eq. 1: lower bound of the time per generated token (seconds)."""
    load = (m.params_sa_bytes + m.params_expert_bytes * exec_experts) / node.memory_bandwidth
    compute = (m.flops_sa + m.flops_expert * exec_experts) / node.bf16_flops
    latency = node.comm_latency * m.layers
    transfer = m.comm_data_bytes / node.comm_bandwidth
    time = max(load, compute) + latency + transfer
    return dict(load=load, compute=compute, latency=latency, transfer=transfer, time=time,
                tp=1.0 / time)


def gb300_moe_layer_time(T: int, distinct_experts: float, hbm_bytes_per_s: float,
                         bf16_flops: float, d_model: int = 6144, ffn_hidden: int = 10752,
                         top_k: int = 4) -> dict:
    """Eq. 1 refit to one MoE layer on one GPU with every expert resident:
    max(load of the distinct selected experts, compute of all T*K slots)."""
    expert_bytes = 3.0 * d_model * ffn_hidden * 2
    load = distinct_experts * expert_bytes / hbm_bytes_per_s
    compute = 2.0 * T * top_k * 3 * d_model * ffn_hidden / bf16_flops
    return dict(load=load, compute=compute, time=max(load, compute),
                bound="load" if load >= compute else "compute")


def expected_distinct_experts(T: int, n_experts: int = 16, top_k: int = 4) -> float:
    """E[#distinct experts] when T tokens each pick K of E uniformly."""
    return n_experts * (1.0 - (1.0 - top_k / n_experts) ** T)
