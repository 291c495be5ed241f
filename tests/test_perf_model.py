"""The performance model (Eq. 1) against the numbers the paper prints:
Table 5 from Table 1's inputs, the RDMA projection, and Table 2's
throughput = 1 / time.  CPU only."""
import json
import os

import pytest

from paper_2506_23635_gb300 import perf_model as pm

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_table5.json")))


@pytest.mark.parametrize("row", [r for r in GOLDEN["printed_rows"] if r["nodes"] <= 4],
                         ids=lambda r: f"{r['nodes']}nodes")
def test_table5_rows_from_table1(row):
    e_exec = GOLDEN["inputs_table1"]["exec_experts_per_node_per_layer"][str(row["nodes"])]
    got = pm.eq1(e_exec)
    for k in ("load", "compute", "latency", "transfer", "time"):
        assert round(got[k], 3) == pytest.approx(row[k], abs=1e-12), k
    assert round(got["tp"], 1) == pytest.approx(row["tp"], abs=1e-9)


@pytest.mark.parametrize("row", [r for r in GOLDEN["printed_rows"] if r["nodes"] > 4],
                         ids=lambda r: f"{r['nodes']}nodes")
def test_table5_rows_without_printed_experts(row):
    """Table 1 does not print E[#experts] for 6 and 8 nodes.  Some load inside
    the printed load's rounding interval must give, through Eq. 1, the
    printed time and throughput; its expert count is about one (1.00-1.12)."""
    m = pm.DbrxSizes()
    bw = pm.Node().memory_bandwidth
    hits = []
    for i in range(1001):
        load = row["load"] - 0.0005 + i * 1e-6
        e_exec = (load * bw - m.params_sa_bytes) / m.params_expert_bytes
        got = pm.eq1(e_exec)
        if (round(got["load"], 3) == row["load"] and round(got["time"], 3) == row["time"]
                and round(got["tp"], 1) == row["tp"] and got["compute"] < row["compute_below"]):
            hits.append(e_exec)
    assert hits, "no load consistent with the printed row"
    assert all(0.99 < e < 1.2 for e in hits)


def test_rdma_projection():
    """Sec. 5.5: with an RDMA NIC the two-node bound rises from 9.7 to about
    16.3 tokens/s (the paper rounds its inputs; within 0.3)."""
    p = GOLDEN["printed_rdma_projection"]
    for nic in p["nics"].values():
        node = pm.Node(comm_latency=nic["latency"], comm_bandwidth=nic["bandwidth_bits"] / 8)
        got = pm.eq1(GOLDEN["inputs_table1"]["exec_experts_per_node_per_layer"]["2"], node)
        assert abs(got["tp"] - p["tp"]) < 0.3


def test_table2_throughput_is_inverse_time():
    """Table 2 prints throughput and time per token separately; they agree to
    within 0.1 token/s (6.1 vs 1/0.166 = 6.02 is the widest)."""
    for tp, t in GOLDEN["printed_table2_times"].values():
        assert abs(1.0 / t - tp) < 0.1


def test_note_sizes():
    """Table 1 notes: ~7e9 attention bytes, ~16e9 expert bytes, ~2e6 exchange bytes."""
    m = pm.DbrxSizes()
    assert abs(m.params_sa_bytes - 7e9) / 7e9 < 0.01
    assert abs(m.params_expert_bytes - 16e9) / 16e9 < 0.01
    assert abs(m.comm_data_bytes - 2e6) / 2e6 < 0.02
    # Sec. 3.2: "each expert has roughly 7.9 billion parameters"
    assert abs(m.params_expert_bytes / 2 - 7.9e9) / 7.9e9 < 0.01


def test_gb300_refit_decode_is_load_bound():
    t1 = pm.gb300_moe_layer_time(1, 4, 6776.3e9, 1910.6e12)
    assert t1["bound"] == "load"
    assert t1["time"] == pytest.approx(4 * 3 * 6144 * 10752 * 2 / 6776.3e9)
    # prefill of 2048 tokens: compute bound
    assert pm.gb300_moe_layer_time(2048, 16, 6776.3e9, 1910.6e12)["bound"] == "compute"
    assert pm.expected_distinct_experts(1) == pytest.approx(4.0)
    assert pm.expected_distinct_experts(64) == pytest.approx(16.0, abs=1e-6)
