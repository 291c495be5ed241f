"""bench.py's multi-process plumbing and its reference arm, on CPU.

The layer does not shard, so N GPUs run N replicas: the only cross-rank
steps are a barrier and the max of the per-rank step time.  Those run here
as gloo ranks (world size 2)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench

    dist = bench.init_dist(world, "gloo")
    bench.barrier(dist)
    v = bench.max_over_ranks(1.5 + rank, dist)
    out[rank] = v
    dist.destroy_process_group()


def test_max_over_ranks_gloo():
    world = 2
    out = mp.Manager().dict()
    mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
    assert dict(out) == {0: 2.5, 1: 2.5}


def _run(args, env=None, timeout=600):
    e = dict(os.environ, **(env or {}))
    e["CUDA_VISIBLE_DEVICES"] = ""  # the reference arm runs on the host cores
    p = subprocess.run([sys.executable] + args, cwd=ROOT, capture_output=True, text=True,
                       timeout=timeout, env=e)
    assert p.returncode == 0, p.stderr[-2000:]
    return [json.loads(l) for l in p.stdout.splitlines() if l.startswith("{")]


def test_reference_arm_tiny():
    lines = _run(["bench.py", "--impl", "reference", "--workload", "tiny-decode-t8",
                  "--steps", "2", "--warmup", "1"])
    assert len(lines) == 1
    l = lines[0]
    assert l["impl"] == "reference" and l["unit"] == "us/token-step"
    assert l["value"] > 0 and l["higher_is_better"] is False
    assert l["cpu_baseline"]["kind"] == "oracle" and l["cpu_baseline"]["cores"] >= 1
    assert l["e2e"]["h2d_bytes_per_step"] == 0
    assert l["config"]["workload"] == "tiny-decode-t8"


def test_reference_arm_under_torchrun_prints_once():
    lines = _run(["-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
                  "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
                  "bench.py", "--impl", "reference", "--workload", "tiny-decode-t8",
                  "--steps", "1", "--warmup", "1", "--gpus", "2"])
    assert len(lines) == 1 and lines[0]["impl"] == "reference"
