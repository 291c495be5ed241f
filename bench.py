"""Benchmark of the DBRX-shaped MoE layer on GB300.

Default workload: one DBRX-shaped layer (D=6144, F=10752, E=16, K=4, bf16
weights, fp32 accumulation) in decode with one token per step -- the
configuration the headline metric (MoE-layer microseconds per token-step and
achieved HBM GB/s) is quoted on.  A step is one pass of the whole layer
(route, dispatch, expert up-projection + GLU, down-projection + combine) over
one fresh token; the tokens cycle through a seeded pool, so the four experts a
step reads change from step to step.  Each step streams about 1.59 GB of
expert weights, far more than the 129 MB L2, so no L2 flush is needed.

Prints ONE JSON line on rank 0.  --impl reference times the fp64 CPU oracle
on the host cores instead (the reference arm of this benchmark).

Launch: python bench.py [--gpus N --steps K --warmup W]; for N > 1 under
torchrun, one rank per GPU, each running an independent replica of the layer.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

from paper_2506_23635_gb300 import inputs as gen  # noqa: E402

METRIC = "MoE-layer us/token-step (DBRX-shaped layer, decode)"
UNIT = "us/token-step"
SEED = 1234
POOL = 64  # distinct token inputs cycled through by the timed steps
HBM_FALLBACK_GBS = 6800.0

WORKLOADS = {
    # name: (shape, tokens per step)
    "dbrx-decode-t1": (gen.DBRX, 1),
    "dbrx-decode-t8": (gen.DBRX, 8),
    "dbrx-decode-t64": (gen.DBRX, 64),
    # the same per-launch work as dbrx-decode-t1 (4 experts streamed) with
    # only 4 experts resident (1.6 GB): the small case for ncu captures
    "dbrx4-decode-t1": (gen.LayerShape(6144, 10752, 4, 4, "bf16"), 1),
}


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=4000)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", choices=sorted(WORKLOADS), default="dbrx-decode-t1")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=12.0,
                   help="time budget of the oracle sample")
    return p.parse_args()


# --------------------------------------------------------------------------
# distributed plumbing (replicas only: the layer does not shard)
# --------------------------------------------------------------------------


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def init_dist(world: int, backend: str):
    if world <= 1:
        return None
    import torch.distributed as dist

    os.environ.setdefault("MASTER_ADDR", "127.0.0.1")
    dist.init_process_group(backend=backend)
    return dist


def max_over_ranks(value: float, dist, device=None) -> float:
    if dist is None:
        return value
    import torch

    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist):
    if dist is not None:
        dist.barrier()


# --------------------------------------------------------------------------
# clocks during the timed region
# --------------------------------------------------------------------------

CLOCK_FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    """nvidia-smi sampled every 100 ms; only samples whose timestamp falls in
    the marked window (the timed region) are summarised."""

    def __init__(self, gpu_index: int):
        self.proc = None
        self.gpu = gpu_index
        self.window = (0.0, 0.0)

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={CLOCK_FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.gpu)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None

    def mark(self, t0: float, t1: float):
        self.window = (t0, t1)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        import datetime

        rows = []
        for line in out.strip().splitlines():
            f = [c.strip() for c in line.split(",")]
            if len(f) < 10:
                continue
            try:
                ts = datetime.datetime.strptime(f[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                rows.append((ts, float(f[2]), float(f[3]), float(f[4]), f[6:10]))
            except ValueError:
                continue
        t0, t1 = self.window
        inside = [r for r in rows if t0 <= r[0] <= t1]
        scope = "timed region"
        if not inside:  # region shorter than the sampling period
            inside = [r for r in rows if r[3] > 0.5 * max(x[3] for x in rows)] if rows else []
            scope = "under load around the timed region"
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in inside for n, v in zip(names, r[4]) if v.lower() == "active"})
        return {"sm_mhz": statistics.median([r[1] for r in inside]) if inside else None,
                "sm_max_mhz": max(r[2] for r in inside) if inside else None,
                "power_w_max": max(r[3] for r in inside) if inside else None,
                "samples": len(inside), "scope": scope, "reasons": reasons}


# --------------------------------------------------------------------------
# roofline bookkeeping
# --------------------------------------------------------------------------


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return json.load(f), "measured"
    except (OSError, ValueError):
        return {"hbm_gbs": HBM_FALLBACK_GBS}, "fallback"


def source_digest() -> str:
    """sha256 over the CUDA sources: ties a committed ncu counter to the code
    it was taken on."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2506_23635_gb300", "csrc")
    for name in sorted(os.listdir(csrc)):
        if name.endswith((".cu", ".cuh")):
            with open(os.path.join(csrc, name), "rb") as f:
                h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def committed_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary for this kernel
    and workload, or None if there is none or the sources changed since."""
    path = os.path.join(ROOT, "profiles", f"ncu_{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    s = re.search(r"source_digest:\s*([0-9a-f]+)", text)
    if not m or not s or s.group(1) != source_digest():
        return None
    return float(m.group(1))


def algorithmic_bytes(kernel: str, shape: gen.LayerShape, T: int, U: float) -> float:
    """Bytes a kernel must move per launch: the weights of the U distinct
    selected experts it streams, plus its activations."""
    D, F, E, K = shape.d_model, shape.ffn_hidden, shape.n_experts, shape.top_k
    S = T * K
    if kernel == "up_glu_gemv":  # fp32 h
        return U * 2 * F * D * 2 + T * D * 2 + S * F * 4
    if kernel == "down_combine_gemv":
        return U * D * F * 2 + S * F * 4 + T * D * 2
    if kernel == "up_glu_stream":  # bf16 h
        return U * 2 * F * D * 2 + T * D * 2 + S * F * 2
    if kernel == "down_combine_stream":
        return U * D * F * 2 + S * F * 2 + T * D * 2
    if kernel in ("route", "route_dispatch_small"):
        return D * E * 2 + T * D * 2 + S * 8
    return 0.0


# --------------------------------------------------------------------------
# our arm
# --------------------------------------------------------------------------


def token_pool(shape, T, seed):
    """POOL gap-conditioned token batches [POOL, T, D] sharing one router."""
    D, E = shape.d_model, shape.n_experts
    w_r = gen.host_normal((D, E), gen.W_STD, shape.dtype, seed, "w_r")
    xs = []
    for i in range(POOL):
        x = gen.host_normal((T, D), gen.X_STD, shape.dtype, seed, "x", i)
        xs.append(gen.gap_condition_tokens(x, w_r, shape, seed + i))
    return np.stack(xs), w_r


def run_ours(args):
    import torch

    from paper_2506_23635_gb300 import moe

    rank, local, world = dist_env()
    torch.cuda.set_device(local)
    dist = init_dist(world, "nccl")
    dev = torch.device("cuda", local)
    shape, T = WORKLOADS[args.workload]
    D, F, E, K = shape.d_model, shape.ffn_hidden, shape.n_experts, shape.top_k

    w1, v1, w2 = gen.device_expert_weights(shape, SEED, dev)
    xs_host, w_r_host = token_pool(shape, T, SEED)
    xs = gen.host_to_torch(xs_host, shape.dtype, dev)  # [POOL, T, D]
    w_r = gen.host_to_torch(w_r_host, shape.dtype, dev)
    d = moe.dims(D, F, E, K, torch.bfloat16)
    ws = moe.alloc_workspace(d, T, dev)
    out = torch.empty((T, D), dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream(dev)

    # distinct experts per step (algorithmic bytes), from the path's own routing
    U = []
    for i in range(POOL):
        idx, _, _ = moe.route(d, xs[i], w_r)
        U.append(len(set(idx.cpu().numpy().reshape(-1).tolist())))
    U_mean = float(np.mean(U))

    def step(i):
        moe.layer_forward(d, xs[i % POOL], w_r, w1, v1, w2, out=out, ws=ws, stream=stream)

    for i in range(args.warmup):
        step(i)
    moe.check_device_errors(stream)

    # ---- timed region: K steps, device-resident inputs ----
    clocks = ClockSampler(local)
    clocks.start()
    t_warm = time.time()
    i = 0
    while time.time() - t_warm < 0.5:  # keep the GPU busy while nvidia-smi starts
        step(i)
        i += 1
        if i % 64 == 0:
            torch.cuda.synchronize()
    barrier(dist)
    torch.cuda.synchronize()
    n_launch0 = moe.launch_count()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    wall0 = time.time()
    ev0.record(stream)
    for i in range(args.steps):
        step(i)
    ev1.record(stream)
    torch.cuda.synchronize()
    clocks.mark(wall0, time.time())
    barrier(dist)
    launches = moe.launch_count() - n_launch0
    ms = ev0.elapsed_time(ev1) / args.steps
    ms_max = max_over_ranks(ms, dist, dev)

    # ---- the same K steps again with every kernel launch bracketed by CUDA
    # events on its own stream: per-kernel durations for the roofline (the
    # events cut the overlap between launches, so this pass is not `value`) ----
    moe.profile_reset()
    moe.profile_enable(True)
    for i in range(args.steps):
        step(i)
    torch.cuda.synchronize()
    moe.profile_enable(False)
    kstats = moe.profile_read()
    clk = clocks.stop()
    moe.check_device_errors(stream)

    # ---- end to end through the public API with host buffers ----
    x_pin = torch.from_numpy(xs_host.view(np.int16)).view(torch.bfloat16).pin_memory()
    out_pin = torch.empty((T, D), dtype=torch.bfloat16).pin_memory()
    x_dev = torch.empty((T, D), dtype=torch.bfloat16, device=dev)
    e2e_steps = max(1, args.steps // 2)

    def e2e_step(i):
        x_dev.copy_(x_pin[i % POOL], non_blocking=True)
        moe.layer_forward(d, x_dev, w_r, w1, v1, w2, out=out, ws=ws, stream=stream)
        out_pin.copy_(out, non_blocking=True)

    for i in range(3):
        e2e_step(i)
    barrier(dist)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(e2e_steps):
        e2e_step(i)
    e1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, dist, dev)

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    # ---- roofline of the dominant kernel ----
    dominant = max(kstats, key=lambda k: kstats[k][1])
    n_dom, ms_dom = kstats[dominant]
    avg_s = ms_dom / n_dom / 1e3
    alg = algorithmic_bytes(dominant, shape, T, U_mean)
    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", HBM_FALLBACK_GBS))
    achieved = alg / avg_s / 1e9
    traffic = committed_traffic(dominant, args.workload)
    step_bytes = sum(algorithmic_bytes(k, shape, T, U_mean) for k in kstats)

    us_per_token = ms_max * 1e3 / (T * world)
    line = {
        "metric": METRIC, "value": round(us_per_token, 3), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_max, 5), "higher_is_better": False,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,0.02^2) bf16 weights, N(0,1) tokens, gap-conditioned router)",
        "config": {
            "workload": args.workload, "d_model": D, "ffn_hidden": F, "n_experts": E,
            "top_k": K, "tokens_per_step": T, "accumulate": "f32",
            "distinct_experts_per_step": U_mean,
            "l2": "inputs larger than L2: each step streams its selected experts' weights "
                  f"({step_bytes / 1e9:.2f} GB) vs 129 MB L2",
            "parallelism": "replicas only" if world > 1 else "single GPU",
        },
        "achieved_hbm_gbs_step": round(step_bytes / (ms_max / 1e3) / 1e9, 1),
        "roofline": {
            "kernel": dominant, "bound": "hbm", "achieved": round(achieved, 1),
            "peak": peak, "unit": "GB/s", "frac": round(achieved / peak, 4),
            "peak_source": f"{peak_src} hbm_gbs" + (" (burst copy)" if peak_src == "measured" else ""),
            "traffic": traffic, "algorithmic_bytes_per_launch": alg,
            "avg_launch_us": round(avg_s * 1e6, 2),
            "timing": "CUDA events around each launch on its stream, over a second "
                      "pass of the same K steps",
        },
        "kernels": {k: {"launches": v[0], "avg_us": round(v[1] / v[0] * 1e3, 2),
                        "share": round(v[1] / sum(s[1] for s in kstats.values()), 4)}
                    for k, v in kstats.items()},
        "gpu_launches": int(launches),
        "clocks": clk,
        "e2e": {"value": round(e2e_ms * 1e3 / (T * world), 3), "unit": UNIT,
                "h2d_bytes_per_step": T * D * 2, "d2h_bytes_per_step": T * D * 2},
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(shape, T, xs_host, w_r_host, (w1, v1, w2),
                                            args.cpu_seconds)
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


# --------------------------------------------------------------------------
# the fp64 oracle on the host cores
# --------------------------------------------------------------------------


def host_weights(shape, weights_dev):
    return [gen.torch_to_host(t, shape.dtype) for t in weights_dev]


def cpu_baseline(shape, T, xs_host, w_r_host, weights_dev, budget_s):
    """The oracle, as it stands, on a bounded sample of the same workload:
    whole token-steps from the same token pool, until the time budget is used."""
    import oracle

    w1, v1, w2 = host_weights(shape, weights_dev)
    n, t_total = 0, 0.0
    while n < POOL and (t_total < budget_s or n == 0):
        t0 = time.perf_counter()
        oracle.layer_tokens(xs_host[n], w_r_host, w1, v1, w2, shape.dtype, shape.top_k)
        t_total += time.perf_counter() - t0
        n += 1
    return {"value": round(t_total / (n * T) * 1e6, 1), "unit": UNIT,
            "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{n} token-steps of {T} token(s) from the same pool "
                      f"({t_total:.1f} s of fp64 CPU work)"}


def run_reference(args):
    """Reference arm: the fp64 oracle timed on this machine's host cores, one
    token-step of the same workload per step; rank 0 only."""
    rank, local, world = dist_env()
    if rank != 0:
        return
    import oracle

    shape, T = WORKLOADS[args.workload]
    xs_host, w_r_host = token_pool(shape, T, SEED)
    try:
        import torch

        if not torch.cuda.is_available():
            raise RuntimeError
        torch.cuda.set_device(local)
        # the same seeded weights as our arm, drawn on the device and copied back
        w = gen.device_expert_weights(shape, SEED, torch.device("cuda", local))
        w1, v1, w2 = host_weights(shape, w)
        del w
        src = "device-drawn seeded weights copied to host"
    except (RuntimeError, ImportError):
        w1, v1, w2 = gen.host_expert_weights(shape, SEED)
        src = "host-drawn seeded weights"
    tw = time.perf_counter()
    for i in range(args.warmup):
        oracle.layer_tokens(xs_host[i % POOL], w_r_host, w1, v1, w2, shape.dtype, shape.top_k)
    per_step = (time.perf_counter() - tw) / max(1, args.warmup)
    # a bounded sample: at most ~150 s of oracle work however large K is
    steps = args.steps if per_step * args.steps <= 150 else max(3, int(150 / max(per_step, 1e-9)))
    t0 = time.perf_counter()
    for i in range(steps):
        oracle.layer_tokens(xs_host[i % POOL], w_r_host, w1, v1, w2, shape.dtype, shape.top_k)
    dt = time.perf_counter() - t0
    ms = dt / steps * 1e3
    us_tok = ms * 1e3 / T
    line = {
        "impl": "reference", "metric": METRIC, "value": round(us_tok, 1), "unit": UNIT,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms, 3), "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": f"synthetic ({src})",
        "config": {"workload": args.workload, "d_model": shape.d_model,
                   "ffn_hidden": shape.ffn_hidden, "n_experts": shape.n_experts,
                   "top_k": shape.top_k, "tokens_per_step": T},
        "cpu_baseline": {"value": round(us_tok, 1), "unit": UNIT, "kind": "oracle",
                         "cores": oracle.num_threads(),
                         "sample": f"{steps} token-steps of {T} token(s) (of {args.steps} requested)"},
        "e2e": {"value": round(us_tok, 1), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        # each oracle step is a whole token-step in fp64
        if "--steps" not in sys.argv:
            args.steps = 20
        if "--warmup" not in sys.argv:
            args.warmup = 3
        args.warmup = max(1, args.warmup)
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
