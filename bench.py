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
METRIC_PREFILL = "MoE-layer prefill TFLOP/s (DBRX-shaped layer)"
UNIT = "us/token-step"
SEED = 1234
POOL = 64  # distinct token inputs cycled through by the timed steps
HBM_FALLBACK_GBS = 6800.0
BF16_FALLBACK_TFLOPS = 1900.0
BF16_SUSTAINED_FALLBACK_TFLOPS = 1700.0

# name: (shape, tokens per step)
WORKLOADS = {
    **{f"dbrx-decode-t{T}": (gen.DBRX, T) for T in (1, 2, 4, 8, 16, 32, 64)},
    "dbrx-prefill-t2048": (gen.DBRX, 2048),
    # the same per-launch work as dbrx-decode-t1 (4 experts streamed) with
    # only 4 experts resident (1.6 GB): the small case for ncu captures
    "dbrx4-decode-t1": (gen.LayerShape(6144, 10752, 4, 4, "bf16"), 1),
    # a 512-token prefill of the same 4-expert layer: the small case for
    # captures of the tensor-core GEMMs
    "dbrx4-prefill-t512": (gen.LayerShape(6144, 10752, 4, 4, "bf16"), 512),
    # DBRX's router (D=6144, E=16, K=4) on 8 tokens with narrow experts
    # (F=1024, 0.6 GB resident): the small case for captures of the cluster
    # route+dispatch kernel, whose work does not depend on F
    "dbrx-router-t8": (gen.LayerShape(6144, 1024, 16, 4, "bf16"), 8),
    # the same narrow-expert layer on a 2048-token prefill (0.9 GB resident):
    # the small case for captures of the prefill routing, dispatch, gather
    # and combine kernels, whose work does not depend on F
    "dbrx-router-t2048": (gen.LayerShape(6144, 1024, 16, 4, "bf16"), 2048),
    # the tiny fp32 layer (D=256, F=512, E=4, K=2), 8 tokens: the reference
    # arm's smallest case (runs anywhere, no GPU needed)
    "tiny-decode-t8": (gen.TINY, 8),
}
PREFILL_MIN_TOKENS = 512

# whole decoder layers (the DBRX self-attention block in front of the MoE
# layer), decode at context 2048: name -> (MoE shape, sequences per step)
DECODER_WORKLOADS = {
    "dbrx-decoder-t1": (gen.DBRX, 1),
    "dbrx-decoder-t8": (gen.DBRX, 8),
    # prefill of one sequence (the paper's prompts are 128 tokens)
    "dbrx-decoder-prefill-t128": (gen.DBRX, 128),
    "dbrx-decoder-prefill-t2048": (gen.DBRX, 2048),
    # 4 DBRX-shaped experts resident (about 2 GB in all): the small cases for
    # ncu captures of the attention block's kernels
    "dbrx4-decoder-t8": (gen.LayerShape(6144, 10752, 4, 4, "bf16"), 8),
    "dbrx4-decoder-prefill-t2048": (gen.LayerShape(6144, 10752, 4, 4, "bf16"), 2048),
}
METRIC_DECODER = "Decoder-layer us/token-step (DBRX-shaped attention + MoE)"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=4000)
    p.add_argument("--warmup", type=int, default=20)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", choices=sorted(WORKLOADS) + sorted(DECODER_WORKLOADS),
                   default="dbrx-decode-t1")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-extra", action="store_true",
                   help="skip the prefill and decode-sweep side measurements")
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


# The CUDA sources each measured kernel is built from (its translation unit
# and the headers it includes); other kernels use every source.
_STREAM_SRC = ("ffn_stream.cu", "ptx.cuh", "moe_internal.cuh")
_GEMM_SRC = ("ffn_tc.cu", "ffn_tc_wm.cu", "tc.cuh", "ptx.cuh", "moe_internal.cuh")
KERNEL_SOURCES = {
    "up_glu_stream": _STREAM_SRC,
    "down_combine_stream": _STREAM_SRC,
    "gemm_up_glu_tc": _GEMM_SRC,
    "gemm_down_tc": _GEMM_SRC,
}


def source_digest(kernel: str = None) -> str:
    """sha256 over the CUDA sources of a kernel (all sources when it has no
    entry in KERNEL_SOURCES): ties a committed ncu counter to the code it was
    taken on."""
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2506_23635_gb300", "csrc")
    names = KERNEL_SOURCES.get(kernel) or [
        n for n in os.listdir(csrc) if n.endswith((".cu", ".cuh"))]
    for name in sorted(names):
        with open(os.path.join(csrc, name), "rb") as f:
            h.update(name.encode() + b"\0" + f.read())
    return h.hexdigest()[:16]


def committed_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary for this kernel
    and workload, or None if there is none or the kernel's sources changed
    since."""
    path = os.path.join(ROOT, "profiles", f"ncu_{kernel}_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", text)
    s = re.search(r"source_digest:\s*([0-9a-f]+)", text)
    if not m or not s or s.group(1) != source_digest(kernel):
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


def token_pool(shape, T, seed, pool=POOL):
    """`pool` gap-conditioned token batches [pool, T, D] sharing one router."""
    D, E = shape.d_model, shape.n_experts
    w_r = gen.host_normal((D, E), gen.W_STD, shape.dtype, seed, "w_r")
    xs = []
    for i in range(pool):
        x = gen.host_normal((T, D), gen.X_STD, shape.dtype, seed, "x", i)
        xs.append(gen.gap_condition_tokens(x, w_r, shape, seed + i))
    return np.stack(xs), w_r


def workload_config(workload, shape, T, U, world):
    """The line's ``config``, the same for both arms of a workload: its
    shape, tokens per step, the mean number of distinct experts a step reads
    (from the routing of the token pool), the L2 note and the parallelism."""
    D, F = shape.d_model, shape.ffn_hidden
    gb = U * 3 * D * F * (2 if shape.dtype == "bf16" else 4) / 1e9
    return {
        "workload": workload, "d_model": D, "ffn_hidden": F, "n_experts": shape.n_experts,
        "top_k": shape.top_k, "tokens_per_step": T, "distinct_experts_per_step": U,
        "l2": (f"inputs larger than L2: each step streams its selected experts' weights "
               f"({gb:.2f} GB) vs 129 MB L2" if gb > 0.129 else
               f"inputs smaller than L2 ({gb * 1e3:.1f} MB of selected weights per step)"),
        "parallelism": "replicas only" if world > 1 else "single GPU",
    }


def oracle_distinct_experts(xs_host, w_r_host, shape):
    """Mean distinct experts per step of a token pool, from the oracle's
    routing (equal to the GPU's: routing is bit-exact)."""
    import oracle

    U = []
    for x in xs_host:
        idx, _ = oracle.topk_gates(oracle.router_logits(x, w_r_host, shape.dtype), shape.top_k)
        U.append(len(set(idx.reshape(-1).tolist())))
    return float(np.mean(U))


def algorithmic_flops(kernel: str, shape: gen.LayerShape, T: int) -> float:
    """Multiply-adds x 2 a GEMM kernel must do per launch."""
    D, F, K = shape.d_model, shape.ffn_hidden, shape.top_k
    S = T * K
    if kernel == "gemm_up_glu_tc":
        return 2.0 * S * 2 * F * D
    if kernel == "gemm_down_tc":
        return 2.0 * S * D * F
    return 0.0


class Layer:
    """One DBRX-shaped layer resident on the device, and a timer for its steps."""

    def __init__(self, moe, shape, dev, dist):
        import torch

        self.moe, self.shape, self.dev, self.dist = moe, shape, dev, dist
        self.w = gen.device_expert_weights(shape, SEED, dev)
        self.d = moe.dims(shape.d_model, shape.ffn_hidden, shape.n_experts, shape.top_k,
                          torch.bfloat16)
        self.stream = torch.cuda.current_stream(dev)
        self._host = None

    def host_weights(self):
        """The expert weights' bytes on the host (copied once, for the oracle)."""
        if self._host is None:
            self._host = host_weights(self.shape, self.w)
        return self._host

    def inputs(self, T, pool):
        import torch

        xs_host, w_r_host = token_pool(self.shape, T, SEED, pool)
        xs = gen.host_to_torch(xs_host, self.shape.dtype, self.dev)
        w_r = gen.host_to_torch(w_r_host, self.shape.dtype, self.dev)
        ws = self.moe.alloc_workspace(self.d, T, self.dev)
        out = torch.empty((T, self.shape.d_model), dtype=torch.bfloat16, device=self.dev)
        return xs_host, w_r_host, xs, w_r, ws, out

    def distinct_experts(self, xs, w_r):
        U = []
        for i in range(xs.shape[0]):
            idx, _, _ = self.moe.route(self.d, xs[i], w_r)
            U.append(len(set(idx.cpu().numpy().reshape(-1).tolist())))
        return float(np.mean(U))

    def time_steps(self, step, steps, clocks=None):
        """ms per step over `steps` steps (CUDA events on the stream, max over
        ranks), then the same steps again with per-kernel events."""
        import torch

        moe = self.moe
        barrier(self.dist)
        torch.cuda.synchronize()
        n0 = moe.launch_count()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        wall0 = time.time()
        ev0.record(self.stream)
        for i in range(steps):
            step(i)
        ev1.record(self.stream)
        torch.cuda.synchronize()
        if clocks is not None:
            clocks.mark(wall0, time.time())
        barrier(self.dist)
        launches = moe.launch_count() - n0
        ms = max_over_ranks(ev0.elapsed_time(ev1) / steps, self.dist, self.dev)
        moe.profile_reset()
        moe.profile_enable(True)
        for i in range(steps):
            step(i)
        torch.cuda.synchronize()
        moe.profile_enable(False)
        kstats = {k: v for k, v in moe.profile_read().items() if v[0] > 0}
        moe.check_device_errors(self.stream)
        return ms, launches, kstats


def kernel_table(kstats):
    tot = sum(v[1] for v in kstats.values())
    return {k: {"launches": v[0], "avg_us": round(v[1] / v[0] * 1e3, 2),
                "share": round(v[1] / tot, 4)} for k, v in kstats.items()}


def hbm_roofline(kstats, shape, T, U, workload):
    dominant = max(kstats, key=lambda k: kstats[k][1])
    n_dom, ms_dom = kstats[dominant]
    avg_s = ms_dom / n_dom / 1e3
    alg = algorithmic_bytes(dominant, shape, T, U)
    peaks, src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", HBM_FALLBACK_GBS))
    achieved = alg / avg_s / 1e9
    return {"kernel": dominant, "bound": "hbm", "achieved": round(achieved, 1), "peak": peak,
            "unit": "GB/s", "frac": round(achieved / peak, 4),
            "peak_source": f"{src} hbm_gbs" + (" (burst copy)" if src == "measured" else ""),
            "traffic": committed_traffic(dominant, workload),
            "algorithmic_bytes_per_launch": alg, "avg_launch_us": round(avg_s * 1e6, 2),
            "timing": "CUDA events around each launch on its stream, over a second pass "
                      "of the same K steps"}


def tensor_roofline(kstats, shape, T, workload):
    gemms = {k: v for k, v in kstats.items() if algorithmic_flops(k, shape, T) > 0}
    dominant = max(gemms, key=lambda k: gemms[k][1])
    n_dom, ms_dom = gemms[dominant]
    avg_s = ms_dom / n_dom / 1e3
    flops = algorithmic_flops(dominant, shape, T)
    peaks, src = measured_peaks()
    # the GEMM is timed in a loop of a few tens of milliseconds (its own
    # launches, event-bracketed): the burst figure is its peak; the
    # seconds-long sustained figure is reported beside it
    peak = float(peaks.get("bf16_tflops", BF16_FALLBACK_TFLOPS))
    sustained = float(peaks.get("bf16_tflops_sustained", BF16_SUSTAINED_FALLBACK_TFLOPS))
    achieved = flops / avg_s / 1e12
    return {"kernel": dominant, "bound": "tensor", "achieved": round(achieved, 1), "peak": peak,
            "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
            "peak_source": f"{src} bf16_tflops (cuBLAS bf16 8192^3 GEMM, burst)",
            "frac_of_sustained_peak": round(achieved / sustained, 4),
            "traffic": committed_traffic(dominant, workload),
            "algorithmic_flops_per_launch": flops, "avg_launch_us": round(avg_s * 1e6, 2),
            "timing": "CUDA events around each launch on its stream, over a second pass "
                      "of the same K steps"}


def burst_gemms(layer, step, shape, T, n=10):
    """The expert GEMMs timed the way the burst peak was measured: single
    steps after a pause, each launch bracketed by its own CUDA events, the
    best of n -- next to the loop of steps above, whose GEMMs run at the
    power cap."""
    import torch

    moe = layer.moe
    torch.cuda.synchronize()
    time.sleep(0.5)
    best = {}
    moe.profile_enable(True)
    for i in range(n):
        moe.profile_reset()
        step(i)
        torch.cuda.synchronize()
        for k, (cnt, ms) in moe.profile_read().items():
            if cnt and algorithmic_flops(k, shape, T) > 0:
                best[k] = min(best.get(k, float("inf")), ms / cnt)
    moe.profile_enable(False)
    peak = float(measured_peaks()[0].get("bf16_tflops", BF16_FALLBACK_TFLOPS))
    out = {}
    for k, ms in best.items():
        tf = algorithmic_flops(k, shape, T) / (ms / 1e3) / 1e12
        out[k] = {"best_us": round(ms * 1e3, 2), "achieved": round(tf, 1),
                  "frac_of_burst_peak": round(tf / peak, 4)}
    return {"method": f"best of {n} single steps (each launch event-bracketed, a sync "
                      "between steps), after a 0.5 s pause", "kernels": out}


def eq1_refit(shape, T, U, ms):
    """The paper's Eq. 1 refit to one layer on this GPU (measured peaks):
    max(load of the selected experts, compute of the slots), vs measured."""
    from paper_2506_23635_gb300 import perf_model

    peaks, _ = measured_peaks()
    m = perf_model.gb300_moe_layer_time(
        T, U, float(peaks.get("hbm_gbs", HBM_FALLBACK_GBS)) * 1e9,
        float(peaks.get("bf16_tflops", BF16_FALLBACK_TFLOPS)) * 1e12, shape.d_model,
        shape.ffn_hidden,
        shape.top_k)
    return {"model_ms": round(m["time"] * 1e3, 4), "bound": m["bound"],
            "measured_over_model": round(ms / (m["time"] * 1e3), 3)}


def measure_extra(layer, workload, steps, warmup, cpu_seconds=None):
    """A secondary workload of the same layer: a few timed steps, and (with
    ``cpu_seconds``) the oracle timed on a bounded sample of it."""
    shape, T = WORKLOADS[workload]
    pool = 4 if T >= PREFILL_MIN_TOKENS else 16
    xs_host, w_r_host, xs, w_r, ws, out = layer.inputs(T, pool)
    w1, v1, w2 = layer.w
    d, moe = layer.d, layer.moe

    def step(i):
        moe.layer_forward(d, xs[i % pool], w_r, w1, v1, w2, out=out, ws=ws, stream=layer.stream)

    for i in range(warmup):
        step(i)
    ms, launches, kstats = layer.time_steps(step, steps)
    r = {"workload": workload, "tokens_per_step": T, "steps": steps,
         "ms_per_step": round(ms, 4), "us_per_token_step": round(ms * 1e3 / T, 3),
         "kernels": kernel_table(kstats)}
    U = layer.distinct_experts(xs, w_r)
    r["eq1_refit"] = eq1_refit(shape, T, U, ms)
    if T >= PREFILL_MIN_TOKENS:
        flops = 2.0 * T * shape.top_k * 3 * shape.d_model * shape.ffn_hidden
        r["tflops"] = round(flops / (ms / 1e3) / 1e12, 1)
        r["roofline"] = tensor_roofline(kstats, shape, T, workload)
        r["burst"] = burst_gemms(layer, step, shape, T)
    else:
        step_bytes = U * 3 * shape.d_model * shape.ffn_hidden * 2
        r["distinct_experts_per_step"] = U
        r["achieved_hbm_gbs_step"] = round(step_bytes / (ms / 1e3) / 1e9, 1)
        peak = float(measured_peaks()[0].get("hbm_gbs", HBM_FALLBACK_GBS))
        r["frac_of_hbm_step"] = round(step_bytes / (ms / 1e3) / 1e9 / peak, 4)
    if cpu_seconds:
        r["cpu_baseline"] = cpu_baseline(shape, T, xs_host, w_r_host, layer.host_weights(),
                                         cpu_seconds)
    return r


def measure_stack(moe, dev, n_layers=16, steps=64, batches=(1, 8), graph=True, decoder=True):
    """The 16-layer DBRX-shaped stack (about 101 GB of bf16 weights resident,
    each layer independently seeded), x_{l+1} = x_l + MoE_l(RMSNorm0(x_l)) with
    an fp32 residual stream; decode at batch 1 and 8 for 64 consecutive steps,
    each step a fresh seeded batch of tokens.  Reports per-token latency over
    the stack; with `graph`, also the same steps replayed from one CUDA graph
    capture of a whole step."""
    import torch

    shape = gen.DBRX
    D, F, E, K = shape.d_model, shape.ffn_hidden, shape.n_experts, shape.top_k
    layers = gen.device_stack_layers(shape, n_layers, SEED, dev)
    sw = moe.StackWeights(layers)
    d = moe.dims(D, F, E, K, torch.bfloat16, torch.bfloat16, torch.float32)
    stream = torch.cuda.current_stream(dev)
    res = {"layers": n_layers, "resident_weight_gb": round(n_layers * 3 * E * D * F * 2 / 1e9, 2),
           "steps": steps}
    for T in batches:
        xs = torch.stack([gen.host_to_torch(gen.stack_batch(shape, T, SEED, s), "bf16",
                                            dev).float() for s in range(steps)])
        resid = torch.empty((T, D), dtype=torch.float32, device=dev)
        ws = torch.empty(moe.stack_workspace_size(d, T), dtype=torch.uint8, device=dev)

        def step(s):
            resid.copy_(xs[s % steps])
            moe.stack_forward(d, sw, resid, ws=ws, stream=stream)

        for s in range(3):
            step(s)
        moe.check_device_errors(stream)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s in range(steps):
            step(s)
        e1.record(stream)
        torch.cuda.synchronize()
        moe.check_device_errors(stream)
        ms = e0.elapsed_time(e1) / steps
        r = {"ms_per_step": round(ms, 4), "us_per_token_step": round(ms * 1e3 / T, 2),
             "tokens_per_s": round(T / (ms / 1e3), 1)}
        if graph:
            try:
                g = torch.cuda.CUDAGraph()
                xin = torch.empty_like(resid)
                gs = torch.cuda.Stream(dev)
                gs.wait_stream(stream)
                with torch.cuda.stream(gs):
                    for _ in range(2):
                        resid.copy_(xin)
                        moe.stack_forward(d, sw, resid, ws=ws, stream=gs)
                torch.cuda.synchronize()
                with torch.cuda.graph(g, stream=gs):
                    resid.copy_(xin)
                    moe.stack_forward(d, sw, resid, ws=ws, stream=gs)
                for s in range(3):
                    xin.copy_(xs[s])
                    g.replay()
                torch.cuda.synchronize()
                e0.record(stream)
                for s in range(steps):
                    xin.copy_(xs[s % steps])
                    g.replay()
                e1.record(stream)
                torch.cuda.synchronize()
                moe.check_device_errors(stream)
                gms = e0.elapsed_time(e1) / steps
                r["graph"] = {"ms_per_step": round(gms, 4),
                              "us_per_token_step": round(gms * 1e3 / T, 2)}
            except Exception as exc:  # report, keep the plain numbers
                r["graph"] = {"error": str(exc)[:200]}
        res[f"batch{T}"] = r
    if decoder:
        res["decoder"] = _decoder_stack(moe, dev, layers, d, n_layers, steps, batches)
    del layers, sw
    torch.cuda.empty_cache()
    return res


def _decoder_stack(moe, dev, moe_layers, d, n_layers, steps, batches, ctx_len=2048):
    """The same 16 MoE layers as full decoder layers: a DBRX self-attention
    block (D_qkv = 8,192) in front of each.  Batch T = T sequences decoding
    64 consecutive positions ending at ctx_len - 1 (caches pre-filled with
    synthetic earlier entries)."""
    import torch

    a_shape = gen.DBRX_ATTN
    a = moe.sa_dims(a_shape.d_model, a_shape.n_heads, a_shape.n_kv_heads, a_shape.head_dim,
                    a_shape.rope_base)
    D = a_shape.d_model
    out = {"layers": n_layers, "context_end": ctx_len, "steps": steps}
    attn_w = [gen.device_attn_weights(a_shape, SEED + 7, dev, layer=l) for l in range(n_layers)]
    stream = torch.cuda.current_stream(dev)
    for T in batches:
        caches = [gen.device_kv_cache(a_shape, T, ctx_len, SEED + 7, dev, layer=l)
                  for l in range(n_layers)]
        W = moe.DecoderWeights([attn_w[l] + moe_layers[l] + caches[l] for l in range(n_layers)])
        xs = torch.stack([gen.host_to_torch(gen.host_normal((T, D), 1.0, "bf16", SEED, "dec-x",
                                                            T, s), "bf16", dev).float()
                          for s in range(steps)])
        seq = torch.arange(T, dtype=torch.int32, device=dev)
        pos = [torch.full((T,), ctx_len - steps + s, dtype=torch.int32, device=dev)
               for s in range(steps)]
        resid = torch.empty((T, D), dtype=torch.float32, device=dev)
        ws = torch.empty(moe.decoder_workspace_size(a, d, T), dtype=torch.uint8, device=dev)

        def step(s):
            resid.copy_(xs[s % steps])
            moe.decoder_forward(a, d, W, resid, seq, pos[s % steps], ws=ws, stream=stream)

        for s in range(3):
            step(s)
        moe.check_device_errors(stream)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for s in range(steps):
            step(s)
        e1.record(stream)
        torch.cuda.synchronize()
        moe.check_device_errors(stream)
        ms = e0.elapsed_time(e1) / steps
        out[f"batch{T}"] = {"ms_per_step": round(ms, 4), "us_per_token_step": round(ms * 1e3 / T, 2),
                            "tokens_per_s": round(T / (ms / 1e3), 1)}
        del W, caches
        torch.cuda.empty_cache()
    del attn_w
    return out


def sa_bytes(a, T, ctx_len):
    """Bytes one self-attention block must move per decode step: W_qkv and
    W_o once, every token's cached keys and values over its context, the new
    keys/values and the activations (fp32 residual in and out, bf16 ctx)."""
    D, Hq, Hkv, dh = a.d_model, a.n_heads, a.n_kv_heads, a.head_dim
    nr = (Hq + 2 * Hkv) * dh
    return (nr * D * 2 + D * Hq * dh * 2 + T * ctx_len * Hkv * dh * 2 * 2
            + T * (2 * D * 4 + Hq * dh * 2 + 2 * Hkv * dh * 2))


def measure_decoder_layer(layer, T, ctx_len=2048, steps=200, warmup=5, prefill=False):
    """One DBRX-shaped decoder layer (the self-attention block with D_qkv =
    8,192 in front of this MoE layer).  Decode: T sequences, one new token
    each, at position ctx_len - 1 of a KV cache filled with synthetic earlier
    entries.  Prefill: one sequence, positions 0..T-1 (causal).  fp32
    residual stream."""
    import torch

    moe, dev = layer.moe, layer.dev
    a_shape = gen.DBRX_ATTN
    a = moe.sa_dims(a_shape.d_model, a_shape.n_heads, a_shape.n_kv_heads, a_shape.head_dim,
                    a_shape.rope_base)
    d32 = moe.dims(layer.shape.d_model, layer.shape.ffn_hidden, layer.shape.n_experts,
                   layer.shape.top_k, torch.bfloat16, torch.bfloat16, torch.float32)
    w_qkv, w_o = gen.device_attn_weights(a_shape, SEED, dev)
    if prefill:
        ctx_len = T
    n_seq = 1 if prefill else T
    pool = 4 if prefill else 16
    kc, vc = gen.device_kv_cache(a_shape, n_seq, ctx_len, SEED, dev)
    xs_host, w_r_host = token_pool(layer.shape, T, SEED, pool)
    w_r = gen.host_to_torch(w_r_host, "bf16", dev)
    xs = gen.host_to_torch(xs_host, "bf16", dev).float()
    w1, v1, w2 = layer.w
    W = moe.DecoderWeights([(w_qkv, w_o, w_r, w1, v1, w2, kc, vc)])
    if prefill:
        seq = torch.zeros(T, dtype=torch.int32, device=dev)
        pos = torch.arange(T, dtype=torch.int32, device=dev)
    else:
        seq = torch.arange(T, dtype=torch.int32, device=dev)
        pos = torch.full((T,), ctx_len - 1, dtype=torch.int32, device=dev)
    resid = torch.empty((T, layer.shape.d_model), dtype=torch.float32, device=dev)
    ws = torch.empty(moe.decoder_workspace_size(a, d32, T), dtype=torch.uint8, device=dev)

    def step(i):
        resid.copy_(xs[i % pool])
        moe.decoder_forward(a, d32, W, resid, seq, pos, ws=ws, stream=layer.stream)

    for i in range(warmup):
        step(i)
    ms, launches, kstats = layer.time_steps(step, steps)
    sa_names = ("sa_prenorm", "qkv_rows_tc", "qkv_gemm_tc", "rope_cache", "attention_tc",
                "attention_decode_tc", "attention", "attn_merge", "o_rows_tc", "o_gemm_tc",
                "residual_add", "residual_prenorm")
    sa_ms = sum(v[1] for k, v in kstats.items() if k in sa_names) / steps
    b = sa_bytes(a, T, ctx_len)
    peak = float(measured_peaks()[0].get("hbm_gbs", HBM_FALLBACK_GBS))
    kv = T * ctx_len * a.n_kv_heads * a.head_dim * 4
    att = kstats.get("attention_decode_tc") or kstats.get("attention")
    if prefill:  # tensor work: projections 2*T*(8192 + 6144)*6144, attention ~2*2*T^2/2*48*128
        sa_flops = 2.0 * T * (a_shape.qkv_rows + a.d_model) * a.d_model \
            + 2.0 * T * (T + 1) * a.n_heads * a.head_dim
        res = {"tokens_per_step": T, "mode": "prefill (one sequence, causal)",
               "ms_per_step": round(ms, 4), "launches_per_step": launches / steps,
               "attention_block": {"us_per_step": round(sa_ms * 1e3, 2),
                                   "tflops": round(sa_flops / (sa_ms / 1e3) / 1e12, 1)},
               "kernels": kernel_table(kstats)}
        del W, w_qkv, w_o, kc, vc
        torch.cuda.empty_cache()
        return res
    res = {"tokens_per_step": T, "context": ctx_len, "ms_per_step": round(ms, 4),
           "launches_per_step": launches / steps,
           "attention_block": {"us_per_step": round(sa_ms * 1e3, 2),
                               "algorithmic_bytes": b,
                               "achieved_gbs": round(b / (sa_ms / 1e3) / 1e9, 1),
                               "frac_of_hbm": round(b / (sa_ms / 1e3) / 1e9 / peak, 4)},
           "kernels": kernel_table(kstats)}
    if att:
        s_att = att[1] / att[0] / 1e3
        res["attention_block"]["kv_read_gbs"] = round(kv / s_att / 1e9, 1)
    del W, w_qkv, w_o, kc, vc
    torch.cuda.empty_cache()
    return res


def measure_dense(layer, T, steps=100, warmup=3):
    """Busy full loading (Sec. 4.2) on the same layer: every expert computes
    every token, unselected gates zero -- the paper's static baseline."""
    shape = layer.shape
    _, _, xs, w_r, _, out = layer.inputs(T, 16)
    w1, v1, w2 = layer.w
    d, moe = layer.d, layer.moe
    import torch

    ws = torch.empty(moe.dense_workspace_size(d, T), dtype=torch.uint8, device=layer.dev)

    def step(i):
        moe.layer_forward_dense(d, xs[i % 16], w_r, w1, v1, w2, out=out, ws=ws, stream=layer.stream)

    for i in range(warmup):
        step(i)
    ms, _, kstats = layer.time_steps(step, steps)
    all_bytes = shape.n_experts * 3 * shape.d_model * shape.ffn_hidden * 2
    peak = float(measured_peaks()[0].get("hbm_gbs", HBM_FALLBACK_GBS))
    return {"tokens_per_step": T, "ms_per_step": round(ms, 4),
            "achieved_hbm_gbs_step": round(all_bytes / (ms / 1e3) / 1e9, 1),
            "frac_of_hbm_step": round(all_bytes / (ms / 1e3) / 1e9 / peak, 4),
            "kernels": kernel_table(kstats)}


def measure_expert_share(layer, T, n_nodes, steps=100, warmup=3):
    """One node's share of the expert-parallel layer (Sec. 4.3): the whole
    routing and experts [0, E/P) of a P-node split, on this GPU, through
    moe_layer_forward_experts -- the per-node MoE compute of Eq. 1, without
    the all-reduce of the partials.  Also the distinct experts of the share
    a step reads (its weight bytes)."""
    import torch

    shape = layer.shape
    E = shape.n_experts
    e_end = E // n_nodes
    pool = 4 if T >= PREFILL_MIN_TOKENS else 16
    xs_host, w_r_host, xs, w_r, ws, _ = layer.inputs(T, pool)
    w1, v1, w2 = layer.w
    d, moe = layer.d, layer.moe
    part = torch.empty((T, shape.d_model), dtype=torch.float32, device=layer.dev)

    def step(i):
        moe.layer_forward_experts(d, xs[i % pool], w_r, 0, e_end, w1[:e_end], v1[:e_end],
                                  w2[:e_end], out=part, ws=ws, stream=layer.stream)

    for i in range(warmup):
        step(i)
    ms, _, kstats = layer.time_steps(step, steps)
    U = []
    for i in range(pool):
        idx, _, _ = moe.route(d, xs[i], w_r)
        U.append(len({e for e in idx.cpu().numpy().reshape(-1).tolist() if e < e_end}))
    u_mean = float(np.mean(U))
    share_bytes = u_mean * 3 * shape.d_model * shape.ffn_hidden * 2
    peak = float(measured_peaks()[0].get("hbm_gbs", HBM_FALLBACK_GBS))
    r = {"nodes": n_nodes, "experts": [0, e_end], "tokens_per_step": T,
         "ms_per_step": round(ms, 4), "distinct_experts_of_share": u_mean,
         "kernels": kernel_table(kstats)}
    if T < PREFILL_MIN_TOKENS:
        r["frac_of_hbm_step"] = round(share_bytes / (ms / 1e3) / 1e9 / peak, 4)
    else:
        flops = 2.0 * T * shape.top_k * 3 * shape.d_model * shape.ffn_hidden / n_nodes
        r["tflops"] = round(flops / (ms / 1e3) / 1e12, 1)
    return r


def decoder_config(workload, shape, T, prefill, ctx_len=2048):
    """The ``config`` of a decoder-layer workload, the same for both arms."""
    return {"workload": workload, "d_model": shape.d_model, "ffn_hidden": shape.ffn_hidden,
            "n_experts": shape.n_experts, "top_k": shape.top_k, "tokens_per_step": T,
            "mode": ("prefill of one sequence, causal" if prefill
                     else f"decode, {T} sequences at context {ctx_len}"),
            "attention": "48 query / 8 key-value heads of 128 (D_qkv = 8192)"}


def run_decoder(args, moe, dev, dist, rank, world):
    """A whole decoder layer as the measured step (device-resident inputs);
    one JSON line with the step time per token and the attention block's
    share and roofline."""
    shape, T = DECODER_WORKLOADS[args.workload]
    prefill = "prefill" in args.workload
    layer = Layer(moe, shape, dev, dist)
    r = measure_decoder_layer(layer, T, steps=args.steps, warmup=max(3, args.warmup),
                              prefill=prefill)
    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return
    line = {
        "metric": METRIC_DECODER, "value": round(r["ms_per_step"] * 1e3 / T, 3),
        "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": max(3, args.warmup),
        "ms_per_step": r["ms_per_step"], "higher_is_better": False, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,0.02^2) bf16 weights, N(0,1) tokens, KV cache "
                "pre-filled with synthetic entries)",
        "config": decoder_config(args.workload, shape, T, prefill),
        "attention_block": r["attention_block"], "kernels": r["kernels"],
        "gpu_launches": int(r["launches_per_step"] * args.steps),
    }
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def run_ours(args):
    import torch

    from paper_2506_23635_gb300 import moe

    rank, local, world = dist_env()
    torch.cuda.set_device(local)
    dist = init_dist(world, "nccl")
    dev = torch.device("cuda", local)
    if args.workload in DECODER_WORKLOADS:
        return run_decoder(args, moe, dev, dist, rank, world)
    shape, T = WORKLOADS[args.workload]
    D, F, E, K = shape.d_model, shape.ffn_hidden, shape.n_experts, shape.top_k
    prefill = T >= PREFILL_MIN_TOKENS

    layer = Layer(moe, shape, dev, dist)
    w1, v1, w2 = layer.w
    pool = 4 if prefill else POOL
    xs_host, w_r_host, xs, w_r, ws, out = layer.inputs(T, pool)
    d, stream = layer.d, layer.stream
    U_mean = layer.distinct_experts(xs, w_r)

    def step(i):
        moe.layer_forward(d, xs[i % pool], w_r, w1, v1, w2, out=out, ws=ws, stream=stream)

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
        if i % 16 == 0:
            torch.cuda.synchronize()
    ms_max, launches, kstats = layer.time_steps(step, args.steps, clocks)
    clk = clocks.stop()

    # ---- end to end through the public API with host buffers: every step
    # copies its tokens in from pinned host memory and reads its output back
    # into pinned host memory.  The copies run on two copy streams with two
    # device buffers each, so step i+1's input and step i-1's output move
    # while step i computes (a serving loop's overlap); the timed region ends
    # when the last output has landed on the host. ----
    x_pin = torch.from_numpy(xs_host.view(np.int16)).view(torch.bfloat16).pin_memory()
    out_pin = torch.empty((2, T, D), dtype=torch.bfloat16).pin_memory()
    x_dev = torch.empty((2, T, D), dtype=torch.bfloat16, device=dev)
    out_dev = torch.empty((2, T, D), dtype=torch.bfloat16, device=dev)
    h2d, d2h = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev = lambda: torch.cuda.Event()  # noqa: E731
    ev_in, ev_done, ev_out = [ev(), ev()], [ev(), ev()], [ev(), ev()]
    e2e_steps = max(1, args.steps // 2)

    def load(i):
        b = i % 2
        h2d.wait_event(ev_done[b])  # step i-2 has finished reading x_dev[b]
        with torch.cuda.stream(h2d):
            x_dev[b].copy_(x_pin[i % pool], non_blocking=True)
        ev_in[b].record(h2d)

    def e2e_run(n, start=None):
        if start is not None:
            h2d.wait_event(start)
        load(0)
        for i in range(n):
            b = i % 2
            if i + 1 < n:
                load(i + 1)
            stream.wait_event(ev_in[b])
            stream.wait_event(ev_out[b])  # step i-2's output has left out_dev[b]
            moe.layer_forward(d, x_dev[b], w_r, w1, v1, w2, out=out_dev[b], ws=ws, stream=stream)
            ev_done[b].record(stream)
            d2h.wait_event(ev_done[b])
            with torch.cuda.stream(d2h):
                out_pin[b].copy_(out_dev[b], non_blocking=True)
            ev_out[b].record(d2h)

    e2e_run(3)
    barrier(dist)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    e2e_run(e2e_steps, start=e0)
    e1.record(d2h)
    torch.cuda.synchronize()
    e2e_ms = max_over_ranks(e0.elapsed_time(e1) / e2e_steps, dist, dev)

    # ---- secondary workloads of the same layer (rank 0's view; no timing
    # contract): the 2048-token prefill and the decode batch sweep ----
    extra = {}
    if not args.no_extra and args.workload == "dbrx-decode-t1":
        # the oracle beside every config (a third of the headline's budget
        # each), on rank 0 of a one-GPU run only
        cpu_s = None if (args.no_cpu_baseline or world > 1) else args.cpu_seconds / 3
        extra["prefill"] = measure_extra(layer, "dbrx-prefill-t2048", 20, 3, cpu_s)
        extra["decode_sweep"] = [measure_extra(layer, f"dbrx-decode-t{t}", 200, 5, cpu_s)
                                 for t in (2, 4, 8, 16, 32, 64)]
        extra["busy_full_loading"] = [measure_dense(layer, t) for t in (1, 8)]
        extra["expert_parallel_share"] = [measure_expert_share(layer, t, p)
                                          for p in (2, 4) for t in (1, 8, 2048)]
        extra["decoder_layer"] = [measure_decoder_layer(layer, t) for t in (1, 8)]
        extra["decoder_prefill"] = [measure_decoder_layer(layer, t, steps=20, warmup=3,
                                                          prefill=True) for t in (128, 2048)]
        extra["stack"] = measure_stack(moe, dev)

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    step_bytes = sum(algorithmic_bytes(k, shape, T, U_mean) for k in kstats)
    step_flops = 2.0 * T * K * 3 * D * F
    if prefill:  # whole-job tensor throughput
        metric, unit, hib = METRIC_PREFILL, "TFLOP/s", True
        value = step_flops * world / (ms_max / 1e3) / 1e12
        e2e_value = step_flops * world / (e2e_ms / 1e3) / 1e12
    else:
        metric, unit, hib = METRIC, UNIT, False
        value = ms_max * 1e3 / (T * world)
        e2e_value = e2e_ms * 1e3 / (T * world)
    line = {
        "metric": metric, "value": round(value, 3), "unit": unit,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms_max, 5), "higher_is_better": hib,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,0.02^2) bf16 weights, N(0,1) tokens, gap-conditioned router)",
        "config": workload_config(args.workload, shape, T, U_mean, world),
        "accumulate": "f32",
        "roofline": (tensor_roofline(kstats, shape, T, args.workload) if prefill
                     else hbm_roofline(kstats, shape, T, U_mean, args.workload)),
        "kernels": kernel_table(kstats),
        "gpu_launches": int(launches),
        "clocks": clk,
        "e2e": {"value": round(e2e_value, 3), "unit": unit,
                "overlap": "input copy of step i+1 and output read of step i-1 on copy "
                           "streams while step i computes",
                "h2d_bytes_per_step": T * D * 2, "d2h_bytes_per_step": T * D * 2},
    }
    if not prefill:
        line["achieved_hbm_gbs_step"] = round(step_bytes / (ms_max / 1e3) / 1e9, 1)
    line["eq1_refit"] = eq1_refit(shape, T, U_mean, ms_max)
    if extra:
        line["extra"] = extra
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(shape, T, xs_host, w_r_host, layer.host_weights(),
                                            args.cpu_seconds)
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


# --------------------------------------------------------------------------
# the fp64 oracle on the host cores
# --------------------------------------------------------------------------


def host_weights(shape, weights_dev):
    return [gen.torch_to_host(t, shape.dtype) for t in weights_dev]


def cpu_baseline(shape, T, xs_host, w_r_host, weights_host, budget_s):
    """The oracle, as it stands, on a bounded sample of the same workload:
    whole decode token-steps from the same token pool (prefill: tokens of the
    first batch), until the time budget is used.  weights_host: the expert
    tensors' bytes on the host."""
    import oracle

    w1, v1, w2 = weights_host
    prefill = T >= PREFILL_MIN_TOKENS
    n, t_total = 0, 0.0
    if prefill:
        chunk = 16
        while n < T and (t_total < budget_s or n == 0):
            toks = np.arange(n, min(T, n + chunk), dtype=np.int32)
            t0 = time.perf_counter()
            oracle.layer_tokens(xs_host[0], w_r_host, w1, v1, w2, shape.dtype, shape.top_k,
                                tokens=toks)
            t_total += time.perf_counter() - t0
            n += toks.size
        flops = 2.0 * n * shape.top_k * 3 * shape.d_model * shape.ffn_hidden
        return {"value": round(flops / t_total / 1e12, 6), "unit": "TFLOP/s",
                "cores": oracle.num_threads(), "kind": "oracle",
                "sample": f"{n} of the {T} tokens of one batch ({t_total:.1f} s of fp64 CPU work)"}
    # decode: whole token-steps, cycling through the token pool until the
    # budget is used (at most 4096 steps)
    pool = xs_host.shape[0]
    while n < 4096 and (t_total < budget_s or n == 0):
        t0 = time.perf_counter()
        oracle.layer_tokens(xs_host[n % pool], w_r_host, w1, v1, w2, shape.dtype, shape.top_k)
        t_total += time.perf_counter() - t0
        n += 1
    return {"value": round(t_total / (n * T) * 1e6, 1), "unit": UNIT,
            "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{n} token-steps of {T} token(s), cycling through a pool of {pool} "
                      f"({t_total:.1f} s of fp64 CPU work)"}


def run_reference(args):
    """Reference arm: the fp64 oracle timed on this machine's host cores on the
    same workload; rank 0 only.  Decode: one token-step per step.  Prefill: a
    step is a bounded sample of 16 tokens of the batch, reported as
    throughput."""
    rank, local, world = dist_env()
    if rank != 0:
        return
    import oracle

    decoder = args.workload in DECODER_WORKLOADS
    shape, T = DECODER_WORKLOADS[args.workload] if decoder else WORKLOADS[args.workload]
    prefill = "prefill" in args.workload if decoder else T >= PREFILL_MIN_TOKENS
    pool = 1 if prefill else POOL
    xs_host, w_r_host = token_pool(shape, T, SEED, pool)
    try:
        import torch

        if not torch.cuda.is_available():
            raise RuntimeError
        torch.cuda.set_device(local)
        # the same seeded weights as our arm, drawn on the device and copied back
        w = gen.device_expert_weights(shape, SEED, torch.device("cuda", local))
        w1, v1, w2 = host_weights(shape, w)
        del w
        torch.cuda.empty_cache()
        src = "device-drawn seeded weights copied to host"
    except (RuntimeError, ImportError):
        w1, v1, w2 = gen.host_expert_weights(shape, SEED)
        src = "host-drawn seeded weights"
    chunk = 16
    if decoder:  # the attention block's weights and caches, host-drawn
        a_shape = gen.DBRX_ATTN
        ctx_len = T if prefill else 2048
        w_qkv, w_o = gen.host_attn_weights(a_shape, SEED)
        kc, vc = (gen.to_f64(c, "bf16")
                  for c in gen.host_kv_cache(a_shape, 1 if prefill else T, ctx_len, SEED))
        seq = np.arange(T, dtype=np.int32) if not prefill else np.zeros(chunk, np.int32)
        pos = np.full(T, ctx_len - 1, np.int32)

    def one(i):
        if decoder:
            if prefill:  # a chunk of 16 consecutive positions over synthetic earlier entries
                t0 = (i * chunk) % T
                x, p = xs_host[0][t0:t0 + chunk], np.arange(t0, t0 + chunk, dtype=np.int32)
            else:
                x, p = xs_host[i % pool], pos
            oracle.decoder_layers(gen.to_f64(x, shape.dtype),
                                  [(w_qkv, w_o, w_r_host, w1, v1, w2)], shape.dtype,
                                  a_shape.n_heads, a_shape.n_kv_heads, a_shape.rope_base, 1e-6,
                                  shape.top_k, seq, p, [(kc, vc)])
        elif prefill:
            t0 = (i * chunk) % T
            toks = np.arange(t0, t0 + chunk, dtype=np.int32)
            oracle.layer_tokens(xs_host[0], w_r_host, w1, v1, w2, shape.dtype, shape.top_k,
                                tokens=toks)
        else:
            oracle.layer_tokens(xs_host[i % pool], w_r_host, w1, v1, w2, shape.dtype, shape.top_k)

    tw = time.perf_counter()
    for i in range(args.warmup):
        one(i)
    per_step = (time.perf_counter() - tw) / max(1, args.warmup)
    # a bounded sample: at most ~150 s of oracle work however large K is
    steps = args.steps if per_step * args.steps <= 150 else max(3, int(150 / max(per_step, 1e-9)))
    t0 = time.perf_counter()
    for i in range(steps):
        one(i)
    dt = time.perf_counter() - t0
    ms = dt / steps * 1e3
    if decoder and prefill:
        metric, unit, hib = METRIC_DECODER, UNIT, False
        value = round(ms * 1e3 / chunk, 1)
        sample = (f"{steps} steps of {chunk} consecutive of the {T} positions over synthetic "
                  f"earlier cache entries (of {args.steps} requested)")
    elif prefill:
        flops = 2.0 * chunk * shape.top_k * 3 * shape.d_model * shape.ffn_hidden
        metric, unit, hib = METRIC_PREFILL, "TFLOP/s", True
        value = round(flops / (ms / 1e3) / 1e12, 6)
        sample = f"{steps} steps of {chunk} of the {T} tokens (of {args.steps} requested)"
    else:
        metric, unit, hib = (METRIC_DECODER if decoder else METRIC), UNIT, False
        value = round(ms * 1e3 / T, 1)
        sample = f"{steps} token-steps of {T} token(s) (of {args.steps} requested)"
    line = {
        "impl": "reference", "metric": metric, "value": value, "unit": unit,
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms, 3), "higher_is_better": hib, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": f"synthetic ({src})",
        "config": (decoder_config(args.workload, shape, T, prefill) if decoder else
                   workload_config(args.workload, shape, T,
                                   oracle_distinct_experts(xs_host, w_r_host, shape), world)),
        "cpu_baseline": {"value": value, "unit": unit, "kind": "oracle",
                         "cores": oracle.num_threads(), "sample": sample},
        "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0,
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
