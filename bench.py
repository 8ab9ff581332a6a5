#!/usr/bin/env python3
"""Decode benchmark of the Llama2-70B-shaped LittleBit stack on GB300.

One step = one decode token through 80 layers x 7 LittleBit linears (q, k, v,
o, gate, up, down; two rank-r paths each) as ONE persistent-kernel launch of
littlebit_stack_forward, weights resident in HBM (0.90 GB, 7x the 129 MB L2,
so every step streams them from DRAM without an explicit flush).

Prints one JSON line: tokens/s (value), HBM GB/s and its fraction of the
measured copy bandwidth (roofline), the same metric end to end through the C
ABI with host buffers (e2e), the fp64 CPU oracle timed on this host's cores
on a bounded sample (cpu_baseline), and the SM clocks seen while timing.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--layers L]
  python bench.py --config 2|3|4|6|7|8 [--steps K] [--warmup W]

--config times the single-linear workloads instead (one JSON line per case,
not the bench line): 2 = 4096x4096 r64 at T = 1, 8 (each also as "graph64":
64 distinct weight copies, one forward each, replayed as one CUDA graph, per
forward); 3 = the FFN triple at
r = 128, 512 and T = 1, 16, 64; 4 = prefill at T = 2048, 8192; 6 = the
latent-state halves (littlebit_linear_latent / _expand: the 70B key
projection at T = 1 and a 4096-token cache, 4096x4096 r512 at T = 2048);
7 = Dual-SVID initialisation of a dense weight into two paths (ms per layer);
8 = one QAT step (forward + SmoothSign backward) at 2048 tokens (TFLOP/s
against the TF32 tensor peak); 10 = the exchange floor of the 70B-shaped
stack: one token's 320 dependent rank-r all-reduces (four per layer, of the
stack's element counts) with nothing between them (littlebit_selftest_exchange).
Cases 2, 3 and the CUDA-core cases of 6 report algorithmic GB/s with L2
flushed before every call; 4 and the tensor-core cases of 6 report TFLOP/s
(2 flops per +-1 MAC, both paths) against the dense bf16 peak.

--impl reference times the CPU oracle (the reference of this build) on the
same metric; under torchrun only rank 0 runs it.  N > 1 runs independent
replicas, one per GPU (the stack does not shard; weak scaling).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "decode HBM GB/s (% of GB300 peak, cold L2) and tokens/s for 70B-shaped stack"
L2_BYTES = 129 * 1024 * 1024


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--layers", type=int, default=80,
                    help="stack depth (80 = the Llama2-70B workload; smaller only for profiling)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--config", type=int, choices=[2, 3, 4, 6, 7, 8, 9, 10], default=None,
                    help="time a single-linear workload instead of the stack")
    ap.add_argument("--only", default=None,
                    help="with --config: only the cases whose 'name:T' contains this text")
    return ap.parse_args()


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """The largest of `value` over the ranks of the default process group (the
    slowest rank's time), or `value` itself when there is one rank.  The
    tensor lives on `device` (a CUDA device under NCCL, the CPU under gloo)."""
    if world <= 1:
        return float(value)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def replica_throughput(world: int, units_per_rank: int, slowest_ms: float) -> float:
    """Whole-job units per second of `world` independent replicas, each doing
    `units_per_rank` units, timed by the slowest rank (weak scaling)."""
    return world * units_per_rank / (slowest_ms / 1e3)


def workload_config(n_layers: int) -> dict:
    from paper_2506_13771_gb300 import inputs
    s = inputs.STACK_70B
    return {"workload": "Llama2-70B-shaped LittleBit decoder stack, decode 1 token (batch 1)",
            "n_layers": n_layers, "d_model": s["d_model"], "d_kv": s["d_kv"], "d_ff": s["d_ff"],
            "ranks": {"q,o": s["r_qo"], "k,v": s["r_kv"], "gate,up,down": s["r_mlp"]},
            "paths": 2, "head_dim": s["head_dim"], "seed": inputs.SEED_BASE + 5}


# ----------------------------------------------------------------- measurement helpers


def measured_peaks() -> dict:
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f)
    except OSError:
        return {}


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples every 200 ms in a thread."""

    FIELDS = ("index,uuid,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, uuid: str | None):
        self.uuid = uuid
        self.samples = []
        self.proc = None
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 10:
                continue
            if self.uuid and self.uuid not in parts[1]:
                continue
            self.samples.append((time.time(), parts))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()

    def summary(self, t0: float, t1: float) -> dict:
        rows = [p for (t, p) in self.samples if t0 - 0.25 <= t <= t1 + 0.25]
        if not rows:
            rows = [p for (_, p) in self.samples]
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None

        sm = [num(p[2]) for p in rows if num(p[2]) is not None]
        mx = [num(p[3]) for p in rows if num(p[3]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for p in rows for i in range(4)
                          if p[6 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows),
                "power_w_max": max((num(p[4]) or 0.0) for p in rows)}


def kernel_source_sha() -> str:
    h = hashlib.sha256()
    for f in ("lb_stack.cu", "lb_common.cuh", "lb_lut.cuh"):
        with open(os.path.join(ROOT, "paper_2506_13771_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_traffic(kernel: str, sha: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken on
    the kernel source as it is now (else None)."""
    path = os.path.join(ROOT, "profiles", "traffic.txt")
    try:
        with open(path) as f:
            for line in f:
                parts = line.split()
                if len(parts) >= 3 and not line.startswith("#") and parts[0] == kernel \
                        and parts[1] == sha:
                    return float(parts[2])
    except OSError:
        pass
    return None


# ----------------------------------------------------------------- CPU oracle legs


def cpu_model() -> str:
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else platform)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    import platform
    return platform.machine()


def host_weight_bytes(layers) -> int:
    """Sign words and fp16 scales of every linear, as the device holds them."""
    return int(sum(P[k].nbytes for L in layers for P in L["paths"]
                   for k in ("v_words", "u_words", "g", "l", "h")))


def stack_io_bytes(n_layers: int) -> int:
    """x0 (bf16) in; the final hidden state, q and k / v of every layer (fp32) out."""
    s = __import__("paper_2506_13771_gb300.inputs", fromlist=["STACK_70B"]).STACK_70B
    return 2 * s["d_model"] + 4 * s["d_model"] + 4 * n_layers * (s["d_model"] + 2 * s["d_kv"])


def line_config(n_layers: int, world: int, weight_bytes: int) -> dict:
    """The bench line's config, the same for both arms."""
    return dict(workload_config(n_layers), parallelism=f"replicas{world}",
                bytes_per_token=weight_bytes + stack_io_bytes(n_layers),
                l2=("no flush: weights %.2f GB > %d MB L2, streamed from DRAM every step"
                    if weight_bytes > L2_BYTES else
                    "no flush: weights %.2f GB fit the %d MB L2 (a shortened profiling stack)")
                   % (weight_bytes / 1e9, L2_BYTES >> 20))


def oracle_chain_seconds(o, layers, x0, n_chain: int, reps: int) -> list:
    """Wall times of `reps` runs of the oracle's decode chain over the first
    n_chain layers (7 linears, attention at position 0, norms; fp64)."""
    times = []
    for _ in range(reps):
        t0 = time.perf_counter()
        o.stack_forward(layers[:7 * n_chain], x0, head_dim=128, want_q=True, want_kv=True)
        times.append(time.perf_counter() - t0)
    return times


def cpu_baseline(layers, x0, n_layers: int) -> dict:
    """The fp64 oracle's decode chain over the whole stack on all host cores,
    repeated until about 10 s of work (median), and a one-thread figure from
    the chain over the first layers (about 5 s), scaled to the whole stack."""
    import oracle
    o = oracle.default()
    o.set_threads(os.cpu_count() or 1)
    t1 = oracle_chain_seconds(o, layers, x0, n_layers, 1)[0]
    reps = max(1, min(50, int(10.0 / max(t1, 1e-3))))
    t = statistics.median(oracle_chain_seconds(o, layers, x0, n_layers, reps)) if reps > 1 else t1
    cores = o.get_threads()
    # one thread: as many leading layers as take about 5 s (the per-layer work is uniform)
    o.set_threads(1)
    per_layer_guess = t / n_layers * max(1, cores)
    n1 = max(1, min(n_layers, int(5.0 / max(per_layer_guess, 1e-4))))
    s1 = oracle_chain_seconds(o, layers, x0, n1, 1)[0] * n_layers / n1
    o.set_threads(cores)
    return {"value": 1.0 / t, "unit": "tokens/s", "cores": cores, "kind": "oracle",
            "cpu_model": cpu_model(),
            "sample": f"fp64 oracle decode chain over all {n_layers} layers on {cores} threads, "
                      f"median of {reps} run(s) of {t:.3f} s",
            "threads_1": {"value": 1.0 / s1, "unit": "tokens/s",
                          "sample": f"chain over the first {n1} of {n_layers} layers on one "
                                    f"thread, scaled by {n_layers}/{n1}"}}


def run_reference(args):
    """The fp64 CPU oracle on the same metric and workload: each step is the
    oracle's decode chain (the full stack, or -- when K + W steps of it would
    take more than about 150 s -- its first n layers, tokens/s scaled by
    n / n_layers) on all host cores; the line's value is the median step."""
    import oracle
    from paper_2506_13771_gb300 import inputs
    world, rank, _ = dist_env()
    if rank != 0:
        return
    kw = {k: v for k, v in inputs.STACK_70B.items() if k not in ("n_layers",)}
    layers, x0 = inputs.make_stack(n_layers=args.layers, **kw)
    o = oracle.default()
    o.set_threads(os.cpu_count() or 1)
    probe = oracle_chain_seconds(o, layers, x0, args.layers, 1)[0]
    n_steps = max(1, args.steps + args.warmup)
    n_chain = args.layers
    if n_steps * probe > 150.0:
        n_chain = max(1, int(150.0 / (n_steps * probe / args.layers)))
    times = oracle_chain_seconds(o, layers, x0, n_chain, n_steps)[args.warmup:] or [probe]
    per_token = statistics.median(times) * args.layers / n_chain
    value = 1.0 / per_token
    sample = (f"fp64 oracle decode chain over {'all' if n_chain == args.layers else 'the first'} "
              f"{n_chain} of {args.layers} layers per step on {o.get_threads()} threads, median "
              f"of {len(times)} step(s)" + ("" if n_chain == args.layers else
                                            f", scaled by {args.layers}/{n_chain}"))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * per_token, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data":
                "synthetic (seeded random sign bits and fp16 scales; no trained weights)",
            "config": line_config(args.layers, world, host_weight_bytes(layers)),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": o.get_threads(),
                             "kind": "oracle", "cpu_model": cpu_model(), "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------- our arm


def run_ours(args):
    import torch
    import torch.distributed as dist

    from paper_2506_13771_gb300 import build as lb_build
    from paper_2506_13771_gb300 import inputs
    from paper_2506_13771_gb300 import littlebit as lb

    world, rank, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    lb_build.build()

    kw = {k: v for k, v in inputs.STACK_70B.items() if k not in ("n_layers",)}
    layers, x0_bits = inputs.make_stack(n_layers=args.layers, **kw)
    S = lb.DeviceStack(layers, kw["head_dim"], dev)
    weight_bytes = S.nbytes
    ws = S.prepare()
    x0 = lb.bf16_tensor(x0_bits, dev)
    out = torch.empty(S.d_model, dtype=torch.float32, device=dev)
    q_out = torch.empty((S.n_layers, S.d_model), dtype=torch.float32, device=dev)
    kv_out = torch.empty((S.n_layers, 2, S.d_kv), dtype=torch.float32, device=dev)
    io_bytes = x0.numel() * 2 + out.numel() * 4 + q_out.numel() * 4 + kv_out.numel() * 4
    step_bytes = weight_bytes + io_bytes
    assert weight_bytes == host_weight_bytes(layers) and io_bytes == stack_io_bytes(args.layers)
    stream = torch.cuda.current_stream(dev)

    def step():
        lb.stack_forward(S, x0, out=out, q_out=q_out, kv_out=kv_out, ws=ws, stream=stream)

    uuid = None
    try:
        uuid = str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    sampler = ClockSampler(uuid)
    sampler.start()
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)
    if lb.poll_error(ws) != lb.LB_OK:
        raise RuntimeError("stack kernel reported an error during warm-up")

    # ---- device-timed region: K steps, per-launch CUDA events on the launch stream
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    if world > 1:
        dist.barrier()
    torch.cuda.synchronize(dev)
    t_wall0 = time.time()
    evs[0].record(stream)
    for i in range(args.steps):
        step()
        evs[i + 1].record(stream)
    torch.cuda.synchronize(dev)
    t_wall1 = time.time()
    if world > 1:
        dist.barrier()
    status = lb.poll_error(ws)
    if status != lb.LB_OK:
        raise RuntimeError(f"stack kernel reported {lb.status_string(status)}")
    per_launch_ms = [evs[i].elapsed_time(evs[i + 1]) for i in range(args.steps)]
    total_ms = max_over_ranks(evs[0].elapsed_time(evs[-1]), world, dev)
    clocks = sampler.summary(t_wall0, t_wall1)
    sampler.stop()

    # ---- end to end through the C ABI with host buffers: pinned x0 in,
    #      the step's result (the final hidden state) out, copies timed
    x_host = torch.from_numpy(x0_bits.view("int16")).pin_memory()
    out_host = torch.empty(S.d_model, dtype=torch.float32).pin_memory()
    x_dev = torch.empty(S.d_model, dtype=torch.int16, device=dev)
    e2e_steps = max(1, min(args.steps, 500))
    for _ in range(3):
        x_dev.copy_(x_host, non_blocking=True)
        lb.stack_forward(S, x_dev.view(torch.bfloat16), out=out, q_out=q_out, kv_out=kv_out,
                         ws=ws, stream=stream)
        out_host.copy_(out, non_blocking=True)
    torch.cuda.synchronize(dev)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    if world > 1:
        dist.barrier()
    e0.record(stream)
    for _ in range(e2e_steps):
        x_dev.copy_(x_host, non_blocking=True)
        lb.stack_forward(S, x_dev.view(torch.bfloat16), out=out, q_out=q_out, kv_out=kv_out,
                         ws=ws, stream=stream)
        out_host.copy_(out, non_blocking=True)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    if lb.poll_error(ws) != lb.LB_OK:
        raise RuntimeError("stack kernel reported an error in the end-to-end loop")

    ms_per_step = total_ms / args.steps
    value = replica_throughput(world, args.steps, total_ms)
    kernel_ms = statistics.mean(per_launch_ms)
    peaks = measured_peaks()
    peak = peaks.get("hbm_gbs")
    peak_src = "measured (MEASURED_PEAKS.json hbm_gbs)"
    if peak is None:
        peak, peak_src = 6800.0, "fallback 6.8 TB/s"
    achieved = step_bytes / (kernel_ms / 1e3) / 1e9
    sha = kernel_source_sha()
    traffic = recorded_traffic("k_stack", sha)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_per_step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded random sign bits and fp16 scales; no trained weights)",
        "config": line_config(args.layers, world, host_weight_bytes(layers)),
        "hbm_gbs": achieved,
        "roofline": {"bound": "hbm", "kernel": "k_stack", "achieved": achieved,
                     "peak": peak, "peak_source": peak_src, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "algorithmic_bytes_per_launch": step_bytes,
                     "kernel_ms": kernel_ms, "kernel_source_sha": sha},
        "e2e": {"value": replica_throughput(world, e2e_steps, e2e_ms), "unit": "tokens/s",
                "h2d_bytes_per_step": x_host.numel() * 2,
                "d2h_bytes_per_step": out_host.numel() * 4},
        "gpu_launches": args.steps,
        "clocks": clocks,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(layers, x0_bits, args.layers)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()


# ----------------------------------------------------------------- single-linear workloads


def run_config(args):
    import torch

    from paper_2506_13771_gb300 import build as lb_build
    from paper_2506_13771_gb300 import inputs
    from paper_2506_13771_gb300 import littlebit as lb

    lb_build.build()
    dev = torch.device("cuda", 0)
    peaks = measured_peaks()
    hbm = float(peaks.get("hbm_gbs", 6800.0))
    tc = float(peaks.get("bf16_tflops", 1900.0))
    l2 = torch.cuda.get_device_properties(dev).L2_cache_size or L2_BYTES
    flush = torch.empty(2 * l2, dtype=torch.uint8, device=dev)
    steps = max(1, min(args.steps, 200))

    def weight_bytes(L):
        return sum(P["v_words"].nbytes + P["u_words"].nbytes + 2 * (L["d_in"] + L["d_out"] + P["r"])
                   for P in L["paths"])

    def time_case(L, x_bits, T, cold, op="forward"):
        """Median ms of one call: the forward, the latent (z fp16) or the
        expansion of an fp16 latent, L2 flushed before each call when cold."""
        D = lb.DeviceLinear(L, dev)
        x = lb.bf16_tensor(x_bits, dev)
        y = torch.empty((T, D.d_out), dtype=torch.bfloat16, device=dev)
        ws = lb.new_workspace(lb.workspace_size(D, T), dev)
        z = torch.empty((T, sum(D.ranks)), dtype=torch.float16, device=dev)
        lb.linear_latent(D, x, z=z, ws=ws)
        if op == "forward":
            def call():
                lb.linear_forward(D, x, y=y, ws=ws)
        elif op == "latent":
            def call():
                lb.linear_latent(D, x, z=z, ws=ws)
        else:
            def call():
                lb.linear_expand(D, z, y=y, ws=ws)
        for _ in range(max(3, args.warmup)):
            call()
        torch.cuda.synchronize(dev)
        ts = []
        for _ in range(steps):
            if cold:
                flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            call()
            e1.record()
            torch.cuda.synchronize(dev)
            ts.append(e0.elapsed_time(e1))
        if lb.poll_error(ws) != lb.LB_OK:
            raise RuntimeError("kernel reported an error")
        return statistics.median(ts)

    def time_graph(L, x_bits, T, copies=64):
        """Sustained single-linear throughput: `copies` distinct device copies of
        the weights (so each forward streams its own), one forward each, captured
        in one CUDA graph; L2 flushed before each replay.  Median ms per forward,
        or None if the forwards cannot be captured."""
        devs = [lb.DeviceLinear(L, dev) for _ in range(copies)]
        x = lb.bf16_tensor(x_bits, dev)
        y = torch.empty((T, devs[0].d_out), dtype=torch.bfloat16, device=dev)
        ws = lb.new_workspace(max(lb.workspace_size(D, T) for D in devs), dev)
        side = torch.cuda.Stream(dev)
        side.wait_stream(torch.cuda.current_stream(dev))
        with torch.cuda.stream(side):
            for D in devs:
                lb.linear_forward(D, x, y=y, ws=ws)
        torch.cuda.current_stream(dev).wait_stream(side)
        torch.cuda.synchronize(dev)
        graph = torch.cuda.CUDAGraph()
        try:
            with torch.cuda.graph(graph):
                for D in devs:
                    lb.linear_forward(D, x, y=y, ws=ws)
        except Exception as exc:  # noqa: BLE001 - reported, not fatal
            print(f"# graph capture unavailable: {exc}", file=sys.stderr)
            return None
        ts = []
        for _ in range(max(5, min(steps, 50))):
            flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            graph.replay()
            e1.record()
            torch.cuda.synchronize(dev)
            ts.append(e0.elapsed_time(e1) / copies)
        if lb.poll_error(ws) != lb.LB_OK:
            raise RuntimeError("kernel reported an error")
        return statistics.median(ts)

    def time_multi(L, x_bits, copies=64, per_launch=24):
        """The same sustained measurement at T = 1 with the forwards grouped:
        `copies` distinct weight copies through littlebit_linear_forward_multi,
        `per_launch` linears per launch, all launches in one CUDA graph; L2
        flushed before each replay.  Median ms per forward."""
        devs = [lb.DeviceLinear(L, dev) for _ in range(copies)]
        x = lb.bf16_tensor(x_bits, dev)[0]
        y = torch.empty((copies, devs[0].d_out), dtype=torch.bfloat16, device=dev)
        groups = [devs[i:i + per_launch] for i in range(0, copies, per_launch)]
        wss = [lb.new_workspace(lb.multi_workspace_size(g), dev) for g in groups]

        def run():
            o = 0
            for g, w in zip(groups, wss):
                lb.linear_forward_multi(g, x, y=y[o:o + len(g)], ws=w)
                o += len(g)
        side = torch.cuda.Stream(dev)
        side.wait_stream(torch.cuda.current_stream(dev))
        with torch.cuda.stream(side):
            run()
        torch.cuda.current_stream(dev).wait_stream(side)
        torch.cuda.synchronize(dev)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            run()
        ts = []
        for _ in range(max(5, min(steps, 50))):
            flush.zero_()
            e0 = torch.cuda.Event(enable_timing=True)
            e1 = torch.cuda.Event(enable_timing=True)
            e0.record()
            graph.replay()
            e1.record()
            torch.cuda.synchronize(dev)
            ts.append(e0.elapsed_time(e1) / copies)
        for w in wss:
            if lb.poll_error(w) != lb.LB_OK:
                raise RuntimeError("kernel reported an error")
        return statistics.median(ts)

    def wanted(name, T):
        return args.only is None or args.only in f"{name}:{T}"

    def emit(name, cfg, T, L, ms, flops_mode, op="forward", mode="single"):
        n1 = sum(P["r"] for P in L["paths"])
        if op == "forward":
            wb = weight_bytes(L)
            act = T * (L["d_in"] + L["d_out"]) * 2
            flops = sum(2 * T * P["r"] * (L["d_in"] + L["d_out"]) for P in L["paths"])
        elif op == "latent":   # V bits, g, l; x in, z (fp16) out
            wb = sum(P["v_words"].nbytes + 2 * (L["d_in"] + P["r"]) for P in L["paths"])
            act = T * (L["d_in"] + n1) * 2
            flops = sum(2 * T * P["r"] * L["d_in"] for P in L["paths"])
        else:                  # U bits, h; z (fp16) in, y out
            wb = sum(P["u_words"].nbytes + 2 * L["d_out"] for P in L["paths"])
            act = T * (n1 + L["d_out"]) * 2
            flops = sum(2 * T * P["r"] * L["d_out"] for P in L["paths"])
        line = {"config": cfg, "case": name, "op": op, "mode": mode, "tokens": T, "ms": ms,
                "us": ms * 1e3, "bytes": wb + act, "flops": flops,
                "gbs": (wb + act) / ms / 1e6, "tflops": flops / ms / 1e9}
        if flops_mode:
            line["roofline"] = {"bound": "tensor", "achieved": line["tflops"], "peak": tc,
                                "unit": "TFLOP/s", "frac": line["tflops"] / tc,
                                "peak_source": "MEASURED_PEAKS.json bf16_tflops (burst)"}
        else:
            line["roofline"] = {"bound": "hbm", "achieved": line["gbs"], "peak": hbm,
                                "unit": "GB/s", "frac": line["gbs"] / hbm,
                                "peak_source": "MEASURED_PEAKS.json hbm_gbs"}
        print(json.dumps(line), flush=True)

    if args.config == 2:
        for T in (1, 8):
            if wanted("4096x4096 r64", T):
                L, x = inputs.config2(T)
                emit("4096x4096 r64", 2, T, L, time_case(L, x, T, True), False)
                ms = time_graph(L, x, T)
                if ms is not None:
                    emit("4096x4096 r64", 2, T, L, ms, False, mode="graph64")
                if T == 1:
                    emit("4096x4096 r64", 2, T, L, time_multi(L, x), False, mode="multi64")
    elif args.config == 3:
        for r in (128, 512):
            for T in (1, 16, 64):
                lins, x, xd = inputs.config3(r, T)
                for nm in ("gate", "up", "down"):
                    if not wanted(f"{nm} r{r}", T):
                        continue
                    xin = xd if nm == "down" else x
                    emit(f"{nm} r{r}", 3, T, lins[nm], time_case(lins[nm], xin, T, True), False)
                    if T == 1:
                        ms = time_graph(lins[nm], xin, T)
                        if ms is not None:
                            emit(f"{nm} r{r}", 3, T, lins[nm], ms, False, mode="graph64")
                        emit(f"{nm} r{r}", 3, T, lins[nm], time_multi(lins[nm], xin), False,
                             mode="multi64")
    elif args.config == 7:
        # Dual-SVID initialisation (one dense weight -> two LittleBit paths):
        # the 4096 x 4096 r64 layer and the 70B gate shape (8192 -> 28672, r320),
        # synthetic weights with a power-law singular spectrum built on the device
        g = torch.Generator(device=dev)
        g.manual_seed(20250607)
        fp32_peak = 152 * 128 * 2 * 1.92e9 / 1e12  # FP32 FMA lanes x 2 flops x SM clock
        for name, m, n, r in (("4096x4096 r64x2", 4096, 4096, 64),
                              ("gate 8192->28672 r320x2", 28672, 8192, 320)):
            if not wanted(name, 0):
                continue
            k0 = 1024
            A = torch.randn((m, k0), generator=g, device=dev) / m ** 0.5
            B = torch.randn((n, k0), generator=g, device=dev) / n ** 0.5
            sig = (1.0 + torch.arange(k0, device=dev, dtype=torch.float32)) ** -0.6
            W = (A * sig) @ B.t() + 1e-3 * torch.randn((m, n), generator=g, device=dev) / n ** 0.5
            del A, B
            lb.dual_svid(W, [r, r], iters=8)  # warm-up (workspace, first launches)
            torch.cuda.synchronize(dev)
            ts = []
            for _ in range(max(1, min(steps, 3))):
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                lb.dual_svid(W, [r, r], iters=8)
                e1.record()
                torch.cuda.synchronize(dev)
                ts.append(e0.elapsed_time(e1))
            ms = statistics.median(ts)
            k = min(r + 8, m, n)
            # GEMM flops of two paths: per path 8 iterations of R Q and R^T Y
            # (2 m n k each), the Rayleigh-Ritz R Q, the Ritz vectors, the residual
            flops = 2 * (8 * 2 * 2 * m * n * k + 2 * m * n * k + 2 * (m + n) * k * r) + 2 * m * n * r
            line = {"config": 7, "case": name, "op": "dual_svid", "ms": ms,
                    "gemm_tflops": flops / ms / 1e9,
                    "roofline": {"bound": "alu", "achieved": flops / ms / 1e9,
                                 "peak": fp32_peak, "unit": "TFLOP/s",
                                 "frac": flops / ms / 1e9 / fp32_peak,
                                 "peak_source": "derived: 152 SMs x 128 FP32 lanes x 2 x 1.92 GHz"}}
            print(json.dumps(line), flush=True)
    elif args.config == 8:
        # one QAT step (forward + SmoothSign backward) of a LittleBit linear on
        # latent fp32 factors, 2048 tokens (the paper's training sequence length)
        g = torch.Generator(device=dev)
        g.manual_seed(20250608)
        tf32_peak = tc * 1.1 / 2.25  # measured dense bf16 x nominal TF32 / bf16 ratio
        for name, d_in, d_out, r in (("4096x4096 r512x2", 4096, 4096, 512),
                                     ("gate 8192->28672 r320x2", 8192, 28672, 320)):
            T = 2048
            if not wanted(name, T):
                continue
            layer = {"d_in": d_in, "d_out": d_out, "paths": [
                {"r": r, "u": 0.02 * torch.randn((d_out, r), generator=g, device=dev),
                 "v": 0.02 * torch.randn((d_in, r), generator=g, device=dev),
                 "g": 0.5 + torch.rand(d_in, generator=g, device=dev),
                 "l": 0.5 + torch.rand(r, generator=g, device=dev),
                 "h": 0.5 + torch.rand(d_out, generator=g, device=dev)} for _ in range(2)]}
            TL = lb.TrainLinear(layer, dev)
            x = torch.randn((T, d_in), generator=g, device=dev)
            dy = torch.randn((T, d_out), generator=g, device=dev)
            ws = TL.workspace(T, dev)
            # the backward reuses the forward's folded factors and latent
            # (littlebit_train_backward_saved), as a framework keeps activations
            for _ in range(3):
                lb.train_forward(TL, x, ws=ws)
                lb.train_backward(TL, x, dy, ws=ws, saved=True)
            torch.cuda.synchronize(dev)
            ts = []
            for _ in range(max(3, min(steps, 20))):
                flush.zero_()
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                lb.train_forward(TL, x, ws=ws)
                lb.train_backward(TL, x, dy, ws=ws, saved=True)
                e1.record()
                torch.cuda.synchronize(dev)
                ts.append(e0.elapsed_time(e1))
            ms = statistics.median(ts)
            flops = 2 * (2 * T * r * (d_in + d_out) + 2 * T * r * (3 * d_in + 2 * d_out))
            if lb.poll_error(ws) != lb.LB_OK:
                raise RuntimeError("QAT step reported an error")
            line = {"config": 8, "case": name, "op": "qat_step", "tokens": T, "ms": ms,
                    "backward": "reuses the forward's workspace state",
                    "tflops": flops / ms / 1e9,
                    "roofline": {"bound": "tensor", "achieved": flops / ms / 1e9,
                                 "peak": tf32_peak, "unit": "TFLOP/s",
                                 "frac": flops / ms / 1e9 / tf32_peak,
                                 "peak_source": "MEASURED_PEAKS.json bf16_tflops x 1.1/2.25 (TF32)"}}
            print(json.dumps(line), flush=True)
    elif args.config == 9:
        # end-to-end decoding of a Llama2-7B-shaped decoder whose linears are
        # LittleBit (the paper's tokens-per-second setting, shape only): 128
        # and 256 new tokens from an empty cache, one decode step per token
        # replayed as a CUDA graph (inputs resident; the step's 162 launches
        # are the per-token critical path)
        S = inputs.DECODER_7B
        for n_new in (128, 256):
            name = f"llama2-7b-shape {n_new} new tokens"
            if not wanted(name, n_new):
                continue
            layers, xs = inputs.decoder7b(n_new)
            dec = lb.DeviceDecoder(layers, S["n_heads"], S["n_kv_heads"], S["head_dim"], n_new,
                                   10000.0, dev)
            xt = lb.bf16_tensor(xs, dev)
            x_static = torch.empty(S["d_model"], dtype=torch.bfloat16, device=dev)
            out = torch.empty(S["d_model"], dtype=torch.float32, device=dev)
            x_static.copy_(xt[0])
            dec.step(x_static, out)  # warm-up outside the capture
            torch.cuda.synchronize(dev)
            cs = torch.cuda.Stream(device=dev)
            with torch.cuda.stream(cs):
                graph = torch.cuda.CUDAGraph()
                with torch.cuda.graph(graph, stream=cs):
                    dec.step(x_static, out, stream=cs)
            runs = []
            for _ in range(2):
                dec.pos.zero_()
                dec.kcache.zero_()
                dec.vcache.zero_()
                torch.cuda.synchronize(dev)
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                for t in range(n_new):
                    x_static.copy_(xt[t])
                    graph.replay()
                e1.record()
                torch.cuda.synchronize(dev)
                runs.append(e0.elapsed_time(e1))
            if dec.poll_error() != lb.LB_OK or int(dec.pos.item()) != n_new:
                raise RuntimeError("decoder reported an error")
            ms = min(runs)
            # bytes per run: every linear's words and scales per token, plus the
            # cache rows read (positions 0..p-1 of keys and values, fp32) and written
            wbytes = dec.nbytes * n_new
            cache = 4 * 2 * S["n_layers"] * S["d_kv"] * (n_new * (n_new - 1) // 2 + n_new)
            gbs = (wbytes + cache) / ms / 1e6
            line = {"config": 9, "case": name, "op": "decode", "tokens": n_new, "ms": ms,
                    "tokens_per_s": n_new / ms * 1e3, "ms_per_token": ms / n_new,
                    "bytes_per_token": (wbytes + cache) / n_new, "gbs": gbs,
                    # per layer q/k/v (grouped, the residual add and norm
                    # folded in), attention, o, gate/up (likewise), down
                    # (SiLU read inside); plus the first norm and the last add
                    "launches_per_token": 2 + 5 * S["n_layers"],
                    "roofline": {"bound": "hbm", "achieved": gbs, "peak": hbm, "unit": "GB/s",
                                 "frac": gbs / hbm, "peak_source": "MEASURED_PEAKS.json hbm_gbs"},
                    "context": "paper Table 12 (A100, Llama2-7B, 0.1 BPW, 128 new tokens): 203.20 "
                               "tokens/s; other hardware and a trained model"}
            print(json.dumps(line), flush=True)
            del dec, graph
    elif args.config == 10:
        # the exchange floor: per layer the four all-reduces on the stack's
        # critical path (t of v + the mean square; o; gate, up + the mean
        # square; down), 80 layers, nothing between them
        s70 = inputs.STACK_70B
        sizes = [2 * s70["r_kv"] + 1, 2 * s70["r_qo"], 4 * s70["r_mlp"] + 1, 2 * s70["r_mlp"]]
        rounds = 4 * s70["n_layers"]
        for words, cluster in ((1, 1), (1, 2), (2, 1), (2, 2)):
            ws = lb.selftest_exchange(rounds, sizes, cluster, words, device=dev)
            torch.cuda.synchronize(dev)
            times = []
            for _ in range(max(3, args.warmup) + steps):
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record()
                lb.selftest_exchange(rounds, sizes, cluster, words, ws=ws, device=dev)
                e1.record()
                torch.cuda.synchronize(dev)
                times.append(e0.elapsed_time(e1))
            if lb.poll_error(ws) != lb.LB_OK:
                raise RuntimeError("exchange diagnostic reported an error")
            ms = statistics.median(times[max(3, args.warmup):])
            print(json.dumps({"config": 10, "case": "exchange floor", "cluster": cluster,
                              "words_per_element": words,
                              "sizes": sizes, "rounds": rounds, "ms_per_token": ms,
                              "us_per_exchange": 1e3 * ms / rounds,
                              "us_per_layer": 4e3 * ms / rounds,
                              "note": "launch included; one cooperative launch per token"}),
                  flush=True)
    elif args.config == 6:
        # latent states (KV cache compression): the 70B key projection's latent
        # for one new token and the expansion of a 4096-token latent cache
        # (CUDA-core stages), and the 4096 x 4096 r512 halves at 2048 tokens
        # (tensor cores)
        rng = inputs.rng_for(6)
        kproj = inputs.make_linear(rng, 8192, 1024, [32, 32], 2, 0.02)
        cases = [("kv 8192->1024 r32", kproj, 1, "latent", False),
                 ("kv 8192->1024 r32", kproj, 4096, "expand", False)]
        L4, x4 = inputs.config4("4096x4096_r512", 2048)
        cases += [("4096x4096_r512", L4, 2048, "latent", True),
                  ("4096x4096_r512", L4, 2048, "expand", True)]
        for name, L, T, op, fl in cases:
            if not wanted(f"{name} {op}", T):
                continue
            x = x4 if T == 2048 else inputs.bf16_normal(rng, (T, L["d_in"]))
            emit(name, 6, T, L, time_case(L, x, T, True, op), fl, op)
    else:
        for shape in inputs.PREFILL_SHAPES:
            for T in (2048, 8192):
                if wanted(shape, T):
                    L, x = inputs.config4(shape, T)
                    emit(shape, 4, T, L, time_case(L, x, T, True), True)


def main():
    args = parse_args()
    if args.impl == "reference":
        run_reference(args)
    elif args.config is not None:
        run_config(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
