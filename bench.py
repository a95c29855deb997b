"""Benchmark: streaming frame-chunk attention (3D RoPE + KV append/evict + chunk
attention) on GB300, one JSON line on rank 0.

A step is one frame chunk through the whole path (frt_chunk_step: RoPE-K fused into
the append, RoPE-Q fused into the attention prologue) at steady state (full window).
The default workload is the largest single-GPU one, stream720p (40 heads x 128, 45x80
latent grid, 3 frames per chunk: Nq 10800, window 6 chunks: Nkv 64800). Workloads
streamed past their window (dit14b: 20 chunks) add a per-chunk leg: every chunk of a
fresh stream timed on its own.
value = attention FLOPs of all ranks' steps / max-over-ranks wall time of the timed
steps (CUDA events); ms_per_step = ms per frame chunk.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
                    [--impl reference]

--impl reference times the fp64 CPU oracle on the host cores (a bounded row
sample of the same workload per step). N > 1 runs under torchrun: one stream per
rank, independent work (weak scaling), no data-path collective.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "chunk-attention TFLOP/s and ms per frame-chunk at 1 GB300; % of bf16 peak"
UNIT = "TFLOP/s"
POOL = 8  # distinct chunk inputs cycled through (larger than L2 for the 1.3B shape)
CPU_HEADS = 12  # heads of the CPU-baseline sample (the whole 1.3B shape)


def describe(wl) -> str:
    return (f"{wl.name}: {wl.streams} stream(s), {wl.heads} heads x {wl.head_dim}, "
            f"{wl.grid_h}x{wl.grid_w} latent grid, {wl.frames} frames/chunk (Nq {wl.n_q}), "
            f"window {wl.window} chunks (Nkv {wl.window * wl.n_q} at steady state)")


def describe_conv(cw) -> str:
    return (f"{cw.name}: Cin {cw.cin}, Cout {cw.cout}, kernel {cw.kt}x{cw.kh}x{cw.kw} "
            f"(causal in time, cache of {cw.kt - 1} frames), {cw.grid_h}x{cw.grid_w} pixels, "
            f"{cw.frames} frames/chunk")


def load_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["bf16_tflops"]), float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 1900.0, 6800.0, "fallback"


def sustained_tf():
    """The measured sustained bf16 rate (a GEMM loop held for seconds under the power
    cap), or None."""
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return float(json.load(f)["bf16_tflops_sustained"])
    except Exception:
        return None


def of_sustained(achieved: float):
    sus = sustained_tf()
    return round(achieved / sus, 4) if sus else None


KERNEL_HEADERS = ("frt_ptx.cuh", "frt_internal.h")


def kernel_sources_sha(kernel_file: str) -> str:
    """sha256 over the kernel's .cu file and the headers it includes, in that order."""
    h = hashlib.sha256()
    for name in (kernel_file, *KERNEL_HEADERS):
        with open(os.path.join(ROOT, "paper_2607_18171_gb300", "csrc", name), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def traffic_record(kernel_file: str, workload: str):
    """DRAM bytes per launch from a committed ncu summary, only if the kernel's sources
    are unchanged since the capture (their sha256, recorded with the counters)."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        rec = json.load(open(path)).get(workload)
        if rec and rec.get("sources_sha256") == kernel_sources_sha(kernel_file):
            return rec.get("dram_bytes_per_launch")
    except Exception:
        pass
    return None


class ClockSampler:
    """nvidia-smi samples during the timed region (clocks, throttle reasons)."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.proc = None
        self.gpu = gpu_index

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-i", str(self.gpu), "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        self.lines = []
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except Exception:
                self.proc.kill()
                out = ""
            self.lines = [l for l in out.splitlines() if l.strip()]
        return False

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in getattr(self, "lines", []):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for n, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "samples": len(sm), "reasons": sorted(reasons)}


def clocks_of(clk, step, local, first):
    """The timed region's clock samples, or, when it was shorter than the sampling
    interval, samples of the same step run back to back for 0.4 s right after it
    (labelled as such; the timed numbers are not taken from that run)."""
    summ = clk.summary()
    if summ["samples"] > 0:
        return summ
    import torch
    torch.cuda.synchronize()
    i = first
    with ClockSampler(local) as probe:
        t = time.perf_counter()
        while time.perf_counter() - t < 0.4:
            for _ in range(20):
                step(i)
                i += 1
            torch.cuda.synchronize()
    summ = probe.summary()
    summ["probe"] = ("the same step run back to back for 0.4 s right after the timed region, "
                     "which is shorter than the sampling interval")
    return summ


def timing_events(n, stream):
    """n (start, stop) CUDA event pairs, recorded once so that the driver-level events
    exist before their handles are handed to the library."""
    import torch
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(n)]
    for a, b in evs:
        a.record(stream)
        b.record(stream)
    torch.cuda.synchronize()
    return evs


def init_dist():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def max_over_ranks(x: float, world: int, device) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------------------
def run_gpu(args, wl, world, rank, local):
    import torch
    from paper_2607_18171_gb300 import frt, synth

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    frt.lib()
    stream = torch.cuda.current_stream()
    peak_tf, peak_gbs, peak_kind = load_peaks()

    if wl.streams > 1:
        return run_gpu_multi(args, wl, world, rank, local, dev, peak_tf, peak_kind)
    if wl.steps > 1:
        return run_gpu_steps(args, wl, world, rank, local, dev, peak_tf, peak_kind)
    if wl.block:
        return run_gpu_block(args, wl, world, rank, local, dev, peak_tf, peak_kind)

    sid = rank  # each rank streams its own independent video (weak scaling)
    st = frt.Stream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                    split=wl.split)
    # prefill to a full window (untimed)
    for c in range(wl.window - 1):
        q, k, v = (t.to(dev) for t in synth.chunk_qkv(wl, sid, c))
        st.chunk_step(q, k, v, st.new_out())
    pool = [tuple(t.to(dev) for t in synth.chunk_qkv(wl, sid, wl.window - 1 + i))
            for i in range(POOL)]
    outs = [st.new_out() for _ in range(2)]
    st.sync()
    flops = wl.attn_flops(wl.window - 1)  # full window from here on

    def step(i):
        q, k, v = pool[i % POOL]
        st.chunk_step(q, k, v, outs[i % 2])

    for i in range(args.warmup):
        step(i)
    st.sync()
    n = args.steps
    ev_a = timing_events(n, stream)
    ev_k = timing_events(n, stream)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0.record(stream)
        for i in range(n):
            st.set_attention_events(*ev_a[i])
            st.set_append_events(*ev_k[i])
            step(args.warmup + i)
        t1.record(stream)
        torch.cuda.synchronize()
    st.set_attention_events(None, None)
    st.set_append_events(None, None)
    st.sync()
    if world > 1:
        torch.distributed.barrier()
    elapsed_ms = t0.elapsed_time(t1)
    attn_ms = [a.elapsed_time(b) for a, b in ev_a]
    app_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_k)
    app_bytes = 2 * 2 * wl.n_q * wl.heads * wl.head_dim * 2   # read + write of K and V
    wall_ms = max_over_ranks(elapsed_ms, world, dev)
    total_flops = flops * n * world
    value = total_flops / (wall_ms * 1e-3) / 1e12
    attn_mean = statistics.mean(attn_ms)
    achieved = flops / (attn_mean * 1e-3) / 1e12

    # e2e through the host-buffer entry point: H2D of q,k,v + step + D2H of out
    n_e2e = max(50, min(n, 200))
    hq, hk, hv = (t.pin_memory() for t in synth.chunk_qkv(wl, sid, 1000))
    hout = torch.empty(st.shape(), dtype=torch.float32).pin_memory()
    for _ in range(2):
        st.chunk_step_host(hq, hk, hv, hout)
    st.sync()
    # wall clock from a synchronised start to frt_stream_sync, which waits for the
    # compute stream and both internal copy streams: every copy is inside the region
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk_e2e:
        w0 = time.perf_counter()
        for _ in range(n_e2e):
            st.chunk_step_host(hq, hk, hv, hout)
        st.sync()
        e2e_ms = max_over_ranks((time.perf_counter() - w0) * 1e3, world, dev)
    e2e_value = flops * n_e2e * world / (e2e_ms * 1e-3) / 1e12
    per_chunk = per_chunk_leg(st, wl, sid, dev, stream, local) if wl.chunks > wl.window else None
    st.close()
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return None

    traffic = traffic_record("frt_attention.cu", wl.name)
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
        "steps": n, "warmup": args.warmup, "ms_per_step": round(wall_ms / n, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) bf16 Q/K/V shaped like the video-DiT workload)",
        "config": {"workload": describe(wl), "path": "frt_chunk_step (RoPE-K in append, "
                   "RoPE-Q in attention prologue)", "parallelism": f"independent streams x{world}",
                   "l2": f"inputs larger than L2: {POOL} distinct chunk inputs "
                   f"({POOL * 3 * wl.n_q * wl.heads * wl.head_dim * 2 / 1e6:.0f} MB) cycled, "
                   f"KV cache {2 * wl.window * wl.n_q * wl.heads * wl.head_dim * 2 / 1e6:.0f} MB",
                   "attn_flops_per_step": flops},
        "roofline": {"bound": "tensor", "achieved": round(achieved, 2), "peak": peak_tf,
                     "unit": "TFLOP/s", "frac": round(achieved / peak_tf, 4),
                     "frac_of_sustained": of_sustained(achieved),
                     "traffic": traffic, "kernel": "attn_kernel<128,1,true>",
                     "peak_kind": f"{peak_kind} bf16 dense burst",
                     "launch_ms": round(attn_mean, 4)},
        "append": {"bound": "hbm", "achieved": round(app_bytes / (app_ms * 1e-3) / 1e9, 1),
                   "peak": peak_gbs, "unit": "GB/s",
                   "frac": round(app_bytes / (app_ms * 1e-3) / 1e9 / peak_gbs, 4),
                   "frac_of_8tbs": round(app_bytes / (app_ms * 1e-3) / 8e12, 4),
                   "kernel": "staged_rows_kernel (KV append, RoPE-K fused)", "launch_ms": round(app_ms, 5),
                   "bytes_per_launch": app_bytes},
        "clocks": clk.summary(),
        "e2e": {"value": round(e2e_value, 2), "unit": UNIT,
                "h2d_bytes_per_step": 3 * wl.n_q * wl.heads * wl.head_dim * 2,
                "d2h_bytes_per_step": wl.n_q * wl.heads * wl.head_dim * 4,
                "steps": n_e2e, "ms_per_step": round(e2e_ms / n_e2e, 4),
                "clocks": clk_e2e.summary()},
        "gpu_launches": 2 * n,
    }
    if per_chunk is not None:
        line["per_chunk"] = per_chunk
    if not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(wl, seconds=args.cpu_seconds)
    return line


PER_CHUNK_REPS = 4


def per_chunk_leg(st, wl, sid, dev, stream, local):
    """Every chunk of a fresh stream of ``wl.chunks`` chunks (the window grows, then
    stays full while chunks are evicted): the attention launch of each chunk timed with
    CUDA events, median of PER_CHUNK_REPS runs, each on a reset stream with the same
    inputs (resident in HBM before the first run). Reported per chunk and as the mean
    over the steady state (chunks whose window is full)."""
    import torch
    inputs = [tuple(t.to(dev) for t in synth_chunk(wl, sid, c)) for c in range(wl.chunks)]
    out = st.new_out()
    evs = timing_events(wl.chunks * PER_CHUNK_REPS, stream)
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        for r in range(PER_CHUNK_REPS):
            st.reset()
            for c in range(wl.chunks):
                st.set_attention_events(*evs[r * wl.chunks + c])
                q, k, v = inputs[c]
                st.chunk_step(q, k, v, out)
            st.sync()
        torch.cuda.synchronize()
    st.set_attention_events(None, None)
    ms = [statistics.median(evs[r * wl.chunks + c][0].elapsed_time(evs[r * wl.chunks + c][1])
                            for r in range(PER_CHUNK_REPS)) for c in range(wl.chunks)]
    tf = [wl.attn_flops(c) / (m * 1e-3) / 1e12 for c, m in enumerate(ms)]
    steady = list(range(wl.window - 1, wl.chunks))
    steady_ms = statistics.mean(ms[c] for c in steady)
    steady_tf = sum(wl.attn_flops(c) for c in steady) / (sum(ms[c] for c in steady) * 1e-3) / 1e12
    return {"chunks": wl.chunks, "reps": PER_CHUNK_REPS, "statistic": "median over reps",
            "n_kv": [wl.n_kv(c) for c in range(wl.chunks)],
            "attention_ms": [round(m, 4) for m in ms], "tflops": [round(t, 1) for t in tf],
            "steady_state": {"chunks": f"{steady[0]}-{steady[-1]}", "mean_ms": round(steady_ms, 4),
                             "tflops": round(steady_tf, 1)},
            "clocks": clk.summary()}


def synth_chunk(wl, sid, c):
    from paper_2607_18171_gb300 import synth
    return synth.chunk_qkv(wl, sid, c)


def run_gpu_multi(args, wl, world, rank, local, dev, peak_tf, peak_kind):
    """Ragged multi-stream step: per stream RoPE + append, then one batched attention
    launch. Stream s keeps fill_s valid chunks (its window is fill_s), so the ragged KV
    lengths persist across steps."""
    import torch
    from paper_2607_18171_gb300 import frt, synth

    stream = torch.cuda.current_stream()
    fills = synth.stream_fills(wl)
    sts = []
    for s, fill in enumerate(fills):
        st = frt.Stream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, fill,
                        split=wl.split)
        for c in range(fill - 1):
            q, k, v = (t.to(dev) for t in synth.chunk_qkv(wl, 100 * rank + s, c))
            st.chunk_step(q, k, v, st.new_out())
        sts.append(st)
    pool = [[tuple(t.to(dev) for t in synth.chunk_qkv(wl, 100 * rank + s, 50 + i))
             for s in range(wl.streams)] for i in range(2)]
    work = [[tuple(x.clone() for x in pool[i][s]) for s in range(wl.streams)] for i in range(2)]
    outs = [st.new_out() for st in sts]
    flops = sum(4 * wl.n_q * f * wl.n_q * wl.head_dim * wl.heads for f in fills)

    def step(i):
        w = work[i % 2]
        for s, st in enumerate(sts):
            q, k, v = w[s]
            st.rope3d_qk(q, k)
            st.kv_append_evict(k, v)
        frt.chunk_attention_batched(sts, [w[s][0] for s in range(wl.streams)], outs)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    n = args.steps
    ev_a = timing_events(n, stream)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0.record(stream)
        for i in range(n):
            sts[0].set_attention_events(*ev_a[i])
            step(args.warmup + i)
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed = max_over_ranks(t0.elapsed_time(t1), world, dev)
    attn_mean = statistics.mean(a.elapsed_time(b) for a, b in ev_a)
    for st in sts:
        st.close()
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return None
    achieved = flops / (attn_mean * 1e-3) / 1e12
    return {
        "metric": METRIC, "value": round(flops * n * world / (elapsed * 1e-3) / 1e12, 2),
        "unit": UNIT, "n_gpus": world, "steps": n, "warmup": args.warmup,
        "ms_per_step": round(elapsed / n, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": describe(wl) + f", fills {fills} (window = fill per stream)",
                   "note": "step re-rotates the same two input sets in place; timing only"},
        "roofline": {"bound": "tensor", "achieved": round(achieved, 2), "peak": peak_tf,
                     "unit": "TFLOP/s", "frac": round(achieved / peak_tf, 4),
                     "frac_of_sustained": of_sustained(achieved), "traffic": None,
                     "kernel": "attn_kernel<128,32,false>", "peak_kind": peak_kind,
                     "launch_ms": round(attn_mean, 4)},
        "clocks": clk.summary(),
        "gpu_launches": (2 * wl.streams + 1) * n,
    }


def run_gpu_steps(args, wl, world, rank, local, dev, peak_tf, peak_kind):
    """Per-denoising-step caches: every tick advances all wl.steps steps by one chunk
    (RoPE + append per step) and runs one batched attention over them, at steady
    state (full windows)."""
    import torch
    from paper_2607_18171_gb300 import frt, synth

    stream = torch.cuda.current_stream()
    grp = frt.Steps(wl.steps, wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames,
                    wl.window, split=wl.split)
    sets = [[tuple(t.to(dev) for t in synth.chunk_qkv(wl, 100 * rank + i, 50 + r))
             for i in range(wl.steps)] for r in range(2)]
    outs = {i: torch.empty(grp.shape(), dtype=torch.float32, device=dev)
            for i in range(wl.steps)}
    act = list(range(wl.steps))

    def tick(t):
        w = sets[t % 2]
        grp.tick(act, {i: w[i][0] for i in act}, {i: w[i][1] for i in act},
                 {i: w[i][2] for i in act}, outs)

    for t in range(wl.window - 1 + args.warmup):   # fill every window, then warm up
        tick(t)
    torch.cuda.synchronize()
    n = args.steps
    flops = wl.steps * wl.attn_flops(wl.window - 1)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0.record(stream)
        for t in range(n):
            tick(t)
        t1.record(stream)
        torch.cuda.synchronize()
    elapsed = max_over_ranks(t0.elapsed_time(t1), world, dev)
    grp.close()
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return None
    return {
        "metric": METRIC, "value": round(flops * n * world / (elapsed * 1e-3) / 1e12, 2),
        "unit": UNIT, "n_gpus": world, "steps": n, "warmup": args.warmup,
        "ms_per_step": round(elapsed / n, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": describe(wl) + f", {wl.steps} denoising steps (own caches), "
                   "one pipeline tick per step: RoPE + append per step, one batched attention",
                   "note": "each tick re-rotates the same two input sets in place; timing only"},
        "clocks": clk.summary(),
        "gpu_launches": (2 * wl.steps + 1) * n,
    }


CONV_METRIC = ("streaming causal 3D convolution (VAE-decoder layer) TFLOP/s per frame-chunk "
               "at 1 GB300")


def run_gpu_conv(args, cw, world, rank, local):
    """One chunk through a streaming causal 3D convolution layer per step (frt_conv_step:
    the convolution on the tensor cores, then the frame-cache update), inputs cycled
    from a pool of distinct chunks."""
    import torch
    from paper_2607_18171_gb300 import frt, synth

    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    frt.lib()
    stream = torch.cuda.current_stream()
    peak_tf, _, peak_kind = load_peaks()
    st = frt.ConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w, cw.frames)
    w, b = (t.to(dev) for t in synth.conv_weights(cw))
    pool = [synth.conv_chunk(cw, rank, i).to(dev) for i in range(POOL)]
    ys = [st.new_out() for _ in range(2)]
    flops = cw.flops()

    def step(i):
        st.step(pool[i % POOL], w, b, ys[i % 2])

    for i in range(args.warmup):
        step(i)
    st.sync()
    n = args.steps
    ev = timing_events(n, stream)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0.record(stream)
        for i in range(n):
            ev[i][0].record(stream)
            step(args.warmup + i)
            ev[i][1].record(stream)
        t1.record(stream)
        torch.cuda.synchronize()
    st.sync()
    elapsed = max_over_ranks(t0.elapsed_time(t1), world, dev)
    step_ms = statistics.mean(a.elapsed_time(b_) for a, b_ in ev)
    clocks = clocks_of(clk, step, local, args.warmup + n)
    st.close()
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return None
    x_bytes = cw.frames * cw.grid_h * cw.grid_w * cw.cin * 2
    return {
        "metric": CONV_METRIC, "value": round(flops * n * world / (elapsed * 1e-3) / 1e12, 2),
        "unit": UNIT, "n_gpus": world, "steps": n, "warmup": args.warmup,
        "ms_per_step": round(elapsed / n, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) channels-last frames, N(0,1/(taps*Cin)) weights)",
        "config": {"workload": describe_conv(cw),
                   "path": "frt_conv_step (implicit GEMM on tcgen05 with the cache update fused: 1 launch)",
                   "l2": f"{POOL} distinct chunks of {x_bytes / 1e6:.1f} MB cycled",
                   "flops_per_step": flops},
        "roofline": {"bound": "tensor", "achieved": round(flops / (step_ms * 1e-3) / 1e12, 2),
                     "peak": peak_tf, "unit": "TFLOP/s",
                     "frac": round(flops / (step_ms * 1e-3) / 1e12 / peak_tf, 4), "traffic": None,
                     "kernel": "conv_kernel (cache update fused)", "peak_kind": peak_kind,
                     "launch_ms": round(step_ms, 4)},
        "clocks": clocks,
        "gpu_launches": n,
    }


BLOCK_METRIC = ("DiT-block attention-slice TFLOP/s (QKV projection + RoPE + KV append + "
                "chunk attention + output projection) per frame-chunk at 1 GB300")


def gemm_label(M, N, qkv, d, what):
    """Name of the projection kernel instance the library picks for C [M, N]."""
    from paper_2607_18171_gb300 import frt

    bn, ctas = frt.gemm_plan(M, N, qkv, d)
    return f"gemm_kernel<{bn}, {'pair' if ctas == 2 else 'single'}> ({what})"


def run_gpu_block(args, wl, world, rank, local, dev, peak_tf, peak_kind):
    """One DiT block's attention slice per step (frt_block_step: QKV projection with
    RoPE and the append in its epilogue, chunk attention, output projection) at steady
    state (full window), hidden states cycled from a pool larger than L2."""
    import torch
    from paper_2607_18171_gb300 import frt, synth

    stream = torch.cuda.current_stream()
    sid = rank
    d = wl.heads * wl.head_dim
    st = frt.Stream(wl.heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                    split=wl.split)
    w_qkv, w_o = (t.to(dev) for t in synth.block_weights(wl))
    q_buf = torch.empty(wl.n_q, d, dtype=torch.bfloat16, device=dev)
    o_buf = torch.empty_like(q_buf)
    ys = [torch.empty(wl.n_q, d, dtype=torch.float32, device=dev) for _ in range(2)]
    for c in range(wl.window - 1):
        st.block_step(synth.chunk_x(wl, sid, c).to(dev), w_qkv, w_o, q_buf, o_buf, ys[0])
    pool = [synth.chunk_x(wl, sid, wl.window - 1 + i).to(dev) for i in range(POOL)]
    st.sync()
    attn_flops = wl.attn_flops(wl.window - 1)
    qkv_flops = 2 * wl.n_q * d * 3 * d
    out_flops = 2 * wl.n_q * d * d
    flops = attn_flops + qkv_flops + out_flops

    def step(i):
        st.block_step(pool[i % POOL], w_qkv, w_o, q_buf, o_buf, ys[i % 2])

    for i in range(args.warmup):
        step(i)
    st.sync()
    n = args.steps
    ev_a, ev_q, ev_o = (timing_events(n, stream) for _ in range(3))
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        t0.record(stream)
        for i in range(n):
            st.set_attention_events(*ev_a[i])
            st.set_block_events(*ev_q[i], *ev_o[i])
            step(args.warmup + i)
        t1.record(stream)
        torch.cuda.synchronize()
    st.set_attention_events(None, None)
    st.set_block_events()
    st.sync()
    elapsed = max_over_ranks(t0.elapsed_time(t1), world, dev)
    attn_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_a)
    qkv_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_q)
    out_ms = statistics.mean(a.elapsed_time(b) for a, b in ev_o)
    clocks = clocks_of(clk, step, local, args.warmup + n)
    st.close()
    if world > 1:
        torch.distributed.destroy_process_group()
    if rank != 0:
        return None

    def tf(f, ms):
        return f / (ms * 1e-3) / 1e12

    step_ms = elapsed / n
    return {
        "metric": BLOCK_METRIC, "value": round(flops * n * world / (elapsed * 1e-3) / 1e12, 2),
        "unit": UNIT, "n_gpus": world, "steps": n, "warmup": args.warmup,
        "ms_per_step": round(step_ms, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) hidden states, N(0,1/d) projection weights)",
        "config": {"workload": describe(wl) + f", d_model {d}",
                   "path": "frt_block_step (3 launches: QKV projection with RoPE + append "
                           "epilogue, chunk attention, output projection)",
                   "l2": f"{POOL} distinct hidden-state inputs cycled, KV cache "
                         f"{2 * wl.window * wl.n_q * d * 2 / 1e6:.0f} MB",
                   "flops_per_step": {"attention": attn_flops, "qkv_projection": qkv_flops,
                                      "out_projection": out_flops}},
        "roofline": {"bound": "tensor", "achieved": round(tf(attn_flops, attn_ms), 2),
                     "peak": peak_tf, "unit": "TFLOP/s",
                     "frac": round(tf(attn_flops, attn_ms) / peak_tf, 4),
                     "frac_of_sustained": of_sustained(tf(attn_flops, attn_ms)), "traffic": None,
                     "kernel": "attn_kernel<128,1,false>", "peak_kind": peak_kind,
                     "launch_ms": round(attn_ms, 4)},
        "projections": {
            "qkv": {"kernel": gemm_label(wl.n_q, 3 * d, True, d, "QKV epilogue"),
                    "launch_ms": round(qkv_ms, 4),
                    "achieved": round(tf(qkv_flops, qkv_ms), 2),
                    "frac": round(tf(qkv_flops, qkv_ms) / peak_tf, 4)},
            "out": {"kernel": gemm_label(wl.n_q, d, False, 0, "plain epilogue, fp32 out"),
                    "launch_ms": round(out_ms, 4), "achieved": round(tf(out_flops, out_ms), 2),
                    "frac": round(tf(out_flops, out_ms) / peak_tf, 4)},
            "unit": "TFLOP/s", "peak": peak_tf},
        "attention_share_of_step": round(attn_ms / step_ms, 4),
        "clocks": clocks,
        "gpu_launches": 3 * n,
    }


# ---------------------------------------------------------------------------------------
# CPU oracle (baseline and reference arm)
# ---------------------------------------------------------------------------------------
def _oracle_stream(wl, sid, heads):
    """Oracle state for the first ``heads`` heads of stream ``sid``, prefilled with the
    window's first W-1 chunks (heads are independent, so a head subset is a faithful
    sample of the computation)."""
    from oracle.frt_oracle import OracleStream
    from paper_2607_18171_gb300 import synth
    orc = OracleStream(heads, wl.head_dim, wl.grid_h, wl.grid_w, wl.frames, wl.window,
                       wl.split)
    for c in range(wl.window - 1):
        q, k, v = (synth.as_f64(t[:, :heads]) for t in synth.chunk_qkv(wl, sid, c))
        q_r, k_r = orc.rope(q, k)
        orc.append(k_r, v)
    return orc


def _oracle_step(orc, wl, sid, chunk, rows):
    """Time one oracle chunk step (RoPE, append, attention of ``rows``)."""
    from paper_2607_18171_gb300 import synth
    h = orc.heads
    q, k, v = (synth.as_f64(t[:, :h]) for t in synth.chunk_qkv(wl, sid, chunk))
    t = time.perf_counter()
    orc.step(q, k, v, rows=rows)
    return time.perf_counter() - t


def cpu_threads() -> int:
    try:
        import threadpoolctl
        info = threadpoolctl.threadpool_info()
        n = max((i.get("num_threads", 1) for i in info), default=0)
        if n:
            return int(n)
    except Exception:
        pass
    return os.cpu_count() or 1


def _rows_for(n_q, count):
    return np.linspace(0, n_q - 1, max(1, min(n_q, int(count)))).astype(np.int64)


def cpu_baseline(wl, seconds: float = 15.0):
    """The oracle as it stands, on a bounded sample: one full-window chunk step (RoPE of
    the chunk, append, exact fp64 attention) for all heads and a subset of query rows.
    TFLOP/s = attention flops of the sampled rows / step time."""
    if wl.streams > 1:
        return None
    heads = min(wl.heads, CPU_HEADS)   # heads are independent: a head subset is a sample
    orc = _oracle_stream(wl, 0, heads)
    nkv = wl.window * wl.n_q
    probe = _rows_for(wl.n_q, 64)
    dt = _oracle_step(orc, wl, 0, wl.window - 1, probe)      # window now full
    rows = _rows_for(wl.n_q, len(probe) * seconds / max(dt, 1e-3))
    dt = _oracle_step(orc, wl, 0, wl.window, rows)          # evicts chunk 0, still full
    flops = 4 * len(rows) * nkv * wl.head_dim * heads
    return {"value": round(flops / dt / 1e12, 6), "unit": UNIT, "cores": cpu_threads(),
            "kind": "oracle",
            "sample": f"one full-window chunk step of {wl.name}: RoPE of the chunk + append + "
                      f"exact fp64 attention for {len(rows)} of {wl.n_q} query rows x "
                      f"{heads} of {wl.heads} heads ({dt:.1f} s)"}


def _reference_line(args, world, metric, value, total, n, config, sample):
    return {"metric": metric, "value": round(value, 6), "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * total / n, 3), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "impl": "reference", "config": config,
            "cpu_baseline": {"value": round(value, 6), "unit": UNIT, "cores": cpu_threads(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": round(value, 6), "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def run_reference(args, wl, world, rank):
    """Reference arm: the oracle timed as it stands on the host cores, one bounded
    sample of the workload per step (one head, a row subset sized so the whole run
    fits --ref-seconds)."""
    if rank != 0:
        return None
    heads = 1
    orc = _oracle_stream(wl, 0, heads)
    nkv = wl.window * wl.n_q
    probe = _rows_for(wl.n_q, 16)
    dt = _oracle_step(orc, wl, 0, wl.window - 1, probe)
    per_step = args.ref_seconds / max(1, args.steps + args.warmup)
    rows = _rows_for(wl.n_q, len(probe) * per_step / max(dt, 1e-3))
    times = []
    for i in range(args.warmup + args.steps):
        t = _oracle_step(orc, wl, 0, wl.window + i, rows)
        if i >= args.warmup:
            times.append(t)
    total = sum(times)
    flops = 4 * len(rows) * nkv * wl.head_dim * heads
    return _reference_line(
        args, world, METRIC, flops * len(times) / total / 1e12, total, len(times),
        {"workload": describe(wl)},
        f"per step: one full-window chunk of {wl.name} (RoPE of the chunk, append, exact "
        f"fp64 attention) for {len(rows)} of {wl.n_q} query rows x {heads} of {wl.heads} heads")


def run_reference_conv(args, cw, world, rank):
    """Reference arm of a convolution workload: the oracle's streaming convolution as it
    stands, one chunk per step for a subset of the output channels (each output channel
    is computed independently of the others), sized so the run fits --ref-seconds."""
    if rank != 0:
        return None
    from oracle.frt_oracle import OracleConvStream
    from paper_2607_18171_gb300 import synth
    w, b = synth.conv_weights(cw)
    w64, b64 = synth.as_f64(w), np.asarray(b, np.float64)
    orc = OracleConvStream(cw.cin, cw.cout, cw.kt, cw.kh, cw.kw, cw.grid_h, cw.grid_w)
    probe = min(cw.cout, 32)
    t = time.perf_counter()
    orc.step(synth.as_f64(synth.conv_chunk(cw, 0, 0)), w64[:, :probe], b64[:probe])
    dt = time.perf_counter() - t
    per_step = args.ref_seconds / max(1, args.steps + args.warmup)
    n_c = max(1, min(cw.cout, int(probe * per_step / max(dt, 1e-3))))
    times = []
    for i in range(args.warmup + args.steps):
        x = synth.as_f64(synth.conv_chunk(cw, 0, 1 + i))
        t = time.perf_counter()
        orc.step(x, w64[:, :n_c], b64[:n_c])
        if i >= args.warmup:
            times.append(time.perf_counter() - t)
    total = sum(times)
    flops = 2 * cw.frames * cw.grid_h * cw.grid_w * n_c * cw.taps * cw.cin
    return _reference_line(
        args, world, CONV_METRIC, flops * len(times) / total / 1e12, total, len(times),
        {"workload": describe_conv(cw)},
        f"per step: one chunk of {cw.name} through the oracle's streaming convolution for "
        f"{n_c} of {cw.cout} output channels")


def run_reference_block(args, wl, world, rank):
    """Reference arm of the DiT-block slice: the oracle's pieces as they stand (linear,
    the chunk step, linear) on one head's share of the block per step — that head's q, k,
    v projection columns for every token (the cache needs k and v of every token), RoPE,
    append and attention for a subset of query rows, and that head's share of the output
    projection for those rows. Heads are independent up to the output projection, whose
    head shares add up."""
    if rank != 0:
        return None
    from oracle.frt_oracle import OracleStream, bf16_round, linear
    from paper_2607_18171_gb300 import synth
    d, D = wl.heads * wl.head_dim, wl.head_dim
    w_qkv, w_o = (synth.as_f64(t) for t in synth.block_weights(wl))
    w_h = np.concatenate([w_qkv[i * d:i * d + D] for i in range(3)])   # head 0's rows
    w_oh = w_o[:, :D]
    orc = OracleStream(1, D, wl.grid_h, wl.grid_w, wl.frames, wl.window, wl.split)

    def step(chunk, rows):
        x = synth.as_f64(synth.chunk_x(wl, 0, chunk))
        t = time.perf_counter()
        qkv = bf16_round(linear(x, w_h))
        q, k, v = (qkv[:, i * D:(i + 1) * D].reshape(wl.n_q, 1, D) for i in range(3))
        o, _, _ = orc.step(q, k, v, rows=rows)
        linear(bf16_round(o).reshape(len(rows), D), w_oh)
        return time.perf_counter() - t

    probe = _rows_for(wl.n_q, 16)
    for c in range(wl.window - 1):
        dt = step(c, probe)
    per_step = args.ref_seconds / max(1, args.steps + args.warmup)
    rows = _rows_for(wl.n_q, len(probe) * per_step / max(dt, 1e-3))
    times = []
    for i in range(args.warmup + args.steps):
        t = step(wl.window - 1 + i, rows)
        if i >= args.warmup:
            times.append(t)
    total = sum(times)
    nkv = wl.window * wl.n_q
    flops = 2 * wl.n_q * d * 3 * D + 4 * len(rows) * nkv * D + 2 * len(rows) * D * d
    return _reference_line(
        args, world, BLOCK_METRIC, flops * len(times) / total / 1e12, total, len(times),
        {"workload": describe(wl) + f", d_model {d}"},
        f"per step: one full-window chunk of {wl.name}, head 0 of {wl.heads}: its q/k/v "
        f"projection for all {wl.n_q} tokens, RoPE, append, exact fp64 attention and its "
        f"output-projection share for {len(rows)} query rows")


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=60)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--workload", default="stream720p")
    ap.add_argument("--impl", default="frt", choices=["frt", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=15.0)
    ap.add_argument("--ref-seconds", type=float, default=90.0)
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    from paper_2607_18171_gb300 import synth
    world, rank, local = init_dist()
    if args.workload in synth.CONV_WORKLOADS:
        cw = synth.CONV_WORKLOADS[args.workload]
        line = (run_reference_conv(args, cw, world, rank) if args.impl == "reference"
                else run_gpu_conv(args, cw, world, rank, local))
        if line is not None:
            print(json.dumps(line), flush=True)
        return
    wl = synth.WORKLOADS[args.workload]
    if args.impl == "reference":
        line = (run_reference_block(args, wl, world, rank) if wl.block
                else run_reference(args, wl, world, rank))
    else:
        line = run_gpu(args, wl, world, rank, local)
    if line is not None:
        print(json.dumps(line), flush=True)


if __name__ == "__main__":
    main()
