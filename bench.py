#!/usr/bin/env python
"""Benchmark of the block-causal attention hot path on GB300.

One step = block-causal attention forward + backward (every stage of the
training path) over the workload B=2, H=12, d=64, 16 chunks x 880 tokens
(N = 14080), bf16, synthetic N(0,1) inputs.  `value` is TFLOP/s counted over
unmasked (query, key) pairs only: fwd 4*d*pairs + bwd 10*d*pairs.

Also reported in the same JSON line: the fractions of the measured bf16
peak (burst and sustained), the median and minimum step time, the roofline
of the dominant kernel (backward key-tile kernel, timed with CUDA events
around it, with its ncu DRAM traffic while the sources match the profiled
build), an end-to-end number through the C ABI with pinned host buffers,
SM clocks sampled during the timed region, the fp64 oracle on the host
cores (cpu_baseline), and secondary workloads (the d=128 peaky config, the
paper's 32 x 600 window, the d=72 layout, the rolling-KV-cache streaming
step, the pipelined 4-chunk window, the sink anchor with and without the
RoPE re-shift, and the QKV-RoPE split).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
    python bench.py --extras-only rolling_cache[,pipelined,...]   # profiling

Under torchrun (N > 1) every rank runs its own batch of the same workload
(independent problems: weak scaling, no collective on the data path); the
timed region is bracketed by barriers and the max over ranks is taken.
"""
from __future__ import annotations

import argparse
import csv
import datetime
import io
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

from workloads import CACHE_CONFIGS, TRAIN_CONFIGS, gen_cache, gen_train  # noqa: E402

METRIC = "block-causal attn TFLOP/s fwd+bwd (% GB300 BF16 peak); rolling-KV chunk latency µs"
WORKLOAD = "train_b12_d64"
L2_FLUSH_BYTES = 256 << 20
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ------------------------------------------------------------------ accounting

def train_pairs(cfg) -> int:
    """Unmasked (query, key) pairs: T^2 n (n+1) / 2 per head."""
    return cfg.B * cfg.H * cfg.T * cfg.T * cfg.n_chunks * (cfg.n_chunks + 1) // 2


def cache_pairs(cfg) -> int:
    """Each of the W*T queries sees the sink anchor and `length` cached keys
    plus its causal share of the in-flight keys."""
    inflight = cfg.T * cfg.T * cfg.W * (cfg.W + 1) // 2
    return cfg.B * cfg.H * (cfg.W * cfg.T * (cfg.sink + cfg.length) + inflight)


def fwd_flops(pairs: int, d: int) -> float:
    return 4.0 * d * pairs


def bwd_flops(pairs: int, d: int) -> float:
    return 10.0 * d * pairs


def bwd_main_bytes(cfg) -> float:
    """Algorithmic bytes of the backward key-tile kernel: read Q, K, V, dO
    (bf16) and the two fp32 row vectors; write dK, dV (bf16); one fp32
    read-modify-write of the dQ accumulator."""
    e = cfg.B * cfg.H * cfg.N * cfg.d
    rows = cfg.B * cfg.H * cfg.N
    return 2.0 * 4 * e + 4.0 * 2 * rows + 2.0 * 2 * e + 8.0 * e


def cache_bytes(cfg) -> float:
    """Read the cached K/V (sink anchor and ring) once, the in-flight Q/K/V,
    write O and LSE, and the commit (read + write of one chunk's K and V)."""
    e_new = cfg.B * cfg.H * cfg.W * cfg.T * cfg.d
    e_ring = cfg.B * cfg.H * (cfg.sink + cfg.length) * cfg.d
    commit = 2.0 * 2 * 2 * cfg.B * cfg.H * cfg.T * cfg.d
    return 2.0 * 2 * e_ring + 2.0 * 3 * e_new + 2.0 * e_new + 4.0 * cfg.B * cfg.H * cfg.W * cfg.T + commit


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p["bf16_tflops"]),
                "bf16_tflops_sustained": float(p.get("bf16_tflops_sustained", p["bf16_tflops"])),
                "source": "measured"}
    except (OSError, KeyError, ValueError):
        return {**FALLBACK_PEAKS, "source": "fallback"}


# ------------------------------------------------------------------ distributed helpers

def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def init_dist(world: int, backend: str):
    if world > 1 and not torch.distributed.is_initialized():
        torch.distributed.init_process_group(backend=backend)


def barrier(world: int):
    if world > 1:
        torch.distributed.barrier()


def max_over_ranks(x: float, world: int, device=None) -> float:
    if world == 1:
        return x
    t = torch.tensor([x], dtype=torch.float64, device=device)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def aggregate_rate(units_per_rank: float, world: int, seconds_max: float) -> float:
    """Whole-job throughput: units processed by all ranks / slowest rank's time."""
    return units_per_rank * world / seconds_max


# ------------------------------------------------------------------ clocks

CLOCK_FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
                "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
                "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")


class ClockSampler:
    """nvidia-smi sampling every 20 ms; the summary keeps the samples taken
    between mark_start() and mark_end() (the timed region)."""

    def __init__(self, gpu_index: int):
        self.gpu_index = gpu_index
        self.proc = None
        self.t0 = self.t1 = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu_index), f"--query-gpu={CLOCK_FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            time.sleep(0.5)  # nvidia-smi is sampling before the timed region starts
        except OSError:
            self.proc = None
        return self

    def mark_start(self):
        self.t0 = datetime.datetime.now()

    def mark_end(self):
        self.t1 = datetime.datetime.now()

    def __exit__(self, *exc):
        self.text = ""
        if self.proc is not None:
            time.sleep(0.1)
            self.proc.terminate()
            try:
                self.text, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
                self.text = ""
        return False

    def summary(self):
        rows = []
        for r in csv.reader(io.StringIO(getattr(self, "text", ""))):
            if len(r) < 10:
                continue
            ts = None
            for fmt in ("%Y/%m/%d %H:%M:%S.%f", "%Y/%m/%d %H:%M:%S"):
                try:
                    ts = datetime.datetime.strptime(r[0].strip(), fmt)
                    break
                except ValueError:
                    pass
            if ts is None:
                continue
            rows.append((ts, r[1:]))
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        inside = [r for ts, r in rows if self.t0 is not None and self.t1 is not None
                  and self.t0 <= ts <= self.t1]
        window = "timed region"
        if not inside:  # region shorter than the sampling period
            inside = [r for _, r in rows]
            window = "whole run (no sample fell inside the timed region)"
        num = lambda v: v.strip().replace(".", "").isdigit()
        sm = [float(r[1]) for r in inside if num(r[1])]
        mx = [float(r[2]) for r in inside if num(r[2])]
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        reasons = sorted({n for r in inside for n, v in zip(names, r[5:9]) if "Active" == v.strip()})
        power = [float(r[3]) for r in inside if num(r[3])]
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(inside), "window": window,
                "power_w_max": max(power) if power else None}


# ------------------------------------------------------------------ CPU baseline (oracle)

def oracle_sample(seconds: float, rank_seed: int = 0, max_heads: int = 24):
    """fp64 oracle fwd+bwd over whole (b, h) heads of the workload until
    `seconds` have passed (at least one head).  Returns (TFLOP/s, heads, s)."""
    import oracle
    cfg = TRAIN_CONFIGS[WORKLOAD]
    x = gen_train(cfg)
    per_head = (fwd_flops(train_pairs(cfg), cfg.d) + bwd_flops(train_pairs(cfg), cfg.d)) / (cfg.B * cfg.H)
    t0 = time.perf_counter()
    heads = 0
    for idx in range(max_heads):
        b, h = divmod(idx % (cfg.B * cfg.H), cfg.H)
        sl = (slice(b, b + 1), slice(h, h + 1))
        q, k, v, do = (x[n][sl] for n in ("q", "k", "v", "do"))
        oracle.fwd(q, k, v, cfg.T, cfg.scale)
        oracle.bwd(q, k, v, do, cfg.T, cfg.scale)
        heads += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    return per_head * heads / dt / 1e12, heads, dt


def oracle_config_baselines(seconds: float = 5.0):
    """The fp64 oracle, as it stands, on the host cores for the other
    workloads: whole (b, h) heads until about `seconds` have passed (at least
    one), scaled to the metric of each (TFLOP/s for training fwd+bwd; for the
    cache workloads the time of one full call, all heads, in microseconds)."""
    import oracle
    res = {}
    cfg = TRAIN_CONFIGS["train_h16_d128_peaky"]
    x = gen_train(cfg)
    per_head = (fwd_flops(train_pairs(cfg), cfg.d) + bwd_flops(train_pairs(cfg), cfg.d)) / (cfg.B * cfg.H)
    t0, heads = time.perf_counter(), 0
    while heads < cfg.B * cfg.H:
        b, h = divmod(heads, cfg.H)
        sl = (slice(b, b + 1), slice(h, h + 1))
        q, k, v, do = (x[n][sl] for n in ("q", "k", "v", "do"))
        oracle.fwd(q, k, v, cfg.T, cfg.scale)
        oracle.bwd(q, k, v, do, cfg.T, cfg.scale)
        heads += 1
        if time.perf_counter() - t0 >= seconds:
            break
    dt = time.perf_counter() - t0
    res["train_h16_d128_peaky"] = {
        "value": round(per_head * heads / dt / 1e12, 6), "unit": "TFLOP/s (fwd+bwd)",
        "cores": torch.get_num_threads(), "kind": "oracle",
        "sample": f"fp64 oracle fwd+bwd of {heads} of {cfg.B * cfg.H} heads ({dt:.1f} s)"}
    for name in ("rolling_cache", "pipelined"):
        cfg = CACHE_CONFIGS[name]
        x = gen_cache(cfg, steps=1)
        q, kn, vn, kr, vr = x["q"][0], x["k_new"][0], x["v_new"][0], x["k_ring"], x["v_ring"]
        t0, heads = time.perf_counter(), 0
        while heads < cfg.B * cfg.H:
            b, h = divmod(heads, cfg.H)
            sl = (slice(b, b + 1), slice(h, h + 1))
            oracle.cache_fwd(q[sl], kn[sl], vn[sl], kr[sl], vr[sl], cfg.cap, cfg.head, cfg.length,
                             cfg.T, cfg.scale)
            heads += 1
            if time.perf_counter() - t0 >= seconds:
                break
        dt = time.perf_counter() - t0
        us = dt / heads * cfg.B * cfg.H * 1e6
        res[name] = {"value": round(us, 1), "unit": "us per call (all heads)",
                     "tflops": round(fwd_flops(cache_pairs(cfg), cfg.d) / (us / 1e6) / 1e12, 6),
                     "cores": torch.get_num_threads(), "kind": "oracle",
                     "sample": f"fp64 oracle cache forward of {heads} of {cfg.B * cfg.H} heads, "
                               f"scaled to all heads ({dt:.1f} s)"}
    return res


def cpu_cores() -> int:
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


# ------------------------------------------------------------------ GPU timing helpers

class Events:
    def __init__(self):
        self.a = torch.cuda.Event(enable_timing=True)
        self.b = torch.cuda.Event(enable_timing=True)

    def start(self):
        self.a.record()

    def stop(self):
        self.b.record()

    def ms(self) -> float:
        return self.a.elapsed_time(self.b)


def time_repeated(fn, reps: int, warmup: int = 3, flush=None):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    ts = []
    for _ in range(reps):
        if flush is not None:
            flush()
        e = Events()
        e.start()
        fn()
        e.stop()
        ts.append(e)
    torch.cuda.synchronize()
    return [e.ms() for e in ts]


# ------------------------------------------------------------------ our arm

def run_extras_only(args):
    """Named secondary workloads alone, on one GPU (for profiling their kernels)."""
    import paper_2608_01127_gb300 as mw

    names = [n.strip() for n in args.extras_only.split(",") if n.strip()]
    unknown = [n for n in names if n not in EXTRA_NAMES]
    if unknown:
        raise SystemExit(f"unknown secondary workloads: {unknown}")
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    extra = run_extras(mw, dev, load_peaks(), only=names)
    print(json.dumps({"extras_only": names, "extra": extra}), flush=True)


def run_ours(args):
    import paper_2608_01127_gb300 as mw

    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    init_dist(world, "nccl")
    peaks = load_peaks()

    workload = args.workload
    cfg = TRAIN_CONFIGS[workload]
    x = gen_train(cfg) if rank == 0 else gen_train(_reseeded(cfg, rank))
    q, k, v, do = (x[n].to(dev) for n in ("q", "k", "v", "do"))
    o = torch.empty_like(q)
    lse = torch.empty(cfg.B, cfg.H, cfg.N, dtype=torch.float32, device=dev)
    dq, dk, dv = torch.empty_like(q), torch.empty_like(k), torch.empty_like(v)
    ws = torch.empty(mw.mw_bca_bwd_workspace_size(cfg.B, cfg.H, cfg.n_chunks, cfg.T, cfg.d),
                     dtype=torch.uint8, device=dev)
    flush_buf = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    lib = mw.library()
    sc = cfg.scale

    def fwd():
        mw._check(lib.mw_bca_fwd(q.data_ptr(), k.data_ptr(), v.data_ptr(), o.data_ptr(),
                                 lse.data_ptr(), cfg.B, cfg.H, cfg.n_chunks, cfg.T, cfg.d, sc,
                                 torch.cuda.current_stream().cuda_stream))

    def bwd_stage(stage):
        mw._check(lib.mw_bca_bwd_stage(stage, q.data_ptr(), k.data_ptr(), v.data_ptr(),
                                       o.data_ptr(), lse.data_ptr(), do.data_ptr(), dq.data_ptr(),
                                       dk.data_ptr(), dv.data_ptr(), ws.data_ptr(), ws.numel(),
                                       cfg.B, cfg.H, cfg.n_chunks, cfg.T, cfg.d, sc,
                                       torch.cuda.current_stream().cuda_stream))

    launches_per_step = 4  # forward kernel + backward pre / main / post
    pairs = train_pairs(cfg)
    step_flops = fwd_flops(pairs, cfg.d) + bwd_flops(pairs, cfg.d)

    for _ in range(args.warmup):
        fwd()
        bwd_stage(0)
    torch.cuda.synchronize()
    barrier(world)
    step_ev, main_ev, fwd_ev = [], [], []
    with ClockSampler(local) as clk:
        barrier(world)
        torch.cuda.synchronize()
        clk.mark_start()
        for _ in range(args.steps):
            flush_buf.zero_()          # L2 flush between steps, outside the events
            s, f, m = Events(), Events(), Events()
            s.start()
            f.start()
            fwd()
            f.stop()
            bwd_stage(1)
            m.start()
            bwd_stage(2)
            m.stop()
            bwd_stage(3)
            s.stop()
            step_ev.append(s)
            main_ev.append(m)
            fwd_ev.append(f)
        torch.cuda.synchronize()
        clk.mark_end()
        barrier(world)
    step_ms = [e.ms() for e in step_ev]
    total_ms = max_over_ranks(sum(step_ms), world, dev)
    value = aggregate_rate(step_flops * args.steps, world, total_ms / 1e3) / 1e12
    ms_per_step = total_ms / args.steps
    main_ms = statistics.mean(e.ms() for e in main_ev)
    fwd_ms = statistics.mean(e.ms() for e in fwd_ev)
    main_flops = bwd_flops(pairs, cfg.d)
    achieved = main_flops / (main_ms / 1e3) / 1e12
    assert mw.mw_device_status() == 0, "a kernel reported a timeout"

    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "TFLOP/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": f"{workload}: block-causal attention fwd+bwd, B={cfg.B} H={cfg.H} "
                               f"d={cfg.d}, {cfg.n_chunks} chunks x {cfg.T} tokens (N={cfg.N})",
                   "global_batch": cfg.B * world, "seq_len": cfg.N, "parallelism": f"dp{world}",
                   "flops_per_step": step_flops, "unmasked_pairs": pairs,
                   "l2": "256 MiB buffer written between timed steps (outside the events)"},
        "frac_of_bf16_peak": round(value / world / peaks["bf16_tflops"], 4),
        "frac_of_bf16_sustained": round(value / world / peaks["bf16_tflops_sustained"], 4),
        "ms_per_step_median": round(statistics.median(step_ms), 4),
        "ms_per_step_min": round(min(step_ms), 4),
        "roofline": {"kernel": f"bca_bwd_kernel<{cfg.d}, {cfg.d}> (backward key-tile kernel)", "bound": "tensor",
                     "achieved": round(achieved, 2), "peak": peaks["bf16_tflops"],
                     "peak_source": peaks["source"] + " bf16 burst", "unit": "TFLOP/s",
                     "frac": round(achieved / peaks["bf16_tflops"], 4),
                     "frac_of_sustained": round(achieved / peaks["bf16_tflops_sustained"], 4),
                     "traffic": profiled_traffic(f"bca_bwd_kernel<{cfg.d},{cfg.d}>", workload),
                     "algorithmic_bytes": bwd_main_bytes(cfg),
                     "ms_per_launch": round(main_ms, 4)},
        "fwd": {"ms": round(fwd_ms, 4),
                "tflops": round(fwd_flops(pairs, cfg.d) / (fwd_ms / 1e3) / 1e12, 2)},
        "gpu_launches": launches_per_step * args.steps,
    }
    out["clocks"] = clk.summary()
    out["e2e"] = run_e2e(mw, cfg, dev, args, world, step_flops)
    if rank == 0 and world == 1 and not args.no_extras:
        out["extra"] = run_extras(mw, dev, peaks, args=args)
        if not args.no_cpu_baseline:
            out["extra"]["cpu_baseline_per_config"] = oracle_config_baselines()
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        tf, heads, dt = oracle_sample(args.cpu_seconds)
        out["cpu_baseline"] = {"value": round(tf, 6), "unit": "TFLOP/s", "cores": torch.get_num_threads(),
                               "host_cores": cpu_cores(), "kind": "oracle",
                               "sample": f"fp64 oracle fwd+bwd of {heads} of {cfg.B * cfg.H} (b,h) heads "
                                         f"of {WORKLOAD} ({dt:.1f} s)"}
    if rank == 0:
        print(json.dumps(out), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()


def _reseeded(cfg, rank):
    import dataclasses
    return dataclasses.replace(cfg, seed=cfg.seed + 1000 * rank)


def run_e2e(mw, cfg, dev, args, world, step_flops):
    """Same step through the public API with pinned host buffers: H2D of
    Q, K, V, dO and D2H of O, LSE, dQ, dK, dV inside the timed region.

    ``value`` overlaps the transfers with the compute the way a training loop
    that prefetches would: two sets of device buffers; step i+1's inputs go
    up on one copy stream while step i computes, and step i's results come
    down on another while step i+1 computes.  ``serial_ms_per_step`` is the
    same step with copy, compute and read-back in sequence on one stream."""
    x = gen_train(cfg)
    host_in = [x[n].pin_memory() for n in ("q", "k", "v", "do")]
    h2d = sum(t.numel() * t.element_size() for t in host_in)
    sets = []
    for _ in range(2):
        din = [torch.empty_like(t, device=dev) for t in host_in]
        dout = [torch.empty_like(din[0]) for _ in range(4)]             # o, dq, dk, dv
        dlse = torch.empty(cfg.B, cfg.H, cfg.N, dtype=torch.float32, device=dev)
        hout = [torch.empty_like(host_in[0]).pin_memory() for _ in range(4)]
        hlse = torch.empty(cfg.B, cfg.H, cfg.N, dtype=torch.float32).pin_memory()
        ws = torch.empty(mw.mw_bca_bwd_workspace_size(cfg.B, cfg.H, cfg.n_chunks, cfg.T, cfg.d),
                         dtype=torch.uint8, device=dev)
        sets.append((din, dout, dlse, hout, hlse, ws))
    d2h = sum(t.numel() * t.element_size() for t in sets[0][3]) + sets[0][4].numel() * 4
    comp = torch.cuda.current_stream()
    up, down = torch.cuda.Stream(), torch.cuda.Stream()

    def compute(b):
        din, dout, dlse, _, _, ws = sets[b]
        q, k, v, do = din
        o, lse = mw.mw_bca_fwd(q, k, v, cfg.T, cfg.scale, out=(dout[0], dlse))
        mw.mw_bca_bwd(q, k, v, o, lse, do, cfg.T, cfg.scale, workspace=ws,
                      out=(dout[1], dout[2], dout[3]))

    def upload(b, stream):
        with torch.cuda.stream(stream):
            for d_, h_ in zip(sets[b][0], host_in):
                d_.copy_(h_, non_blocking=True)

    def download(b, stream):
        _, dout, dlse, hout, hlse, _ = sets[b]
        with torch.cuda.stream(stream):
            for h_, d_ in zip(hout, dout):
                h_.copy_(d_, non_blocking=True)
            hlse.copy_(dlse, non_blocking=True)

    def run_pipelined(n):
        in_ready = [torch.cuda.Event() for _ in range(2)]
        done = [torch.cuda.Event() for _ in range(2)]
        out_free = [torch.cuda.Event() for _ in range(2)]
        upload(0, up)
        in_ready[0].record(up)
        for i in range(n):
            b = i % 2
            comp.wait_event(in_ready[b])
            if i >= 2:
                comp.wait_event(out_free[b])      # step i-2's results have left set b
            compute(b)
            done[b].record(comp)
            if i + 1 < n:                          # next inputs, once step i-1 freed the set
                if i >= 1:
                    up.wait_event(done[1 - b])
                upload(1 - b, up)
                in_ready[1 - b].record(up)
            down.wait_event(done[b])
            download(b, down)
            out_free[b].record(down)
        comp.wait_stream(down)

    def run_serial(n):
        for _ in range(n):
            upload(0, comp)
            compute(0)
            download(0, comp)

    # as many steps as the device-timed measurement, so the pipeline's fill
    # (the first upload) and drain (the last read-back) are spread alike
    reps = max(3, args.steps)
    run_pipelined(2)
    run_serial(1)
    torch.cuda.synchronize()
    barrier(world)
    t0 = time.perf_counter()
    e = Events()
    e.start()
    run_pipelined(reps)
    e.stop()
    torch.cuda.synchronize()
    wall = (time.perf_counter() - t0) * 1e3 / reps
    ms = max_over_ranks(e.ms(), world, dev)
    es = Events()
    es.start()
    run_serial(reps)
    es.stop()
    torch.cuda.synchronize()
    ms_serial = max_over_ranks(es.ms(), world, dev)
    return {"value": round(aggregate_rate(step_flops * reps, world, ms / 1e3) / 1e12, 2),
            "unit": "TFLOP/s", "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": round(ms / reps, 4), "wall_ms_per_step": round(wall, 4),
            "serial_ms_per_step": round(ms_serial / reps, 4),
            "overlap": "H2D of step i+1 and D2H of step i-1 run on two copy streams "
                       "during step i's compute (double-buffered device sets)"}


EXTRA_NAMES = ("train_h16_d128_peaky", "train_1b_32x600", "train_05b_d72", "rolling_cache",
               "pipelined", "sink_anchor", "qkv_rope_split")


def run_extras(mw, dev, peaks, only=None, args=None):
    """The secondary workloads (all, or the names in `only`)."""
    flush_buf = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    flush = flush_buf.zero_
    extra = {}
    want = set(EXTRA_NAMES if only is None else only)
    # forward / backward of the other training workloads: d=128 with peaky
    # logits, the paper's 32-chunk window of 600-token chunks at the
    # MiniWorld-1B head layout (12 heads of 128), and the 0.5B head dim (72,
    # run on the 128-wide kernels with zero-filled columns)
    for name in ("train_h16_d128_peaky", "train_1b_32x600", "train_05b_d72"):
        if name not in want:
            continue
        cfg = TRAIN_CONFIGS[name]
        x = gen_train(cfg)
        q, k, v, do = (x[n].to(dev) for n in ("q", "k", "v", "do"))
        o, lse = mw.mw_bca_fwd(q, k, v, cfg.T, cfg.scale)
        ws = torch.empty(mw.mw_bca_bwd_workspace_size(cfg.B, cfg.H, cfg.n_chunks, cfg.T, cfg.d),
                         dtype=torch.uint8, device=dev)
        grads = tuple(torch.empty_like(q) for _ in range(3))
        pairs = train_pairs(cfg)
        tf = time_repeated(lambda: mw.mw_bca_fwd(q, k, v, cfg.T, cfg.scale), 10, flush=flush)
        tb = time_repeated(lambda: mw.mw_bca_bwd(q, k, v, o, lse, do, cfg.T, cfg.scale,
                                                 workspace=ws, out=grads), 10, flush=flush)
        fm, bm = statistics.median(tf), statistics.median(tb)
        extra[name] = {
            "fwd_ms": round(fm, 4), "bwd_ms": round(bm, 4),
            "fwd_tflops": round(fwd_flops(pairs, cfg.d) / fm / 1e9, 2),
            "fwd_bwd_tflops": round((fwd_flops(pairs, cfg.d) + bwd_flops(pairs, cfg.d))
                                    / (fm + bm) / 1e9, 2)}
        if name == "train_h16_d128_peaky":
            # the largest training workload, reported like the headline: its
            # dominant kernel (the backward key-tile kernel, timed alone) and
            # the step end to end through the API with host buffers
            mw.mw_bca_bwd(q, k, v, o, lse, do, cfg.T, cfg.scale, workspace=ws, out=grads, stage=1)
            tm = time_repeated(lambda: mw.mw_bca_bwd(q, k, v, o, lse, do, cfg.T, cfg.scale,
                                                     workspace=ws, out=grads, stage=2), 10, flush=flush)
            mm = statistics.median(tm)
            ach = bwd_flops(pairs, cfg.d) / mm / 1e9
            extra[name]["roofline"] = {
                "kernel": f"bca_bwd_kernel<{cfg.d}, {cfg.d}> (backward key-tile kernel)",
                "bound": "tensor", "achieved": round(ach, 2), "peak": peaks["bf16_tflops"],
                "peak_source": peaks["source"] + " bf16 burst", "unit": "TFLOP/s",
                "frac": round(ach / peaks["bf16_tflops"], 4),
                "frac_of_sustained": round(ach / peaks["bf16_tflops_sustained"], 4),
                "traffic": profiled_traffic(f"bca_bwd_kernel<{cfg.d},{cfg.d}>", name),
                "algorithmic_bytes": bwd_main_bytes(cfg), "ms_per_launch": round(mm, 4),
                "share_of_step": round(mm / (fm + bm), 4)}
            if args is not None:
                extra[name]["e2e"] = run_e2e(mw, cfg, dev, args, 1,
                                             fwd_flops(pairs, cfg.d) + bwd_flops(pairs, cfg.d))
        del q, k, v, do, o, lse, ws, grads
    if "rolling_cache" in want:
        extra["rolling_cache"] = bench_rolling(mw, dev, peaks)
    if "pipelined" in want:
        extra["pipelined"] = bench_pipelined(mw, dev, peaks, flush)
    if "sink_anchor" in want:
        extra["sink_anchor"] = bench_sink(mw, dev, peaks, flush)
    if "qkv_rope_split" in want:
        extra["qkv_rope_split"] = bench_qkv_split(mw, dev, peaks, flush)
    return extra


def bench_qkv_split(mw, dev, peaks, flush):
    """The QKV split with the temporal RoPE of Q and K at the d=64 training
    layout (B2 H12, 16 x 880 tokens, 32 rotated channels, 440 tokens per
    frame): HBM-bound, every element read and written once."""
    cfg = TRAIN_CONFIGS["train_b12_d64"]
    N = cfg.n_chunks * cfg.T
    g = torch.Generator(device=dev).manual_seed(21)
    qkv = torch.randn(cfg.B, N, 3, cfg.H, cfg.d, generator=g, device=dev).to(torch.bfloat16)
    out = tuple(torch.empty(cfg.B, cfg.H, N, cfg.d, dtype=torch.bfloat16, device=dev)
                for _ in range(3))
    ts = time_repeated(lambda: mw.mw_qkv_rope_split(qkv, 32, 10000.0, 440, 0, out=out), 20,
                       flush=flush)
    med = statistics.median(ts) * 1e3
    nbytes = 2 * qkv.numel() * qkv.element_size()
    gbs = nbytes / (med / 1e6) / 1e9
    return {"us_median": round(med, 2), "l2": "flushed between runs",
            "bytes_algorithmic": nbytes, "gbs_algorithmic": round(gbs, 1),
            "frac_hbm": round(gbs / peaks["hbm_gbs"], 4), "rope_dims": 32,
            "tokens_per_frame": 440}


def _cache_roofline(cfg, us, peaks):
    flops = fwd_flops(cache_pairs(cfg), cfg.d)
    nbytes = cache_bytes(cfg)
    t_tensor = flops / (peaks["bf16_tflops"] * 1e12)
    t_hbm = nbytes / (peaks["hbm_gbs"] * 1e9)
    s = us / 1e6
    return {"tflops": round(flops / s / 1e12, 2), "frac_tensor": round(t_tensor / s, 4),
            "gbs_algorithmic": round(nbytes / s / 1e9, 1), "frac_hbm": round(t_hbm / s, 4),
            "roofline_frac": round(max(t_tensor, t_hbm) / s, 4),
            "bound": "tensor" if t_tensor >= t_hbm else "hbm"}


def bench_rolling(mw, dev, peaks):
    """64 streaming steps: cache forward of one 880-token chunk against the
    8-chunk ring, then commit of that chunk (FIFO eviction), through the
    one-call streaming step; per-step latency.  The same steps as separate
    forward and commit calls are timed beside it."""
    cfg = CACHE_CONFIGS["rolling_cache"]
    x = gen_cache(cfg)
    kr, vr = x["k_ring"].to(dev), x["v_ring"].to(dev)
    qs, ks, vs = x["q"].to(dev), x["k_new"].to(dev), x["v_new"].to(dev)
    ws_bytes = mw.mw_bca_cache_workspace_size(cfg.B, cfg.H, cfg.W, cfg.T, cfg.d, cfg.length)
    ws = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=dev)
    o = torch.empty_like(qs[0])
    plan = []
    ring = mw.RingState(cfg.cap, cfg.head, cfg.length)
    for _ in range(cfg.steps):
        head, length = ring.head, ring.length
        plan.append((head, length, ring.commit(cfg.T)))

    def step(s):
        h, ln, slot = plan[s]
        mw.mw_bca_cache_step(qs[s], ks[s], vs[s], kr, vr, h, ln, slot, cfg.T, cfg.T, cfg.scale,
                             need_lse=False, workspace=ws, out=o)

    def step_separate(s):
        h, ln, slot = plan[s]
        mw.mw_bca_cache_fwd(qs[s], ks[s], vs[s], kr, vr, h, ln, cfg.T, cfg.scale, need_lse=False,
                            workspace=ws, out=o)
        mw.mw_bca_cache_commit(kr, vr, slot, ks[s], vs[s])

    for s in range(3):
        step(s)
    torch.cuda.synchronize()
    evs = []
    for s in range(cfg.steps):
        e = Events()
        e.start()
        step(s)
        e.stop()
        evs.append(e)
    torch.cuda.synchronize()
    us = sorted(e.ms() * 1e3 for e in evs)
    med = statistics.median(us)
    # the same 64 steps captured once as a CUDA graph and replayed: device
    # time per step without host launch overhead
    def graph_us(fn):
        graph = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            with torch.cuda.graph(graph, stream=side, capture_error_mode="relaxed"):
                for s in range(cfg.steps):
                    fn(s)
        torch.cuda.current_stream().wait_stream(side)
        graph.replay()
        torch.cuda.synchronize()
        reps = []
        for _ in range(5):
            e = Events()
            e.start()
            graph.replay()
            e.stop()
            torch.cuda.synchronize()
            reps.append(e.ms() * 1e3 / cfg.steps)
        return statistics.median(reps)
    g_us = graph_us(step)
    g_sep_us = graph_us(step_separate)
    res = {"steps": cfg.steps, "us_per_step_median": round(med, 2),
           "us_per_step_p90": round(us[int(0.9 * (len(us) - 1))], 2),
           "us_per_step_graph": round(g_us, 2),
           "us_per_step_graph_separate_calls": round(g_sep_us, 2),
           "gpu_launches_per_step": 2,
           "note": "mw_bca_cache_step (forward, then the split combine and the ring commit in "
                   "one launch); eager: per-step events with host launch in the loop; graph: "
                   "the 64 steps replayed as one CUDA graph; separate_calls: forward and "
                   "commit as two API calls. The ring (57.7 MB) stays L2-resident across "
                   "steps, as in streaming"}
    # the roofline fields at the top level are from the graph time; the same
    # fields from the eager median sit under "eager"
    res.update(_cache_roofline(cfg, g_us, peaks))
    res["roofline_time"] = "us_per_step_graph"
    res["eager"] = {"us_per_step": round(med, 2), **_cache_roofline(cfg, med, peaks)}
    # the same stream through the RoPE re-shift entry point (32 rotated
    # channels; keys stored as rotated at their stream frames, two 440-token
    # frames per chunk, so each step's eviction moves the window by two
    # frames): without a sink no score changes, and the call is the plain
    # forward
    def step_rope(s):
        h, ln, slot = plan[s]
        mw.mw_bca_cache_fwd_rope(qs[s], ks[s], vs[s], None, None, kr, vr, h, ln, cfg.T, 32,
                                 10000.0, 2 * (s + 1), cfg.scale, need_lse=False, workspace=ws,
                                 out=o)
        mw.mw_bca_cache_commit(kr, vr, slot, ks[s], vs[s])

    for s in range(3):
        step_rope(s)
    torch.cuda.synchronize()
    evs = []
    for s in range(cfg.steps):
        e = Events()
        e.start()
        step_rope(s)
        e.stop()
        evs.append(e)
    torch.cuda.synchronize()
    res["rope_reshift_us_per_step_median"] = round(statistics.median(e.ms() * 1e3 for e in evs), 2)
    return res


def bench_pipelined(mw, dev, peaks, flush):
    cfg = CACHE_CONFIGS["pipelined"]
    x = gen_cache(cfg)
    kr, vr = x["k_ring"].to(dev), x["v_ring"].to(dev)
    q, kn, vn = x["q"][0].to(dev), x["k_new"][0].to(dev), x["v_new"][0].to(dev)
    ws_bytes = mw.mw_bca_cache_workspace_size(cfg.B, cfg.H, cfg.W, cfg.T, cfg.d, cfg.length)
    ws = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=dev)
    o = torch.empty_like(q)
    ts = time_repeated(lambda: mw.mw_bca_cache_fwd(q, kn, vn, kr, vr, cfg.head, cfg.length, cfg.T,
                                                   cfg.scale, need_lse=False, workspace=ws, out=o),
                       20, flush=flush)
    med = statistics.median(ts) * 1e3
    res = {"us_median": round(med, 2), "l2": "flushed between runs"}
    res.update(_cache_roofline(cfg, med, peaks))
    return res


def bench_sink(mw, dev, peaks, flush):
    """Eight in-flight chunks against the 12-chunk ring behind a one-frame sink
    anchor (the cache forward with its sink segment and split-KV combine)."""
    cfg = CACHE_CONFIGS["sink_anchor"]
    x = gen_cache(cfg)
    kr, vr = x["k_ring"].to(dev), x["v_ring"].to(dev)
    ks, vs = x["k_sink"].to(dev), x["v_sink"].to(dev)
    q, kn, vn = x["q"][0].to(dev), x["k_new"][0].to(dev), x["v_new"][0].to(dev)
    ws_bytes = mw.mw_bca_cache_workspace_size(cfg.B, cfg.H, cfg.W, cfg.T, cfg.d,
                                              cfg.sink + cfg.length)
    ws = torch.empty(max(ws_bytes, 1), dtype=torch.uint8, device=dev)
    o = torch.empty_like(q)
    ts = time_repeated(lambda: mw.mw_bca_cache_fwd_sink(q, kn, vn, ks, vs, kr, vr, cfg.head,
                                                        cfg.length, cfg.T, cfg.scale,
                                                        need_lse=False, workspace=ws, out=o),
                       20, flush=flush)
    med = statistics.median(ts) * 1e3
    res = {"us_median": round(med, 2), "l2": "flushed between runs", "sink_tokens": cfg.sink}
    res.update(_cache_roofline(cfg, med, peaks))
    # the same call with RoPE re-shifting: the first 32 channels carry the
    # temporal rotation, every key rotated at its stream frame, and 24 frames
    # (12 chunks of two 440-token frames) already evicted, so the one-frame
    # sink turns by 24 frames as it is read
    ts = time_repeated(lambda: mw.mw_bca_cache_fwd_rope(q, kn, vn, ks, vs, kr, vr, cfg.head,
                                                        cfg.length, cfg.T, 32, 10000.0, 24,
                                                        cfg.scale, need_lse=False, workspace=ws,
                                                        out=o),
                       20, flush=flush)
    med_r = statistics.median(ts) * 1e3
    res["rope_reshift"] = {"us_median": round(med_r, 2), "rope_dims": 32, "shift_frames": 24,
                           "overhead": round(med_r / med - 1, 4), **_cache_roofline(cfg, med_r, peaks)}
    return res


def profiled_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if it was taken
    on the current kernel sources (matched by the build digest)."""
    path = os.path.join(ROOT, "profiles", "ncu_traffic.txt")
    try:
        from paper_2608_01127_gb300 import _build
        digest = _build._digest()[:16]
        with open(path) as f:
            for line in f:
                parts = dict(p.split("=", 1) for p in line.split() if "=" in p)
                if parts.get("kernel") == kernel and parts.get("workload") == workload \
                        and parts.get("src") == digest:
                    return float(parts["bytes_per_launch"])
    except (OSError, ValueError, KeyError):
        pass
    return None


# ------------------------------------------------------------------ reference arm (the oracle)

def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    cfg = TRAIN_CONFIGS[WORKLOAD]
    per_head = (fwd_flops(train_pairs(cfg), cfg.d) + bwd_flops(train_pairs(cfg), cfg.d)) / (cfg.B * cfg.H)
    import oracle
    x = gen_train(cfg)

    def one(idx):
        b, h = divmod(idx % (cfg.B * cfg.H), cfg.H)
        sl = (slice(b, b + 1), slice(h, h + 1))
        qq, kk, vv, dd = (x[n][sl] for n in ("q", "k", "v", "do"))
        oracle.fwd(qq, kk, vv, cfg.T, cfg.scale)
        oracle.bwd(qq, kk, vv, dd, cfg.T, cfg.scale)

    for i in range(args.warmup):
        one(i)
    t0 = time.perf_counter()
    for i in range(args.steps):
        one(args.warmup + i)
    dt = time.perf_counter() - t0
    value = per_head * args.steps / dt / 1e12
    out = {"impl": "reference", "metric": METRIC, "value": round(value, 6), "unit": "TFLOP/s",
           "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(dt * 1e3 / args.steps, 2), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": f"{WORKLOAD}: block-causal attention fwd+bwd; each step is one "
                                  f"(b,h) head of B={cfg.B} H={cfg.H} d={cfg.d}, "
                                  f"{cfg.n_chunks} chunks x {cfg.T} tokens"},
           "cpu_baseline": {"value": round(value, 6), "unit": "TFLOP/s", "kind": "oracle",
                            "cores": torch.get_num_threads(),
                            "sample": f"one (b,h) head of {WORKLOAD} per step, fp64 oracle"},
           "e2e": {"value": round(value, 6), "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--no-extras", action="store_true", help="skip the secondary workloads")
    ap.add_argument("--extras-only", default=None,
                    help="comma-separated secondary workloads to run alone, without the "
                         "headline step (profiling; prints their results only): "
                         + ", ".join(EXTRA_NAMES))
    ap.add_argument("--workload", choices=sorted(n for n, c in TRAIN_CONFIGS.items() if c.backward),
                    default=WORKLOAD,
                    help="training workload of the timed step (default: the headline one)")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="budget of the oracle CPU baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true",
                    help="skip the oracle CPU baseline (profiling runs)")
    args = ap.parse_args(argv)
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    world, _, _ = dist_env()
    if world != args.gpus and world > 1:
        ap.error(f"--gpus {args.gpus} but WORLD_SIZE={world}")
    if args.impl == "reference":
        run_reference(args)
    elif args.extras_only:
        run_extras_only(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
