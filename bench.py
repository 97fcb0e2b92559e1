#!/usr/bin/env python
"""Benchmark of the layer-wise visual KV-memory build (embedding adapter, Sec. 3.1-3.2).

One step = one build of every layer's visual K/V cache entries for one batch of synthetic
visual embeddings: row statistics, stacked down-projection + SiLU, RMS statistics, and the
K/V projection with RoPE and the bf16 cache store, all in the library's CUDA kernels.

The headline workload is the largest synthetic configuration that fits one GPU, the
LLaVA-NeXT-7B-shaped high-resolution batch (d = 4096, L = 32, 32 x 128 MHA, r = 128,
8 x 2880 visual tokens). The line also carries ``per_config``: the LLaVA-1.5-7B-shaped and
both Qwen2.5-VL-7B-shaped workloads, each device-timed with its own roofline.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl dv|reference]
                    [--shard replicas|tokens|layers]

Prints ONE JSON line on rank 0. Under torchrun (N > 1) the ranks split the work as --shard
says: every rank builds its own batch (replicas, weak scaling, no collective on the data path),
or the ranks split one batch's tokens (no collective) or its layers (x0 broadcast from rank 0
every step); timing is the max over ranks.
``--impl reference`` times the fp64 oracle on the host cores instead (bounded samples).
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

METRIC = "visual tokens/sec of layer-wise visual KV-memory build; % of BF16 tensor roofline"
UNIT = "visual tokens/s"
DEFAULT_WORKLOAD = "llava_next_7b"
# device-timed beside the headline (each with its own roofline)
PER_CONFIG = ["llava15_7b", "qwen25vl_7b_image", "qwen25vl_7b_video"]
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# NVIDIA's published GB300 figures, reported beside the measured peaks: 2.25 PFLOP/s dense bf16
# per GPU (its 36 PFLOP/s for eight GPUs counts 2:4 sparsity) and 7.9 TB/s of HBM3e.
NOMINAL_PEAKS = {"bf16_tflops": 2250.0, "hbm_gbs": 7900.0}
GEMM_SOURCES = ["paper_2609_34972_gb300/csrc/dv_kv2sm.cu", "paper_2609_34972_gb300/csrc/dv_pair_tm.cu",
                "paper_2609_34972_gb300/csrc/dv_ptx.cuh",
                "paper_2609_34972_gb300/csrc/dv_epilogue.cuh", "paper_2609_34972_gb300/csrc/dv_internal.h"]


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def kernel_source_hash() -> str:
    h = hashlib.sha256()
    for rel in GEMM_SOURCES:
        with open(os.path.join(ROOT, rel), "rb") as f:
            h.update(f.read())
    return h.hexdigest()[:16]


def profiled_traffic(workload: str):
    """DRAM bytes per launch of the K/V kernel from the committed ncu summary, if that summary
    was taken on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", f"kv_proj_rope_store_{workload}.md")
    if not os.path.exists(path):
        return None
    text = open(path).read()
    m = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
    s = re.search(r"kernel_source_sha256_16:\s*([0-9a-f]+)", text)
    if not m or not s or s.group(1) != kernel_source_hash():
        return None
    return float(m.group(1))


class ClockSampler:
    """Samples nvidia-smi clocks and throttle reasons while the timed region runs."""

    FIELDS = ["index", "clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.active",
              "clocks_event_reasons.hw_slowdown", "clocks_event_reasons.hw_thermal_slowdown",
              "clocks_event_reasons.sw_thermal_slowdown", "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu_id: str | None):
        self.proc = None
        self.gpu_id = gpu_id

    def start(self):
        cmd = ["nvidia-smi", "--query-gpu=" + ",".join(self.FIELDS), "--format=csv,noheader,nounits",
               "-lms", "100"]
        if self.gpu_id:
            cmd += ["-i", self.gpu_id]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, ValueError):
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.15)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            # Every wait here is bounded: an nvidia-smi that does not exit (a driver query that
            # blocks) must not hold the bench; the line then carries no clock record.
            self.proc.kill()
            try:
                out, _ = self.proc.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                return None
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.splitlines():
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(ms: float, dist=None, device=None) -> float:
    """The slowest rank's time (the job's time): all_reduce MAX over the process group."""
    if dist is None:
        return float(ms)
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_value(world: int, tokens_per_rank: int, steps: int, ms_max: float) -> float:
    """Whole-job visual tokens/s: every rank builds its own batch of the workload (replicas,
    no collective on the data path), so the job processes world * tokens_per_rank per step."""
    return world * tokens_per_rank * steps / (ms_max / 1000.0)


def stratified_tokens(cfg, n: int, seed: int = 0):
    """n flat token ids spread over every batch element: each element gets its share at evenly
    spaced positions with a random offset, so the sample covers the whole position range."""
    import numpy as np
    rng = np.random.default_rng(seed)
    n = int(max(1, min(n, cfg.tokens)))
    per = [n // cfg.batch + (1 if b < n % cfg.batch else 0) for b in range(cfg.batch)]
    out = []
    for b, k in enumerate(per):
        if k == 0:
            continue
        step = cfg.n_vis / k
        idx = np.floor(np.arange(k) * step + rng.uniform(0, step, size=k)).astype(np.int64)
        out.append(b * cfg.n_vis + np.minimum(idx, cfg.n_vis - 1))
    return np.unique(np.concatenate(out))


def strong_scaling_value(tokens_per_step: int, steps: int, ms_max: float) -> float:
    """Whole-job visual tokens/s when the ranks split one batch (by tokens or by layers): the
    job processes the batch's tokens once per step, whatever the rank count."""
    return tokens_per_step * steps / (ms_max / 1000.0)


def time_oracle_sample(inp, budget_s: float, seed: int = 0, min_tokens: int = 0):
    """Oracle throughput (tokens/s) on a bounded, stratified sample of whole tokens (all
    layers): at least min_tokens, else as many as about budget_s of oracle time allows."""
    import numpy as np
    import oracle
    cfg = inp.cfg
    t0 = time.perf_counter()
    oracle.build_tokens(inp, np.array([0], dtype=np.int64))
    t1 = time.perf_counter() - t0
    n = int(max(1, min(cfg.tokens, max(min_tokens, budget_s / max(t1, 1e-6)))))
    toks = stratified_tokens(cfg, n, seed)
    t0 = time.perf_counter()
    oracle.build_tokens(inp, toks)
    dt = time.perf_counter() - t0
    return {"value": len(toks) / dt, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
            "sample": f"{len(toks)} of {cfg.tokens} tokens (all {cfg.n_layers} layers each), "
                      f"spread evenly over all {cfg.batch} batch elements, of the {cfg.name} "
                      f"workload, fp64, {dt:.1f} s; tokens/s = sampled tokens / oracle time"}


def workload_config(args):
    """The synthetic workload of --config, with --layers and --adapter applied."""
    from dataclasses import replace
    import synth
    cfg = synth.CONFIGS[args.config]
    if args.layers:
        cfg = replace(cfg, n_layers=args.layers, name=f"{cfg.name}_L{args.layers}")
    if args.adapter == "recurrent":
        cfg = replace(cfg, adapter="recurrent", name=f"{cfg.name}_recurrent",
                      description=cfg.description + "; recurrent adapter (Sec. 3.1 Eq. 6)")
        if args.split_chain:
            cfg = replace(cfg, split_chain=True, name=cfg.name + "_split",
                          description=cfg.description + ", split-bf16 chain")
    return cfg


def run_reference(args):
    """The oracle as the reference arm: every step is a bounded sample of (token, layer) pairs."""
    import numpy as np
    import oracle
    import synth
    rank, world, _ = dist_env()
    if rank != 0:
        return
    cfg = workload_config(args)
    inp = synth.make_inputs(cfg)
    rng = np.random.default_rng(0)
    # The recurrent chain of a layer needs every layer before it: evaluate whole tokens.
    whole = cfg.adapter == "recurrent"
    t0 = time.perf_counter()
    oracle.build_tokens(inp, np.array([0], dtype=np.int64), layers=None if whole else [0])
    t_pair = max(time.perf_counter() - t0, 1e-4) / (cfg.n_layers if whole else 1)
    n_steps = args.warmup + args.steps
    cores = oracle.num_threads()
    # one random layer per step, evaluated for per_step random tokens (parallel over tokens)
    per_step = max(1, int(min(cfg.tokens, (args.ref_budget_s / n_steps) / t_pair * cores)))
    total_t, total_pairs = 0.0, 0
    for step in range(n_steps):
        toks = np.sort(rng.choice(cfg.tokens, size=per_step, replace=False)).astype(np.int64)
        if whole:
            toks = toks[:max(1, per_step // cfg.n_layers)]
        lay = None if whole else [int(rng.integers(0, cfg.n_layers))]
        t0 = time.perf_counter()
        oracle.build_tokens(inp, toks, layers=lay)
        dt = time.perf_counter() - t0
        if step >= args.warmup:
            total_t += dt
            total_pairs += len(toks) * (cfg.n_layers if whole else 1)
    value = (total_pairs / cfg.n_layers) / total_t
    out = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": 1000.0 * total_t / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": cfg.name, "description": cfg.description,
                   "sample_per_step": (f"{max(1, per_step // cfg.n_layers)} tokens x all layers"
                                       if whole else f"{per_step} tokens x 1 random layer")},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle.num_threads(), "kind": "oracle",
                         "sample": (f"{max(1, per_step // cfg.n_layers)} random whole tokens per "
                                    f"step of the {cfg.name} workload" if whole else
                                    f"{per_step} random tokens at one random layer per step of the "
                                    f"{cfg.name} workload; tokens/s = (token, layer) pairs/s / "
                                    f"{cfg.n_layers} layers")},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(out), flush=True)


def roofline_of(dv, plan, work, stage_ms, n_timed, ms_total, ms_step, peaks, peak_src, tokens):
    """Roofline of the dominant kernel (K/V projection + RoPE + store) and of the whole step."""
    kv_ms = stage_ms[3] / max(n_timed, 1)
    kv_flops = 4.0 * work.d * work.kv * work.tokens * work.n_layers
    # The K/V kernel is timed inside a run of back-to-back builds. Once that run lasts as long
    # as the seconds-long cuBLAS loop behind the sustained figure (the power cap then sets the
    # clock), its peak is that sustained rate; shorter runs are compared with the burst rate.
    sustained = ms_total >= 2000.0
    peak_tf = peaks["bf16_tflops_sustained"] if sustained else peaks["bf16_tflops"]
    peak_name = "bf16_tflops_sustained" if sustained else "bf16_tflops (burst)"
    achieved_tf = kv_flops / (kv_ms * 1e-3) / 1e12
    t_roof_ms = max(work.flops() / (peaks["bf16_tflops"] * 1e12),
                    work.min_bytes() / (peaks["hbm_gbs"] * 1e9)) * 1e3
    t_roof_sus = max(work.flops() / (peaks["bf16_tflops_sustained"] * 1e12),
                     work.min_bytes() / (peaks["hbm_gbs"] * 1e9)) * 1e3
    roof = {"bound": "tensor", "achieved": achieved_tf, "peak": peak_tf, "unit": "TFLOP/s",
            "frac": achieved_tf / peak_tf, "traffic": profiled_traffic(work.name),
            "kernel": dv.kv_kernel(plan, tokens) + ": K/V projection + RoPE + cache store",
            "peak_source": f"{peak_name} of {peak_src}; timed region {ms_total:.0f} ms of "
                           f"back-to-back builds",
            "frac_burst": achieved_tf / peaks["bf16_tflops"],
            "frac_sustained": achieved_tf / peaks["bf16_tflops_sustained"],
            "frac_nominal": achieved_tf / NOMINAL_PEAKS["bf16_tflops"],
            "flops_per_launch": kv_flops, "ms_per_launch": kv_ms}
    t_roof_nom = max(work.flops() / (NOMINAL_PEAKS["bf16_tflops"] * 1e12),
                     work.min_bytes() / (NOMINAL_PEAKS["hbm_gbs"] * 1e9)) * 1e3
    step = {"t_roof_ms": t_roof_ms, "frac": t_roof_ms / ms_step, "frac_sustained": t_roof_sus / ms_step,
            "frac_nominal": t_roof_nom / ms_step,
            "plain_flops": work.flops(), "min_bytes": work.min_bytes()}
    return roof, step


def time_builds(dv, plan, build, steps, warmup, stream, barrier=None, clocks=None):
    """Device time (ms) of `steps` back-to-back builds after `warmup` untimed ones, CUDA events
    on the build stream; then the per-stage times from a second run with the plan's stage events
    (kept out of the timed run: an event between two kernels stops the next one from starting
    early)."""
    import torch
    for _ in range(warmup):
        build()
    torch.cuda.synchronize()
    st = dv.plan_status(plan)
    if st != dv.DV_OK:
        raise RuntimeError(f"device status after warm-up: {dv.error_string(st)}")
    if barrier:
        barrier()
    torch.cuda.synchronize()
    if clocks:
        clocks.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        build()
    e1.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop() if clocks else None
    if barrier:
        barrier()
    ms_total = e0.elapsed_time(e1)
    dv.timing_enable(plan, True)
    for _ in range(min(steps, 200)):
        build()
    torch.cuda.synchronize()
    stage_ms, n_timed = dv.timing_read(plan)
    dv.timing_enable(plan, False)
    st = dv.plan_status(plan)
    if st != dv.DV_OK:
        raise RuntimeError(f"device status after timed region: {dv.error_string(st)}")
    return ms_total, clk, stage_ms, n_timed


def gpu_id_of(dev, local):
    import torch
    try:
        return "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        return str(local)


def measure_config(dv, cfg, args, dev, peaks, peak_src, skip=None):
    """Device-timed build of one more workload (inputs resident), for the per_config and
    variants blocks. ``skip`` = (F, K): no visual memory at the first F and last K layers (App. J
    adapter skipping, DV_LAYER_DROP); the algorithmic work then counts the built layers."""
    import numpy as np
    import torch
    import synth
    from dataclasses import replace
    from tests import gpu_util as gu
    inp = synth.make_inputs(cfg)
    modes, work = None, cfg
    if skip:
        f, k = skip
        modes = [dv.DV_LAYER_DROP if (l < f or l >= cfg.n_layers - k) else dv.DV_LAYER_ADAPTER
                 for l in range(cfg.n_layers)]
        work = replace(cfg, n_layers=cfg.n_layers - f - k, name=f"{cfg.name}_skip{f}_{k}")
    plan = dv.memory_plan(gu.dv_config(cfg), gu.device_weights(inp, dev), layer_modes=modes)
    x0 = gu.torch_bf16(inp.x0, dev)
    pos = torch.from_numpy(np.ascontiguousarray(inp.pos)).to(dev)
    shape = (cfg.n_layers, cfg.batch, cfg.n_vis, cfg.n_kv_heads, cfg.head_dim)
    kc = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
    vc = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream()
    build = lambda: dv.build_visual_memory(plan, x0, pos, kc, vc, stream=stream)
    ms_total, clk, stage_ms, n_timed = time_builds(dv, plan, build, args.steps, args.warmup, stream,
                                                   clocks=ClockSampler(gpu_id_of(dev, 0)))
    ms_step = ms_total / args.steps
    roof, step = roofline_of(dv, plan, work, stage_ms, n_timed, ms_total, ms_step, peaks, peak_src,
                             cfg.tokens)
    out = {"workload": work.name, "description": cfg.description +
           (f"; no visual memory at the first {skip[0]} and last {skip[1]} layers (App. J)" if skip else ""),
           "layers_with_visual_memory": work.n_layers, "tokens_per_step": cfg.tokens,
           "value": cfg.tokens * args.steps / (ms_total / 1000.0), "unit": UNIT,
           "ms_per_step": ms_step, "steps": args.steps, "clocks": clk, "roofline": roof,
           "roofline_step": step,
           "stage_ms_per_step": dict(zip(dv.stage_names(plan), [x / max(n_timed, 1) for x in stage_ms]))}
    dv.free(plan)
    del kc, vc, x0, pos
    torch.cuda.empty_cache()
    return out


def run_dv(args):
    import numpy as np
    import torch
    import synth
    from paper_2609_34972_gb300.build import build_library
    build_library()
    import paper_2609_34972_gb300 as dv
    from paper_2609_34972_gb300 import shard as sh
    from tests import gpu_util as gu

    rank, world, local = dist_env()
    if world != args.gpus:
        raise SystemExit(f"--gpus {args.gpus} but {world} process(es): launch N > 1 under torchrun "
                         f"with --nproc-per-node N")
    dist = None
    if world > 1:
        import torch.distributed as tdist
        tdist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
        dist = tdist
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    cfg = workload_config(args)
    peaks, peak_src = load_peaks()
    mode = args.shard if world > 1 else "replicas"
    if mode == "layers" and cfg.adapter == "recurrent":
        raise SystemExit("the recurrent adapter chains the layers: split it by tokens")
    modes = None
    if args.skip_layers:
        first, last = (int(x) for x in args.skip_layers.split(","))
        modes = [dv.DV_LAYER_DROP if (l < first or l >= cfg.n_layers - last) else dv.DV_LAYER_ADAPTER
                 for l in range(cfg.n_layers)]
    if mode == "layers":
        modes = sh.layer_modes(cfg.n_layers, world, rank, modes)
    layers_built = cfg.n_layers if modes is None else sum(m != dv.DV_LAYER_DROP for m in modes)

    # ---- inputs (host, seeded) -> device; plan once outside the timing
    inp = synth.make_inputs(cfg)
    x0_full = gu.torch_bf16(inp.x0, "cpu")
    pos_np = np.ascontiguousarray(inp.pos)
    if mode == "tokens":
        part = sh.token_shard(cfg.batch, cfg.n_vis, world, rank)
        B, N = 1, part.tokens
        x0_h = x0_full.reshape(cfg.tokens, cfg.d)[part.start:part.stop].reshape(1, N, cfg.d).contiguous()
        pos_h = torch.from_numpy(sh.shard_positions(pos_np, part))
    else:
        B, N = cfg.batch, cfg.n_vis
        x0_h, pos_h = x0_full, torch.from_numpy(pos_np)
    T = B * N
    from dataclasses import replace as _replace
    # the algorithmic work this rank does: its tokens and the layers that get visual memory
    work = _replace(cfg, batch=B, n_vis=N, n_layers=layers_built,
                    name=cfg.name + (f"_skip{args.skip_layers.replace(',', '_')}" if args.skip_layers else ""))
    weights = gu.device_weights(inp, dev)
    plan = dv.memory_plan(gu.dv_config(cfg, max_batch=B, max_n_vis=N), weights, layer_modes=modes)
    del weights
    x0 = x0_h.to(dev)
    pos = pos_h.to(dev)
    shape = (cfg.n_layers, B, N, cfg.n_kv_heads, cfg.head_dim)
    kc = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
    vc = torch.zeros(shape, dtype=torch.bfloat16, device=dev)
    stream = torch.cuda.current_stream()

    def barrier():
        if dist is not None:
            dist.barrier()

    def build():
        if mode == "layers":
            dist.broadcast(x0, src=0)   # E from rank 0: the one collective of the layer split
        dv.build_visual_memory(plan, x0, pos, kc, vc, stream=stream)

    # ---- timed region (device-resident inputs)
    ms_total, clk, stage_ms, n_timed = time_builds(dv, plan, build, args.steps, args.warmup, stream,
                                                   barrier, ClockSampler(gpu_id_of(dev, local)))
    ms_total = max_over_ranks(ms_total, dist, dev)
    ms_step = ms_total / args.steps
    # replicas: every rank builds its own batch; token / layer splits: the ranks build one batch
    job_tokens = world * T if mode == "replicas" else cfg.tokens
    value = (weak_scaling_value(world, T, args.steps, ms_total) if mode == "replicas"
             else strong_scaling_value(cfg.tokens, args.steps, ms_total))

    # ---- end to end through the C ABI from page-locked host buffers: every step copies its E
    #      and positions host-to-device and its built K/V device-to-host inside the timed region
    #      (dv_build_visual_memory_host); the copy-out of one step overlaps the next build
    x0_p = x0_h.pin_memory()
    pos_p = pos_h.pin_memory()
    k_p = torch.empty(shape, dtype=torch.bfloat16).pin_memory()
    v_p = torch.empty(shape, dtype=torch.bfloat16).pin_memory()
    e2e_steps = max(5, min(args.steps, args.e2e_steps))
    pipe = dv.HostPipeline(plan, B, N, depth=2)
    for _ in range(max(3, args.warmup)):   # also the first touches of the host pages
        pipe.submit(x0_p, pos_p, k_p, v_p, stream=stream)
    pipe.join(stream)
    torch.cuda.synchronize()
    barrier()
    s0, s1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s0.record(stream)
    for _ in range(e2e_steps):
        pipe.submit(x0_p, pos_p, k_p, v_p, stream=stream)
    pipe.join(stream)
    s1.record(stream)
    torch.cuda.synchronize()
    barrier()
    ms_e2e = max_over_ranks(s0.elapsed_time(s1), dist, dev)
    e2e_value = job_tokens * e2e_steps / (ms_e2e / 1000.0)
    h2d = x0_p.numel() * 2 + pos_p.numel() * 4
    d2h = 2 * layers_built * T * cfg.kv * 2
    st = dv.plan_status(plan)
    if st != dv.DV_OK:
        raise RuntimeError(f"device status after the end-to-end region: {dv.error_string(st)}")
    pipe.close()
    del pipe, k_p, v_p

    roof, roof_step = roofline_of(dv, plan, work, stage_ms, n_timed, ms_total, ms_step, peaks,
                                  peak_src, T)
    stage = dict(zip(dv.stage_names(plan), [x / max(n_timed, 1) for x in stage_ms]))
    launches = args.steps * dv.kernels_per_build(plan)
    dv.free(plan)
    del kc, vc
    torch.cuda.empty_cache()

    cpu = None
    per_config = None
    variants = None
    if rank == 0 and world == 1:
        if not args.no_per_config and args.config == DEFAULT_WORKLOAD and not args.layers \
                and args.adapter == "embedding" and not args.skip_layers:
            import synth
            from dataclasses import replace
            per_config = [measure_config(dv, synth.CONFIGS[n], args, dev, peaks, peak_src)
                          for n in PER_CONFIG]
            # the variants of the path beside the embedding adapter: on the LLaVA-1.5 shape the
            # recurrent adapter (Sec. 3.1 Eq. 6) and the consumer of the memory (Sec. 3.2)
            rec = replace(synth.CONFIGS["llava15_7b"], adapter="recurrent",
                          name="llava15_7b_recurrent",
                          description=synth.CONFIGS["llava15_7b"].description +
                          "; recurrent adapter (Sec. 3.1 Eq. 6)")
            # on the Qwen2.5-VL video shape (128 token blocks, rank 256) the recurrent adapter
            # runs the rearranged chain: E D^T, the r-wide recurrence, the running sum of M_l
            vid = synth.CONFIGS["qwen25vl_7b_video"]
            rec_v = replace(vid, adapter="recurrent", name="qwen25vl_7b_video_recurrent",
                            description=vid.description + "; recurrent adapter (Sec. 3.1 Eq. 6)")
            # and the Qwen3-VL-4B-shaped build (the paper's default backbone: per-head K norm,
            # interleaved M-RoPE)
            # with the App. J skipping of its first 5 and last 10 adapters
            q3 = synth.CONFIGS["qwen3vl_4b_image"]
            variants = [measure_config(dv, rec, args, dev, peaks, peak_src),
                        measure_config(dv, rec_v, args, dev, peaks, peak_src),
                        measure_config(dv, q3, args, dev, peaks, peak_src),
                        measure_config(dv, q3, args, dev, peaks, peak_src, skip=(5, 10)),
                        measure_consumer(dv, synth.CONFIGS["llava15_7b"], args, peaks)]
        if not args.no_cpu_baseline:
            cpu = time_oracle_sample(inp, args.cpu_budget_s,
                                     min_tokens=min(cfg.tokens, 512) if cfg.batch > 1 else 0)

    if rank == 0:
        par = {"replicas": "replicas (weak scaling, no collective)",
               "tokens": "token split of one batch (strong scaling, no collective)",
               "layers": "layer split of one batch (strong scaling, x0 broadcast per step)"}[mode]
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
            "scaling": "weak" if mode == "replicas" else "strong", "vs_baseline": None,
            "dtype": "bf16", "data": "synthetic",
            "config": {"workload": work.name, "description": cfg.description,
                       "layers_with_visual_memory": layers_built if mode != "layers" else cfg.n_layers,
                       "tokens_per_step": job_tokens, "tokens_per_step_per_gpu": T,
                       "layers": cfg.n_layers,
                       "l2": f"inputs larger than L2: the {layers_built}-layer weight set "
                             f"({(work.min_bytes() - work.tokens * work.n_layers * 4 * work.kv) / 1e9:.2f} GB "
                             f"incl. x0) is streamed from HBM every step",
                       "parallelism": par if world > 1 else "1 GPU"},
            "clocks": clk,
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                    "d2h_bytes_per_step": d2h, "steps": e2e_steps,
                    "ms_per_step": ms_e2e / e2e_steps,
                    "how": "C ABI dv_build_visual_memory_host (dv_host_pipeline, 2 staging sets): "
                           "per step one cudaMemcpyAsync each of E and the positions host-to-device "
                           "from page-locked memory, the build, and one cudaMemcpyAsync each of K "
                           "and V device-to-host; the copy-out of a step overlaps the next build"},
            "gpu_launches": launches,
            "roofline": roof,
            "roofline_step": roof_step,
            "stage_ms_per_step": stage,
            "cpu_baseline": cpu,
            "per_config": per_config,
            "variants": variants,
        }
        print(json.dumps(out), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def measure_consumer(dv, cfg, args, peaks):
    """The consumer of the visual memory (Sec. 3.2): one step = the causal attention of the
    prefill's text queries over every layer's cache (system-prompt text slots, the visual slots
    written by the build, the text slots), through dv_text_attention, one launch per layer."""
    import torch
    import synth
    from tests import gpu_util as gu
    n_sys, n_text, hq = args.consumer_sys, args.consumer_text, cfg.n_heads
    B, Nv, H, D, L = cfg.batch, cfg.n_vis, cfg.n_kv_heads, cfg.head_dim, cfg.n_layers
    S = n_sys + Nv + n_text
    inp = synth.make_inputs(cfg)
    k, v, plan = gu.run_build(inp, seq_len=S, slot0=n_sys)
    dv.free(plan)
    gen = torch.Generator(device="cuda").manual_seed(7)
    for l in range(L):
        k[l, :, :n_sys].normal_(generator=gen)
        v[l, :, :n_sys].normal_(generator=gen)
        k[l, :, n_sys + Nv:].normal_(generator=gen)
        v[l, :, n_sys + Nv:].normal_(generator=gen)
    q = torch.randn((L, B, hq, n_text, D), generator=gen, device="cuda").to(torch.bfloat16)
    out = torch.empty((B, hq, n_text, D), dtype=torch.bfloat16, device="cuda")
    nk = torch.full((B,), S, dtype=torch.int32, device="cuda")
    qs = (n_sys + Nv + torch.arange(n_text, dtype=torch.int32, device="cuda")).repeat(B, 1)
    scale = 1.0 / D ** 0.5

    def step():
        for l in range(L):
            dv.text_attention(q[l], k, v, l, nk, qs, scale, out=out)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    # A decoder calls the attention layer by layer; a serving engine replays that sequence as a
    # CUDA graph, so the step is captured once and replayed (no per-call host cost in the timing).
    graph = torch.cuda.CUDAGraph()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()
    torch.cuda.current_stream().wait_stream(side)
    with torch.cuda.graph(graph):
        step()
    graph.replay()
    torch.cuda.synchronize()
    clk = ClockSampler(os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")[0] or None)
    clk.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record()
    for _ in range(args.steps):
        graph.replay()
    e1.record()
    torch.cuda.synchronize()
    clocks = clk.stop()
    assert dv.text_attention_status() == dv.DV_OK
    ms = e0.elapsed_time(e1) / args.steps
    # each query row sees all S slots (the text slots up to its own): keys read once per layer
    kv_bytes = L * B * H * S * D * 2 * 2
    qo_bytes = L * B * hq * n_text * D * 2 * 2
    flops = sum(4.0 * B * hq * D * (n_sys + Nv + t + 1) for t in range(n_text)) * L
    gbs = (kv_bytes + qo_bytes) / (ms * 1e-3) / 1e9
    del graph, k, v
    torch.cuda.empty_cache()
    return {
        "metric": "text-query attention over the visual memory: text tokens/s (all layers)",
        "value": B * n_text / (ms * 1e-3), "unit": "text tokens/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
        "dtype": "bf16", "data": "synthetic",
        "config": {"workload": cfg.name + "_consumer", "layers": L, "batch": B,
                   "slots": {"system": n_sys, "visual": Nv, "text": n_text},
                   "q_heads": hq, "kv_heads": H, "head_dim": D,
                   "l2": f"{(kv_bytes + qo_bytes) / 1e6:.0f} MB read per step (> L2)",
                   "timing": "the step (one dv_text_attention per layer) captured in a CUDA graph "
                             "and replayed"},
        "roofline": {"bound": "hbm", "achieved": gbs, "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": gbs / peaks["hbm_gbs"], "traffic": None,
                     "kernel": "dv_attn_kernel", "bytes_per_step": kv_bytes + qo_bytes,
                     "tflops": flops / (ms * 1e-3) / 1e12},
        "clocks": clocks, "gpu_launches": args.steps * L,
    }


def run_consumer(args):
    """``--consumer``: the consumer's own JSON line (see measure_consumer)."""
    import torch
    from paper_2609_34972_gb300.build import build_library
    build_library()
    import paper_2609_34972_gb300 as dv
    rank, world, local = dist_env()
    if rank != 0:
        return
    torch.cuda.set_device(local)
    peaks, _ = load_peaks()
    print(json.dumps(measure_consumer(dv, workload_config(args), args, peaks)), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__, formatter_class=argparse.RawDescriptionHelpFormatter)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--config", default=DEFAULT_WORKLOAD)
    ap.add_argument("--layers", type=int, default=0,
                    help="override the layer count (smaller profiling cases of the same shape)")
    ap.add_argument("--skip-layers", default="",
                    help="F,K: no visual memory at the first F and last K layers (App. J adapter "
                         "skipping, DV_LAYER_DROP)")
    ap.add_argument("--adapter", choices=["embedding", "recurrent"], default="embedding",
                    help="embedding adapter (Sec. 3.1 Eq. 5, the default workload) or the "
                         "recurrent adapter (Eq. 6)")
    ap.add_argument("--split-chain", action="store_true",
                    help="recurrent adapter: the chain's GEMMs read hi + lo bf16 operands")
    ap.add_argument("--impl", choices=["dv", "reference"], default="dv")
    ap.add_argument("--consumer", action="store_true",
                    help="measure the consumer instead: causal text-query attention over every "
                         "layer's cache (dv_text_attention)")
    ap.add_argument("--consumer-sys", type=int, default=35, help="system-prompt slots before the visual slots")
    ap.add_argument("--consumer-text", type=int, default=64, help="text query tokens after them")
    ap.add_argument("--e2e-steps", type=int, default=100)
    ap.add_argument("--shard", choices=["replicas", "tokens", "layers"], default="replicas",
                    help="N > 1: every rank builds its own batch (weak scaling), or the ranks "
                         "split one batch by tokens or by layers (strong scaling)")
    ap.add_argument("--no-per-config", action="store_true",
                    help="skip the per_config block (the other workloads, device-timed)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget-s", type=float, default=15.0)
    ap.add_argument("--ref-budget-s", type=float, default=120.0)
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)   # at least 3 untimed warm-up steps
    if args.steps > 4096:
        ap.error("--steps must be <= 4096 (per-stage timing records at most 4096 builds)")
    if args.impl == "reference":
        run_reference(args)
    elif args.consumer:
        run_consumer(args)
    else:
        run_dv(args)


if __name__ == "__main__":
    main()
