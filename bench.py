#!/usr/bin/env python
"""Benchmark of the X-Cache chunk step on GB300.

One step = one chunk of the AR rollout: S = 4 denoising passes (each through
all B blocks, gate + reuse or recompute per block) + 1 KV-update pass, with the
Euler update between passes.  Inputs (noise, clean latents, actions) are
resident in HBM before the timed region; the per-chunk working set (KV ring,
residual cache, weights) is larger than L2.

Default workload: the small multi-camera DiT (8 blocks, d 512, 8 heads x 64,
FFN 2048, 6 cameras x 3 frames x 16 x 28 = 8064 tokens per chunk, KV ring of 4
chunks = 32256 keys), bf16 with fp32 accumulation, synthetic AR(1) latents.

Prints one JSON line (rank 0).  ``--impl reference`` times the CPU oracle
instead (bounded sample, rank 0 only).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import xc_inputs as X  # noqa: E402

METRIC = "ms/chunk & chunks/s, X-Cache vs all-blocks; block skip rate; % BF16 TC peak"
WORKLOADS = {"small": X.SMALL_BF16, "1p3b": X.DIT_1P3B, "14b": X.DIT_14B, "tiny": X.TINY_F32}
# Gate thresholds giving a mid-range skip rate on this synthetic workload (other
# knobs: Table 1 defaults).
GATE = dict(tau_floor=0.93, tau_dev=3.0)
SIGMAS = (1.0, 0.75, 0.5, 0.25, 0.0)


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=8)
    ap.add_argument("--warmup", type=int, default=4)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="small", choices=sorted(WORKLOADS))
    ap.add_argument("--tau-floor", type=float, default=GATE["tau_floor"])
    ap.add_argument("--tau-dev", type=float, default=GATE["tau_dev"])
    ap.add_argument("--kv-period", type=int, default=0,
                    help="KV-update pass only on chunks n mod P == P-1, whose denoising passes "
                         "run in force-compute mode (0 = KV-update pass after every chunk)")
    ap.add_argument("--view-groups", default="",
                    help="view groups of the chunk as CAMSxHxW,... (e.g. 3x20x36,2x16x28,2x12x20); "
                         "default: the workload's single camera grid")
    ap.add_argument("--xattn", type=int, default=0,
                    help="add cross-attention to up to N condition tokens of width d_model per chunk "
                         "(count varying per chunk in [3N/4, N]); 0 = none")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--calibrate", action="store_true", help="print gate-metric quantiles and exit")
    ap.add_argument("--sweep", action="store_true",
                    help="threshold sweep on the stress rollout (1.3B shape, closed loop); prints one JSON line")
    ap.add_argument("--sweep-chunks", type=int, default=200)
    # gate aggressiveness ladder: tau_floor:margin:tau_dev (Eq. 9 floor, EMA
    # margin m, deviation threshold of Eq. 7); the first point is Table 1
    ap.add_argument("--sweep-points",
                    default="0.97:0.02:2.0,0.95:0.05:3.0,0.9:0.1:4.0,0.8:0.2:6.0,0.6:0.4:10.0,0.3:0.7:20.0")
    return ap.parse_args()


# ------------------------------------------------------------------ helpers
def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """The largest per-rank value over all ranks (the slowest replica's
    time); one all-reduce of one scalar, no data-path collective."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(units_per_rank: int, world: int, seconds: float) -> float:
    """Weak scaling: the units all replicas processed over the slowest
    replica's time."""
    return units_per_rank * world / seconds


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 200 ms."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.gpu = gpu
        self.proc = None
        # raw samples go to $XC_BENCH_OUT (default: the system temp directory)
        out = os.environ.get("XC_BENCH_OUT") or tempfile.gettempdir()
        self.path = os.path.join(out, f"xc_clocks_gpu{gpu}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        self.proc.wait(timeout=5)
        self.fh.close()
        sm, mx, reasons = [], None, set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in open(self.path):
            f = [c.strip() for c in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for name, val in zip(names, f[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        load = [s for s in sm if mx and s > 0.5 * mx] or sm
        return {"sm_mhz": statistics.median(load) if load else None, "sm_max_mhz": mx,
                "samples": len(sm), "reasons": sorted(reasons)}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "of measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "of fallback"


def traffic_record(kernel: str):
    """dram bytes per launch of `kernel` from the committed ncu summary, or
    None when absent or taken on a different source revision of the kernel."""
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    rec = json.load(open(p)).get(kernel)
    if not rec:
        return None
    import hashlib
    src = os.path.join(ROOT, "paper_2604_20289_gb300", "csrc", rec["source"])
    if not os.path.exists(src) or hashlib.sha256(open(src, "rb").read()).hexdigest()[:16] != rec["sha"]:
        return None
    return rec


# ------------------------------------------------------------------ oracle
def oracle_block_sample(cfg, seed: int = 0) -> float:
    """Seconds the CPU oracle takes for ONE block forward at full ring
    (all cfg.tokens queries x kv_window * tokens keys) on this host."""
    import oracle as O
    w = {k: X.make_weight(cfg, k, seed) for k in ("t_w1", "t_b1", "t_w2", "t_b2", "a_w1", "a_b1", "a_w2",
                                                   "a_b2", "mod_w", "mod_b", "head_w", "head_b", "head_tab",
                                                   "pe_w", "pe_b", "out_w", "out_b")}
    per_block = ("blk_mod", "qkv_w", "qkv_b", "o_w", "o_b", "f1_w", "f1_b", "f2_w", "f2_b")
    if cfg.d_ctx:
        per_block += ("ca_ln_w", "ca_ln_b", "ca_q_w", "ca_q_b", "ca_kv_w", "ca_kv_b", "ca_o_w", "ca_o_b")
    for k in per_block:
        w[k] = X.make_weight(cfg, k, seed, block=0)[None]
    m = O.OracleModel(cfg, w)
    mods, _ = m.cond(0.75, np.array([0.1, -0.2]))
    L, d, H, hd = cfg.tokens, cfg.d_model, cfg.n_heads, cfg.head_dim
    R = O.to_bf16 if cfg.dtype == "bf16" else (lambda a: a)
    x = R(X.random_tensor(seed, "bench/x", (L, d)).astype(np.float64))
    past_k = [R(X.random_tensor(seed, f"bench/k{i}", (L, H, hd)).astype(np.float64))
              for i in range(cfg.kv_window - 1)]
    past_v = [R(X.random_tensor(seed, f"bench/v{i}", (L, H, hd)).astype(np.float64))
              for i in range(cfg.kv_window - 1)]
    pos = O.group_token_positions(cfg.groups, cfg.frames, cfg.kv_window)
    ctx = None
    if cfg.d_ctx:
        tokens = X.random_tensor(seed, "bench/ctx", (cfg.max_ctx, cfg.d_ctx)).astype(np.float64)
    t0 = time.perf_counter()
    if cfg.d_ctx:
        ctx = m.context_kv(0, tokens)
    m.block(0, x, mods[0], past_k, past_v, pos, ctx)
    return time.perf_counter() - t0


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    cfg = workload_cfg(args)
    passes = cfg.n_blocks * (cfg.n_steps + (1 if cfg.kv_period == 0 else 1.0 / cfg.kv_period))
    times = []
    for i in range(args.warmup + args.steps):
        t = oracle_block_sample(cfg, seed=i)
        if i >= args.warmup:
            times.append(t)
    t_block = sum(times) / len(times)
    chunk_s = t_block * passes
    v = 1.0 / chunk_s
    cores = os.cpu_count()
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "chunks/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": chunk_s * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_of(cfg, args),
            "cpu_baseline": {"kind": "oracle", "value": v, "unit": "chunks/s", "cores": cores,
                             "sample": f"each step = one oracle block forward at full ring ({cfg.tokens} "
                                       f"queries x {cfg.kv_window * cfg.tokens} keys, fp64 numpy); "
                                       f"chunk time = mean step time x {passes} block-passes "
                                       f"(all blocks computed)"},
            "e2e": {"value": v, "unit": "chunks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def workload_cfg(args):
    """The named workload with the --view-groups / --kv-period overrides."""
    cfg = WORKLOADS[args.workload]
    if args.view_groups:
        groups = tuple(tuple(int(v) for v in g.split("x")) for g in args.view_groups.split(","))
        cfg = cfg.replace(name=f"{cfg.name}_groups_{args.view_groups}", view_groups=groups,
                          n_cams=sum(g[0] for g in groups), grid_h=groups[0][1], grid_w=groups[0][2])
    if args.kv_period:
        cfg = cfg.replace(name=f"{cfg.name}_kvperiod{args.kv_period}", kv_period=args.kv_period)
    if args.xattn:
        cfg = cfg.replace(name=f"{cfg.name}_xattn{args.xattn}", d_ctx=cfg.d_model, max_ctx=args.xattn)
    return cfg


def has_kv_pass(cfg, n: int) -> bool:
    """Chunk n ends with a KV-update pass (every chunk when kv_period = 0)."""
    P = cfg.kv_period
    return P == 0 or n % P == P - 1


def config_of(cfg, args):
    return {"workload": cfg.name, "blocks": cfg.n_blocks, "d_model": cfg.d_model,
            "heads": f"{cfg.n_heads}x{cfg.head_dim}", "d_ffn": cfg.d_ffn,
            "tokens_per_chunk": cfg.tokens, "kv_window_chunks": cfg.kv_window,
            "keys_max": cfg.kv_window * cfg.tokens,
            "passes_per_chunk": cfg.n_steps + 1 if cfg.kv_period == 0 else
            f"{cfg.n_steps} + a KV-update pass every {cfg.kv_period} chunks",
            "view_groups": [list(g) for g in cfg.groups],
            "cross_attention": None if cfg.d_ctx == 0 else
            {"d_ctx": cfg.d_ctx, "max_ctx": cfg.max_ctx, "tokens_per_chunk": "3/4 max_ctx .. max_ctx"},
            "gate": {"tau_floor": args.tau_floor, "tau_dev": args.tau_dev, "other": "Table 1 defaults"},
            "l2": "not flushed: per-chunk working set (KV ring + residual cache + weights) > 129 MB L2",
            "parallelism": f"replicas x{args.gpus}"}


# --------------------------------------------------------------- GPU arm
def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
        return
    if args.sweep:
        sweep(args)
        return
    import torch
    from paper_2604_20289_gb300 import xcache as xb

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    cfg = workload_cfg(args)
    n_total = args.warmup + args.steps
    traj = X.Trajectory(cfg, n_chunks=n_total)
    w = X.make_weights(cfg)
    dev = torch.device("cuda", local)
    noise = torch.stack([torch.from_numpy(traj.noise(n)) for n in range(n_total)]).to(dev)
    clean = torch.stack([torch.from_numpy(traj.clean(n)) for n in range(n_total)]).to(dev)
    acts = [traj.action(n) for n in range(n_total)]
    ctx_tok = [torch.from_numpy(traj.context(n)).to(dev) for n in range(n_total)] if cfg.d_ctx else None
    stream = torch.cuda.current_stream()
    xc = xb.XCache(cfg, w, stream=stream)
    L, C, S = cfg.tokens, cfg.c_latent, cfg.n_steps
    x = torch.empty(L, C, device=dev)
    v = torch.empty_like(x)

    def chunk(n, gate):
        if ctx_tok is not None:
            xc.set_context(ctx_tok[n])
        x.copy_(noise[n])
        for t in range(S):
            xc.chunk_step(x, acts[n], SIGMAS[t], t, False, gate, v_out=v, want_stats=False)
            xc.euler(x, v, SIGMAS[t + 1] - SIGMAS[t])
        if has_kv_pass(cfg, n):
            xc.chunk_step(clean[n], acts[n], 0.0, S, True, gate, want_stats=False)

    # kind of every timed pass, in issue order: True = KV-update pass
    kv_of_pass = [p for n in range(args.warmup, n_total) for p in [False] * S + [True] * has_kv_pass(cfg, n)]

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    def timed(gate, profile: bool):
        xc.reset()
        for n in range(args.warmup):
            chunk(n, gate)
        if profile:
            xc.profile_start(kinds=("attn",), capacity=cfg.n_blocks * (S + 1) * args.steps + 16)
        barrier()
        l0 = xc.launch_count
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
        ev[0].record(stream)
        for i, n in enumerate(range(args.warmup, n_total)):
            chunk(n, gate)
            ev[i + 1].record(stream)
        barrier()
        ms = ev[0].elapsed_time(ev[-1])
        per_chunk = [ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)]
        launches = xc.launch_count - l0
        recs = xc.profile_stop() if profile else []
        ms = max_over_ranks(ms, world, dev)
        return ms, launches, recs, per_chunk

    gate = xb.gate_params(tau_floor=args.tau_floor, tau_dev=args.tau_dev)
    if args.calibrate:
        calibrate(xc, chunk, cfg, args)
        return

    # Timed runs without profiling (the per-pass block loop then replays its
    # CUDA graphs); attention launch times and decisions come from separate
    # profiled runs of the same chunks (decisions are deterministic).
    sampler = ClockSampler(local)
    sampler.start()
    ms_x, launches, _, pc_x = timed(gate, profile=False)
    clocks = sampler.stop()
    ms_all, _, _, pc_all = timed(xb.gate_params(enabled=0), profile=False)
    _, _, recs, _ = timed(gate, profile=True)
    _, _, recs_all, _ = timed(xb.gate_params(enabled=0), profile=True)
    xc.sync()

    # skip rates over the timed chunks (decisions logged per (pass, block))
    dec = np.array([r["decision"] for r in recs])
    den = np.array([not kv_of_pass[r["pass_seq"]] for r in recs])
    skip_all = float(np.mean(dec == xb.XC_DEC_SKIP)) if len(dec) else 0.0
    skip_den = float(np.mean(dec[den] == xb.XC_DEC_SKIP)) if den.any() else 0.0

    # roofline of the dominant kernel (attention: ~91% of a recomputed block's flops)
    peaks, peak_src = measured_peaks()
    work = [r for r in recs + recs_all if r["decision"] != xb.XC_DEC_SKIP]
    flops = [4.0 * L * r["n_keys"] * cfg.d_model for r in work]
    avg_ms = float(np.mean([r["ms"] for r in work]))
    achieved = float(np.mean(flops)) / (avg_ms * 1e-3) / 1e12
    peak = float(peaks.get("bf16_tflops_sustained", peaks.get("bf16_tflops")))
    trec = traffic_record(f"attn_tc_kernel<{cfg.head_dim}>")
    roofline = {"kernel": f"attn_tc_kernel<{cfg.head_dim}>", "bound": "tensor", "achieved": achieved,
                "peak": peak, "unit": "TFLOP/s", "frac": achieved / peak,
                "peak_source": f"bf16_tflops_sustained {peak_src}",
                "traffic": None if trec is None else trec["bytes_per_launch"],
                "algorithmic_flops_per_launch": float(np.mean(flops)), "avg_launch_ms": avg_ms,
                "launches": len(work)}

    n_chunks = args.steps * world
    value = whole_job_rate(args.steps, world, ms_x * 1e-3)
    line = {"metric": METRIC, "value": value, "unit": "chunks/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_x / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": cfg.dtype, "data": "synthetic",
            "config": config_of(cfg, args),
            "skip_rate": {"all_passes": skip_all, "denoise_passes": skip_den},
            "ms_per_chunk_p50": float(np.median(pc_x)),
            "all_blocks": {"ms_per_chunk": ms_all / args.steps, "ms_per_chunk_p50": float(np.median(pc_all)),
                           "chunks_per_s": n_chunks / (ms_all * 1e-3)},
            "speedup_vs_all_blocks": ms_all / ms_x,
            "predicted_speedup": None,
            "roofline": roofline, "gpu_launches": int(launches), "clocks": clocks}
    pred, kernel_us = predicted_speedup(xc, chunk, gate, args, cfg, ms_all / args.steps)
    line["predicted_speedup"] = pred
    # warm mean per launch of each kernel kind in the all-blocks arm (us; CUDA events
    # around each launch of the profiled re-run; "attn" includes the partial merge)
    line["kernel_us"] = kernel_us

    if not args.no_e2e:
        line["e2e"] = e2e(xc, traj, acts, cfg, args, gate, world, dev)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        t_block = oracle_block_sample(cfg)
        computed = (1.0 - skip_all) * cfg.n_blocks * len(kv_of_pass) / args.steps
        line["cpu_baseline"] = {
            "kind": "oracle", "value": 1.0 / (t_block * computed), "unit": "chunks/s",
            "cores": os.cpu_count(),
            "sample": f"one oracle block forward at full ring ({L} queries x {cfg.kv_window * L} keys, "
                      f"fp64 numpy, {t_block:.1f} s) x {computed:.1f} computed block-passes per chunk "
                      f"(the GPU run's skip rate; skipped blocks counted as free)"}
    if rank == 0:
        print(json.dumps(line), flush=True)
    xc.close()
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def predicted_speedup(xc, chunk, gate, args, cfg, t_all):
    """Speedup predicted from kernel times (untimed, profiled re-run of both
    arms over the same chunks): T_all / (T_all - sum over skipped block-passes
    of (T_block - T_gate - T_reuse) + sum over gated block-passes of T_gate),
    per chunk, T_block from the all-blocks arm at the same (pass, block)."""
    from paper_2604_20289_gb300 import xcache as xb
    S = cfg.n_steps
    n_total = args.warmup + args.steps

    def run(g):
        xc.reset()
        for n in range(args.warmup):
            chunk(n, g)
        xc.profile_start(kinds=xb.KERNEL_KINDS, capacity=cfg.n_blocks * (S + 1) * args.steps * 12 + 64)
        for n in range(args.warmup, n_total):
            chunk(n, g)
        return xc.profile_stop()

    block_kinds = {"ln", "qkv", "attn", "oproj", "xattn", "ffn1", "ffn2"}
    t_block = {}
    recs_all = run(xb.gate_params(enabled=0))
    kernel_us = {}
    for kind in xb.KERNEL_KINDS:
        ms = [r["ms"] for r in recs_all if r["kind"] == kind]
        if ms:
            kernel_us[kind] = round(1e3 * float(np.mean(ms)), 2)
    for r in recs_all:
        if r["kind"] in block_kinds:
            key = (r["pass_seq"], r["block"])
            t_block[key] = t_block.get(key, 0.0) + r["ms"]
    saved = gated = 0.0
    per = {}
    for r in run(gate):
        if r["kind"] in ("gate", "reuse") and r["block"] >= 0:
            key = (r["pass_seq"], r["block"])
            d = per.setdefault(key, {"dec": r["decision"], "gate": 0.0, "reuse": 0.0})
            d[r["kind"]] += r["ms"]
    for key, d in per.items():
        if d["dec"] == xb.XC_DEC_FORCED:
            continue
        gated += d["gate"]
        if d["dec"] == xb.XC_DEC_SKIP:
            saved += t_block.get(key, 0.0) - d["gate"] - d["reuse"]
    saved /= args.steps
    gated /= args.steps
    return t_all / (t_all - saved + gated), kernel_us


def sweep(args):
    """Closed-loop stress rollout (each chunk's KV pass takes the chunk's own
    denoised latent, so caching errors can accumulate through the KV ring):
    an all-blocks reference, then one X-Cache rollout per tau_floor.  Per
    point: skip rates (denoise and KV passes), time per chunk and speedup,
    rel-L2 of every chunk's final latent against the reference rollout, and
    the per-block skip counts."""
    import torch
    from paper_2604_20289_gb300 import xcache as xb
    cfg = X.STRESS_1P3B
    N = args.sweep_chunks
    S, B = cfg.n_steps, cfg.n_blocks
    traj = X.Trajectory(cfg, X.STRESS_TRAJ, n_chunks=N)
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(0)
    noise = torch.stack([torch.from_numpy(traj.noise(n)) for n in range(N)]).to(dev)
    acts = [traj.action(n) for n in range(N)]
    stream = torch.cuda.current_stream()
    xc = xb.XCache(cfg, X.make_weights(cfg), stream=stream)
    x = torch.empty(cfg.tokens, cfg.c_latent, device=dev)
    v = torch.empty_like(x)

    def chunk(n, gate):
        x.copy_(noise[n])
        for t in range(S):
            xc.chunk_step(x, acts[n], SIGMAS[t], t, False, gate, v_out=v, want_stats=False)
            xc.euler(x, v, SIGMAS[t + 1] - SIGMAS[t])
        xc.chunk_step(x, acts[n], 0.0, S, True, gate, want_stats=False)

    def rollout(gate, ref=None):
        xc.reset()
        xc.profile_start(kinds=("ln",), capacity=N * (S + 1) * B * 2 + 64)
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(N)]
        finals, rel = [], []
        for n in range(N):
            ev[n][0].record(stream)
            chunk(n, gate)
            ev[n][1].record(stream)
            if ref is None:
                finals.append(x.clone())
            else:
                rel.append(torch.linalg.vector_norm(x - ref[n]) / torch.linalg.vector_norm(ref[n]))
        torch.cuda.synchronize()
        recs = xc.profile_stop()
        ms = [a.elapsed_time(b) for a, b in ev]
        dec = {}
        for r in recs:
            if r["block"] >= 0:
                dec[(r["pass_seq"], r["block"])] = r["decision"]
        den = [d for (ps, b), d in dec.items() if ps % (S + 1) < S]
        kv = [d for (ps, b), d in dec.items() if ps % (S + 1) == S]
        per_block = [0] * B
        for (ps, b), d in dec.items():
            if ps % (S + 1) < S and d == xb.XC_DEC_SKIP:
                per_block[b] += 1
        out = {"ms_per_chunk": float(np.mean(ms[1:])), "ms_per_chunk_p50": float(np.median(ms[1:])),
               "skip_denoise": float(np.mean([d == xb.XC_DEC_SKIP for d in den])) if den else 0.0,
               "skips_on_kv_passes": int(sum(d == xb.XC_DEC_SKIP for d in kv)),
               "per_block_denoise_skips": per_block}
        if ref is not None:
            rl = np.array([float(t) for t in rel])
            out.update({"rel_l2_mean": float(rl.mean()), "rel_l2_max": float(rl.max()),
                        "rel_l2_first20": float(rl[:20].mean()), "rel_l2_last20": float(rl[-20:].mean())})
        return out, finals

    base, ref = rollout(xb.gate_params(enabled=0))
    points = []
    for pt in args.sweep_points.split(","):
        tau, margin, dev_t = (float(t) for t in pt.split(":"))
        res, _ = rollout(xb.gate_params(tau_floor=tau, margin=margin, tau_dev=dev_t), ref=ref)
        res.update({"tau_floor": tau, "margin": margin, "tau_dev": dev_t})
        res["speedup"] = base["ms_per_chunk"] / res["ms_per_chunk"]
        points.append(res)
    line = {"sweep": cfg.name, "chunks": N, "trajectory": "rho 0.95 -> 0.5, action jump +-0.8 every 20 chunks",
            "closed_loop": True, "timing": "mean over chunks 1..N-1, CUDA events",
            "all_blocks_ms_per_chunk": base["ms_per_chunk"], "points": points}
    print(json.dumps(line), flush=True)
    xc.close()


def e2e(xc, traj, acts, cfg, args, gate, world, dev):
    """Same metric through the public API with HOST buffers: every pass
    copies its latent from pinned host memory and reads v back; the Euler
    update runs on the host."""
    import torch
    L, C, S = cfg.tokens, cfg.c_latent, cfg.n_steps
    xh = torch.empty(L, C, dtype=torch.float32).pin_memory()
    vh = torch.empty(L, C, dtype=torch.float32).pin_memory()
    ch = torch.empty(L, C, dtype=torch.float32).pin_memory()
    x_np, v_np, c_np = xh.numpy(), vh.numpy(), ch.numpy()

    def chunk(n):
        if cfg.d_ctx:
            xc.set_context(traj.context(n))
        x_np[:] = traj.noise(n)
        for t in range(S):
            xc.chunk_step(x_np, acts[n], SIGMAS[t], t, False, gate, v_out=v_np, want_stats=False)
            np.add(x_np, np.float32(SIGMAS[t + 1] - SIGMAS[t]) * v_np, out=x_np)
        if has_kv_pass(cfg, n):
            c_np[:] = traj.clean(n)
            xc.chunk_step(c_np, acts[n], 0.0, S, True, gate, want_stats=False)

    xc.reset()
    for n in range(args.warmup):
        chunk(n)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for n in range(args.warmup, args.warmup + args.steps):
        chunk(n)
    torch.cuda.synchronize()
    sec = max_over_ranks(time.perf_counter() - t0, world, dev)
    nbytes = L * C * 4
    kv = sum(has_kv_pass(cfg, n) for n in range(args.warmup, args.warmup + args.steps)) / args.steps
    ctx_b = 0.0
    if cfg.d_ctx:
        ctx_b = sum(traj.context(n).nbytes for n in range(args.warmup, args.warmup + args.steps)) / args.steps
    return {"value": whole_job_rate(args.steps, world, sec), "unit": "chunks/s",
            "h2d_bytes_per_step": (S + kv) * (nbytes + cfg.action_dim * 4) + ctx_b,
            "d2h_bytes_per_step": S * nbytes}


def calibrate(xc, chunk, cfg, args):
    """Force-compute rollout with the gate evaluated; quantiles of s_cos, d_max."""
    from paper_2604_20289_gb300 import xcache as xb
    import torch
    g = xb.gate_params(tau_floor=2.0)
    xc.reset()
    S = cfg.n_steps
    s_all, d_all = [], []
    L, C = cfg.tokens, cfg.c_latent
    traj = X.Trajectory(cfg, n_chunks=args.warmup + args.steps)
    x = torch.empty(L, C, device="cuda")
    v = torch.empty_like(x)
    for n in range(args.warmup + args.steps):
        if cfg.d_ctx:
            xc.set_context(traj.context(n))
        x.copy_(torch.from_numpy(traj.noise(n)))
        for t in range(S):
            st = xc.chunk_step(x, traj.action(n), SIGMAS[t], t, False, g, v_out=v)
            xc.euler(x, v, SIGMAS[t + 1] - SIGMAS[t])
            ok = st["decision"] == xb.XC_DEC_COMPUTE
            s_all += list(st["s_cos"][ok])
            d_all += list(st["d_max"][ok])
        if has_kv_pass(cfg, n):
            xc.chunk_step(torch.from_numpy(traj.clean(n)).cuda(), traj.action(n), 0.0, S, True, g)
    q = [0.1, 0.25, 0.5, 0.75, 0.9]
    print(json.dumps({"s_cos_q": dict(zip(map(str, q), np.quantile(s_all, q).tolist())),
                      "d_max_q": dict(zip(map(str, q), np.quantile(d_all, q).tolist())),
                      "n": len(s_all)}))


if __name__ == "__main__":
    main()
