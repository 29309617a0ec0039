#!/usr/bin/env python
"""Benchmark of the X-Cache chunk step on GB300.

One step = one chunk of the AR rollout: S = 4 denoising passes (each through
all B blocks, gate + reuse or recompute per block) + 1 KV-update pass, with the
Euler update between passes.  Inputs (noise, clean latents, actions) are
resident in HBM before the timed region; the per-chunk working set (KV ring,
residual cache, weights) is larger than L2.

Default workload: the 14B-class multi-camera DiT (40 blocks, d 5120, 40 heads
x 128, FFN 13824, 6 cameras x 3 frames x 20 x 36 = 12960 tokens per chunk, KV
ring of 3 chunks = 38880 keys), bf16 with fp32 accumulation, random-init
weights generated on the device by the seeded input generator, synthetic
AR(1) latents.  ``--workload small|1p3b|tiny`` selects the other shapes.

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
    ap.add_argument("--warmup", type=int, default=5,
                    help="untimed chunks first; >= 2 kv_window - 1 so that every pass signature of a "
                         "full ring has been captured into a CUDA graph before the timed region")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="14b", choices=sorted(WORKLOADS))
    ap.add_argument("--oracle-rows", default="32,256",
                    help="query-row counts of the oracle's sampled block forwards (CPU baseline)")
    ap.add_argument("--prof-chunks", type=int, default=2,
                    help="timed chunks of the profiled all-blocks re-run (per-kernel times)")
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
    ap.add_argument("--chain", action="store_true",
                    help="lazy residual chaining over runs of skipped blocks (X-Cache arm)")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--calibrate", action="store_true", help="print gate-metric quantiles and exit")
    ap.add_argument("--sweep", action="store_true",
                    help="threshold sweep on the stress rollout (1.3B shape, closed loop); prints one JSON line")
    ap.add_argument("--sweep-chunks", type=int, default=200)
    ap.add_argument("--op", default="",
                    choices=["", "gate", "reuse", "ln", "qkv", "oproj", "ffn1", "ffn2", "attn"],
                    help="time one kernel through its xc_op_* entry point at the workload's shape "
                         "(random device inputs) and print one JSON line; for per-kernel profiles")
    ap.add_argument("--iters", type=int, default=20, help="timed launches of --op (after 3 warm-up launches)")
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
class OracleSample:
    """The CPU oracle on a bounded sample of one block-pass of the workload
    (block 0's weights, a full KV ring of random keys / values, the rounding of
    the model's dtype).

    * block(R): OracleModel.block on R sampled query rows; keys and values are
      projected for every token of the chunk.  Two row counts give the
      per-row cost and the fixed cost (LN, K / V projection of all tokens), so
      a full block forward costs fixed + L x per-row.
    * gate(): the oracle's fingerprint of the block input and Eq. 5-6 against
      a cached fingerprint (Section 2.3).
    * reuse(): the reuse path round(x + r_hat) (Eq. 4)."""

    def __init__(self, cfg, seed: int = 0):
        import oracle as O
        self.O, self.cfg = O, cfg
        w = {k: X.make_weight(cfg, k, seed) for k in ("t_w1", "t_b1", "t_w2", "t_b2", "a_w1", "a_b1", "a_w2",
                                                       "a_b2", "mod_w", "mod_b", "head_w", "head_b", "head_tab",
                                                       "pe_w", "pe_b", "out_w", "out_b")}
        per_block = ("blk_mod", "qkv_w", "qkv_b", "o_w", "o_b", "f1_w", "f1_b", "f2_w", "f2_b")
        if cfg.d_ctx:
            per_block += ("ca_ln_w", "ca_ln_b", "ca_q_w", "ca_q_b", "ca_kv_w", "ca_kv_b", "ca_o_w", "ca_o_b")
        for k in per_block:
            w[k] = X.make_weight(cfg, k, seed, block=0)[None]
        self.m = O.OracleModel(cfg, w)
        self.mods, _ = self.m.cond(0.75, np.array([0.1, -0.2]))
        L, d, H, hd = cfg.tokens, cfg.d_model, cfg.n_heads, cfg.head_dim
        R = O.to_bf16 if cfg.dtype == "bf16" else (lambda a: a)
        self.R = R
        self.x = R(X.random_tensor(seed, "bench/x", (L, d)).astype(np.float64))
        self.r_hat = R(0.1 * X.random_tensor(seed, "bench/r", (L, d)).astype(np.float64))
        self.past_k = [R(X.random_tensor(seed, f"bench/k{i}", (L, H, hd)).astype(np.float64))
                       for i in range(cfg.kv_window - 1)]
        self.past_v = [R(X.random_tensor(seed, f"bench/v{i}", (L, H, hd)).astype(np.float64))
                       for i in range(cfg.kv_window - 1)]
        self.pos = O.group_token_positions(cfg.groups, cfg.frames, cfg.kv_window)
        self.ctx = None
        if cfg.d_ctx:
            self.ctx = self.m.context_kv(0, X.random_tensor(seed, "bench/ctx", (cfg.max_ctx, cfg.d_ctx))
                                         .astype(np.float64))
        self.xc = O.OracleXCache(cfg, w)
        self.act = np.array([0.3, -0.4])
        self.cached = self.xc.fingerprint(R(0.9 * self.x), self.act, 32)

    def block(self, n_rows: int) -> float:
        L = self.cfg.tokens
        rows = np.unique(np.linspace(0, L - 1, min(n_rows, L)).astype(np.int64))
        t0 = time.perf_counter()
        self.m.block(0, self.x, self.mods[0], self.past_k, self.past_v, self.pos, self.ctx, rows=rows)
        return time.perf_counter() - t0

    def gate(self) -> float:
        t0 = time.perf_counter()
        phi = self.xc.fingerprint(self.x, self.act, 32)
        self.O.gate_metrics(phi, self.cached, 1e-6)
        return time.perf_counter() - t0

    def reuse(self) -> float:
        t0 = time.perf_counter()
        self.R(self.x + self.r_hat)
        return time.perf_counter() - t0


def fit_block(samples: dict, L: int) -> dict:
    """Per-row and fixed cost of the oracle block from mean times at two
    row counts; a full forward is fixed + L x per-row."""
    (r1, t1), (r2, t2) = sorted((r, float(np.mean(t))) for r, t in samples.items())
    per_row = max((t2 - t1) / (r2 - r1), 0.0)
    fixed = max(t1 - r1 * per_row, 0.0)
    return {"rows": [r1, r2], "s_at_rows": [t1, t2], "fixed_s": fixed, "per_row_s": per_row,
            "block_s": fixed + L * per_row}


def oracle_rows(args):
    return tuple(int(v) for v in args.oracle_rows.split(","))


def run_reference(args):
    """The oracle as the reference arm: every step is a bounded sample of the
    workload (see OracleSample); steps alternate between the two row counts.
    The tiny fp32 workload instead runs whole oracle chunks (X-Cache rollout
    with the benchmark's gate), one chunk per step."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    cfg = workload_cfg(args)
    cores = os.cpu_count()
    S, B = cfg.n_steps, cfg.n_blocks
    base = {"impl": "reference", "metric": METRIC, "unit": "chunks/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": config_of(cfg, args)}
    if cfg.tokens <= 4096:
        import oracle as O
        n_total = args.warmup + args.steps
        traj = X.Trajectory(cfg, n_chunks=n_total)
        oc = O.OracleXCache(cfg, X.make_weights(cfg))
        p = O.GateParams(tau_floor=args.tau_floor, tau_dev=args.tau_dev)
        times = []
        for n in range(n_total):
            t0 = time.perf_counter()
            x = np.asarray(traj.noise(n), np.float64)
            for t in range(S):
                v, _ = oc.chunk_step(x, traj.action(n), SIGMAS[t], t, False, p)
                x = x + (SIGMAS[t + 1] - SIGMAS[t]) * v
            if oc.is_kv_chunk(n):
                oc.chunk_step(traj.clean(n), traj.action(n), 0.0, S, True, p)
            if n >= args.warmup:
                times.append(time.perf_counter() - t0)
        step_s = float(np.mean(times))
        value = 1.0 / step_s
        sample = (f"whole oracle chunks (X-Cache rollout, gate tau_floor {args.tau_floor} tau_dev "
                  f"{args.tau_dev}, fp64 numpy), one chunk per step")
    else:
        smp = OracleSample(cfg)
        r1, r2 = oracle_rows(args)
        times = {r1: [], r2: []}
        step_t = []
        for i in range(args.warmup + args.steps):
            r = r1 if i % 2 == 0 else r2
            t = smp.block(r)
            if i >= args.warmup:
                times[r].append(t)
                step_t.append(t)
        if not times[r2]:                               # one timed step: take the other count untimed
            times[r2].append(smp.block(r2))
        fit = fit_block(times, cfg.tokens)
        passes = S + (1 if cfg.kv_period == 0 else 1.0 / cfg.kv_period)
        chunk_s = passes * B * fit["block_s"]
        step_s = float(np.mean(step_t))
        value = 1.0 / chunk_s
        sample = (f"each step = one oracle block forward (fp64 numpy, block 0 weights, full ring of "
                  f"{cfg.kv_window * cfg.tokens} keys) on {r1} or {r2} sampled query rows (alternating), "
                  f"keys / values projected for all {cfg.tokens} tokens; fixed {fit['fixed_s']:.2f} s + "
                  f"{fit['per_row_s'] * 1e3:.2f} ms per query row -> {fit['block_s']:.1f} s per block "
                  f"forward; chunk = {passes:g} passes x {B} blocks, every block computed (the oracle's "
                  f"own gate decisions are not simulated at this size)")
    line = dict(base, value=value, ms_per_step=step_s * 1e3,
                cpu_baseline={"kind": "oracle", "value": value, "unit": "chunks/s", "cores": cores,
                              "sample": sample},
                e2e={"value": value, "unit": "chunks/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0})
    print(json.dumps(line), flush=True)


def cpu_baseline(cfg, args, counts: dict) -> dict:
    """The oracle's time for one chunk of the workload on this host, from a
    bounded sample: block forwards at two query-row counts (fitted to a full
    forward), the gate and the reuse path, charged per block-pass with the
    GPU run's decisions."""
    smp = OracleSample(cfg)
    r1, r2 = oracle_rows(args)
    smp.block(r1)                                   # untimed: first-call costs (thread pools, page faults)
    times = {r1: [smp.block(r1)], r2: [smp.block(r2)]}
    fit = fit_block(times, cfg.tokens)
    t_gate = min(smp.gate() for _ in range(2))
    t_reuse = min(smp.reuse() for _ in range(2))
    chunk_s = (counts["computed"] * fit["block_s"] + counts["gate_launches"] * t_gate
               + counts["skipped"] * t_reuse)
    return {"kind": "oracle", "value": 1.0 / chunk_s, "unit": "chunks/s", "cores": os.cpu_count(),
            "sample": f"oracle (fp64 numpy) block forward on {r1} and {r2} sampled query rows with all "
                      f"{cfg.tokens} tokens' keys / values, fitted to {fit['block_s']:.1f} s per full forward; "
                      f"gate {t_gate:.2f} s, reuse {t_reuse:.2f} s; per chunk {counts['computed']:.1f} "
                      f"computed block-passes, {counts['gate_launches']:.1f} gate evaluations, "
                      f"{counts['skipped']:.1f} reuses (this run's decisions)",
            "fit": fit}


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
            "gate": {"tau_floor": args.tau_floor, "tau_dev": args.tau_dev, "other": "Table 1 defaults",
                     "lazy_chaining": bool(getattr(args, "chain", False))},
            "l2": "not flushed: per-chunk working set (KV ring + residual cache + weights) > 129 MB L2",
            "parallelism": f"replicas x{args.gpus}"}


# --------------------------------------------------------------- GPU arm
# Algorithmic work per launch of each kernel kind (bytes for the bandwidth-bound
# kernels, FLOP for the contractions) and the roofline it is held against.
def kernel_work(cfg, kind: str, n_keys: int) -> tuple[str, float]:
    L, d, F = cfg.tokens, cfg.d_model, cfg.d_ffn
    es = 2 if cfg.dtype == "bf16" else 4
    if kind == "attn":
        return "tensor", 4.0 * L * n_keys * d
    if kind == "qkv":
        return "tensor", 2.0 * L * 3 * d * d
    if kind == "oproj":
        return "tensor", 2.0 * L * d * d
    if kind in ("ffn1", "ffn2"):
        return "tensor", 2.0 * L * d * F
    if kind == "gate":
        return "hbm", float(L * d * es)                 # reads the block input once
    if kind == "reuse":
        return "hbm", float(3 * L * d * es)             # x, r_hat in; x + r_hat out
    if kind == "ln":
        return "hbm", float(2 * L * d * es)
    C = cfg.c_latent
    if kind == "embed":                                 # latent + pe_w in, X0 out
        return "hbm", float(L * C * 4 + C * d * 4 + L * d * es)
    if kind == "head":                                  # block output + W_out in, velocity out
        return "hbm", float(L * d * es + d * C * 4 + L * C * 4)
    if kind == "cond":                                  # the conditioning MLP weights (fp32) + per-block tables
        B, tf, A = cfg.n_blocks, cfg.t_freq, cfg.action_dim
        return "hbm", float(4 * (tf * d + A * d + 2 * d * d + 6 * d * d + 2 * d * d) + 2 * 4 * B * 6 * d)
    return "", 0.0


def choose_peak(peaks: dict, clocks: dict) -> tuple[float, str]:
    """Burst bf16 peak when the SM clock held its maximum with no power cap
    during the timed region, else the sustained (power-capped) peak."""
    capped = "sw_power_cap" in (clocks.get("reasons") or [])
    mhz, mx = clocks.get("sm_mhz"), clocks.get("sm_max_mhz")
    low = mhz is not None and mx is not None and mhz < 0.97 * mx
    if capped or low:
        return float(peaks["bf16_tflops_sustained"]), "bf16_tflops_sustained"
    return float(peaks["bf16_tflops"]), "bf16_tflops"


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
        return
    if args.sweep:
        sweep(args)
        return
    if args.op:
        op_bench(args)
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
    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream()
    # weights: the seeded generator run on the device (same values as the
    # numpy generator the oracle uses), handed to xc_init as device pointers
    w = X.make_weights_torch(cfg, dev)
    xc = xb.XCache(cfg, w, stream=stream)
    del w
    torch.cuda.empty_cache()
    noise = torch.stack([torch.from_numpy(traj.noise(n)) for n in range(n_total)]).to(dev)
    clean = torch.stack([torch.from_numpy(traj.clean(n)) for n in range(n_total)]).to(dev)
    acts = [traj.action(n) for n in range(n_total)]
    ctx_tok = [torch.from_numpy(traj.context(n)).to(dev) for n in range(n_total)] if cfg.d_ctx else None
    L, C, S, B = cfg.tokens, cfg.c_latent, cfg.n_steps, cfg.n_blocks
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

    # kind of every pass of chunks [warmup, warmup + k), in issue order: True = KV-update pass
    def kv_passes(k):
        return [p for n in range(args.warmup, args.warmup + k) for p in [False] * S + [True] * has_kv_pass(cfg, n)]

    # pass index t within its chunk (S = the KV-update pass) of the same passes
    def pass_index(k):
        return [t for n in range(args.warmup, args.warmup + k) for t in list(range(S)) + [S] * has_kv_pass(cfg, n)]

    def barrier():
        torch.cuda.synchronize()
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    def timed(gate, n_timed: int, profile: bool):
        """W untimed chunks, then n_timed chunks bracketed by events on the
        library's stream (synchronised, barrier on both sides)."""
        xc.reset()
        for n in range(args.warmup):
            chunk(n, gate)
        if profile:
            xc.profile_start(kinds=xb.KERNEL_KINDS, capacity=B * (S + 1) * n_timed * 14 + 64)
        barrier()
        l0 = xc.launch_count
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(n_timed + 1)]
        ev[0].record(stream)
        for i, n in enumerate(range(args.warmup, args.warmup + n_timed)):
            chunk(n, gate)
            ev[i + 1].record(stream)
        barrier()
        ms = ev[0].elapsed_time(ev[-1])
        per_chunk = [ev[i].elapsed_time(ev[i + 1]) for i in range(n_timed)]
        launches = xc.launch_count - l0
        recs = xc.profile_stop() if profile else []
        ms = max_over_ranks(ms, world, dev)
        return ms, launches, recs, per_chunk

    gate = xb.gate_params(tau_floor=args.tau_floor, tau_dev=args.tau_dev, chain=int(args.chain))
    if args.calibrate:
        calibrate(xc, chunk, cfg, args)
        return

    # Timed runs without profiling (the per-pass block loop replays its CUDA
    # graphs).  Per-launch kernel times and the gate decisions come from
    # profiled re-runs of the same chunks (decisions are deterministic): the
    # X-Cache arm over all timed chunks, the all-blocks arm over a few (its
    # work per chunk does not change once the ring is full).
    sampler = ClockSampler(local)
    sampler.start()
    ms_x, launches, _, pc_x = timed(gate, args.steps, profile=False)
    clocks = sampler.stop()
    ms_all, _, _, pc_all = timed(xb.gate_params(enabled=0), args.steps, profile=False)
    n_prof_all = max(1, min(args.prof_chunks, args.steps))
    _, _, recs, _ = timed(gate, args.steps, profile=True)
    _, _, recs_all, _ = timed(xb.gate_params(enabled=0), n_prof_all, profile=True)
    xc.sync()

    # decisions per (pass, block) of the timed chunks, skip rates, per-chunk counts
    kv_of_pass = kv_passes(args.steps)
    dec = {}
    for r in recs:
        if r["block"] >= 0:
            dec[(r["pass_seq"], r["block"])] = r["decision"]
    d_all = np.array(list(dec.values()))
    d_den = np.array([dd for (ps, b), dd in dec.items() if not kv_of_pass[ps]])
    skip_all = float(np.mean(d_all == xb.XC_DEC_SKIP)) if len(d_all) else 0.0
    skip_den = float(np.mean(d_den == xb.XC_DEC_SKIP)) if len(d_den) else 0.0
    counts = {"computed": float(np.sum(d_all != xb.XC_DEC_SKIP)) / args.steps,
              "skipped": float(np.sum(d_all == xb.XC_DEC_SKIP)) / args.steps,
              "gate_launches": sum(1 for r in recs if r["kind"] == "gate") / args.steps}

    # per-kernel warm launch times and roofline fractions (computed launches
    # of both arms; the reuse path over launches of skipped blocks; the gate
    # over launches that evaluated or refreshed the fingerprint)
    peaks, peak_src = measured_peaks()
    tflops_peak, tflops_name = choose_peak(peaks, clocks)
    kernels = {}
    for kind in xb.KERNEL_KINDS:
        rs = [r for r in recs + recs_all if r["kind"] == kind]
        if kind == "reuse":
            rs = [r for r in rs if r["decision"] == xb.XC_DEC_SKIP]
        elif kind != "gate":
            rs = [r for r in rs if r["decision"] != xb.XC_DEC_SKIP]
        if not rs:
            continue
        ms_k = float(np.mean([r["ms"] for r in rs]))
        bound, work = kernel_work(cfg, kind, int(np.mean([r["n_keys"] for r in rs])))
        ent = {"us": round(ms_k * 1e3, 2), "launches": len(rs)}
        if bound == "tensor":
            ach = work / (ms_k * 1e-3) / 1e12
            ent.update({"TFLOP/s": round(ach, 1), "frac": round(ach / tflops_peak, 3)})
        elif bound == "hbm":
            ach = work / (ms_k * 1e-3) / 1e9
            ent.update({"GB/s": round(ach, 1), "frac": round(ach / float(peaks["hbm_gbs"]), 3)})
        kernels[kind] = ent

    # roofline of the dominant kernel (attention: most of a recomputed block's flops)
    work = [r for r in recs + recs_all if r["kind"] == "attn" and r["decision"] != xb.XC_DEC_SKIP]
    flops = [4.0 * L * r["n_keys"] * cfg.d_model for r in work]
    avg_ms = float(np.mean([r["ms"] for r in work]))
    achieved = float(np.mean(flops)) / (avg_ms * 1e-3) / 1e12
    kname = f"attn_tc_kernel<{cfg.head_dim}>" if cfg.dtype == "bf16" else "attn_simt"
    trec = traffic_record(kname)
    roofline = {"kernel": kname, "bound": "tensor", "achieved": achieved, "peak": tflops_peak,
                "unit": "TFLOP/s", "frac": achieved / tflops_peak,
                "peak_source": f"{tflops_name} {peak_src} (chosen by the timed region's clocks)",
                "frac_of_burst": achieved / float(peaks["bf16_tflops"]),
                "frac_of_sustained": achieved / float(peaks["bf16_tflops_sustained"]),
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
            "predicted_speedup": predicted_speedup(recs, recs_all, ms_all / args.steps, pass_index(args.steps),
                                                   pass_index(n_prof_all), args.steps, n_prof_all),
            "roofline": roofline, "kernels": kernels, "gpu_launches": int(launches), "clocks": clocks}

    if not args.no_e2e:
        line["e2e"] = e2e(xc, traj, acts, cfg, args, gate, world, dev)
    xc.close()
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg, args, counts)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def predicted_speedup(recs, recs_all, t_all, t_of, t_of_all, n_chunks, n_chunks_all):
    """Speedup predicted from kernel times: T_all / (T_all - sum over skipped
    block-passes of (T_block - T_gate - T_reuse) + sum over gated block-passes
    of T_gate), per chunk.  T_block(t, b) is the mean time of block b's
    kernels in pass t (t_of / t_of_all map a profiled pass to t) of the
    profiled all-blocks chunks; gate and reuse times and the decisions come
    from the profiled X-Cache chunks."""
    from paper_2604_20289_gb300 import xcache as xb
    block_kinds = {"ln", "qkv", "attn", "oproj", "xattn", "ffn1", "ffn2"}
    tb, cnt = {}, {}
    for r in recs_all:
        if r["kind"] in block_kinds and r["pass_seq"] < len(t_of_all):
            key = (t_of_all[r["pass_seq"]], r["block"])
            tb[key] = tb.get(key, 0.0) + r["ms"]
    for ps in range(len(t_of_all)):
        cnt[t_of_all[ps]] = cnt.get(t_of_all[ps], 0) + 1
    for (t, b) in tb:
        tb[(t, b)] /= cnt[t]
    per = {}
    for r in recs:
        if r["kind"] in ("gate", "reuse", "chain") and r["block"] >= 0:
            key = (r["pass_seq"], r["block"])
            d = per.setdefault(key, {"dec": r["decision"], "gate": 0.0, "reuse": 0.0})
            d["gate" if r["kind"] == "gate" else "reuse"] += r["ms"]
    saved = gated = 0.0
    for (ps, b), d in per.items():
        if d["dec"] == xb.XC_DEC_FORCED:
            continue
        gated += d["gate"]
        if d["dec"] == xb.XC_DEC_SKIP:
            saved += tb.get((t_of[ps], b), 0.0) - d["gate"] - d["reuse"]
    saved /= n_chunks
    gated /= n_chunks
    del n_chunks_all
    return t_all / (t_all - saved + gated)


def op_bench(args):
    """One kernel of the chunk step at the workload's shape, through its
    operator entry point, on seeded random device inputs.  The inputs each
    launch reads rotate over enough copies to exceed twice the L2 (129 MB),
    so every launch reads from HBM.  The GPU is first held busy (a device
    sleep) while 3 + iters launches are queued behind a start event; the
    mean time per launch between the events after the 3 warm-up launches is
    reported (back-to-back launches on one stream; the gate's includes the
    ticket reset its entry point issues)."""
    import torch
    from paper_2604_20289_gb300 import xcache as xb
    cfg = workload_cfg(args)
    torch.cuda.set_device(0)
    dev = torch.device("cuda", 0)
    gen = torch.Generator(device=dev)
    gen.manual_seed(0)
    L, d, F, H, hd = cfg.tokens, cfg.d_model, cfg.d_ffn, cfg.n_heads, cfg.head_dim
    dt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    L2 = 129 << 20

    def rnd(*shape, std=1.0, dtype=dt):
        return (torch.randn(*shape, device=dev, generator=gen) * std).to(dtype)

    def copies(nbytes):
        return max(1, -(-2 * L2 // max(nbytes, 1)))

    keys = cfg.kv_window * L
    peaks, _ = measured_peaks()
    k = args.op
    es = 2 if cfg.dtype == "bf16" else 4
    if k in ("qkv", "oproj", "ffn1", "ffn2"):
        N, K = {"qkv": (3 * d, d), "oproj": (d, d), "ffn1": (F, d), "ffn2": (d, F)}[k]
        nc = copies((L * K + N * K) * es)
        As, Wts = [rnd(L, K) for _ in range(nc)], [rnd(N, K, std=K ** -0.5) for _ in range(nc)]
        bias, gate = rnd(N, std=0.05, dtype=torch.float32), rnd(N, std=0.1, dtype=torch.float32)
        out = torch.empty(L, N, device=dev, dtype=dt)
        resid, xin, rhat = rnd(L, N), rnd(L, N), torch.empty(L, N, device=dev, dtype=dt)
        epi = {"qkv": xb.XC_EPI_BIAS, "oproj": xb.XC_EPI_RESID_GATE, "ffn1": xb.XC_EPI_GELU,
               "ffn2": xb.XC_EPI_RESID_CACHE}[k]
        if k == "qkv":
            q, kk, vv = (torch.empty(L, d, device=dev, dtype=dt) for _ in range(3))
            G = cfg.groups[0]

            def launch(i):
                xb.op_qkv_rope(cfg.dtype, G[0], cfg.frames, G[1], G[2], 1, hd, cfg.rope_theta, As[i % nc],
                               Wts[i % nc], bias, q, kk, vv)
        else:
            def launch(i):
                xb.op_linear(cfg.dtype, epi, As[i % nc], Wts[i % nc], bias, out, gate=gate, resid=resid, xin=xin,
                             rhat=rhat if epi == xb.XC_EPI_RESID_CACHE else None)
        work, unit = 2.0 * L * N * K, "TFLOP/s"
        shape = {"M": L, "N": N, "K": K}
    elif k == "attn":
        nc = copies(2 * keys * d * es)
        q = rnd(L, d)
        kvs = [(rnd(keys, d), rnd(keys, d)) for _ in range(nc)]
        o = torch.empty(L, d, device=dev, dtype=dt)
        nb = xb.op_attention_workspace_bytes(cfg.dtype, hd)
        ws = torch.empty(max(nb, 1), dtype=torch.uint8, device=dev) if nb else None

        def launch(i):
            xb.op_attention(cfg.dtype, H, hd, q, kvs[i % nc][0], kvs[i % nc][1], o, workspace=ws)
        work, unit = 4.0 * L * keys * d, "TFLOP/s"
        shape = {"Lq": L, "keys": keys, "heads": H, "head_dim": hd}
    elif k == "ln":
        nc = copies(2 * L * d * es)
        xs, outs = [rnd(L, d) for _ in range(nc)], [torch.empty(L, d, device=dev, dtype=dt) for _ in range(nc)]
        sh, sc = rnd(d, std=0.1, dtype=torch.float32), rnd(d, std=0.1, dtype=torch.float32)

        def launch(i):
            xb.op_ln_mod(cfg.dtype, xs[i % nc], sh, sc, outs[i % nc])
        work, unit = 2.0 * L * d * es, "GB/s"
        shape = {"M": L, "d": d}
    elif k == "reuse":
        nc = copies(3 * L * d * es)
        xs = [rnd(L, d) for _ in range(nc)]
        rs = [rnd(L, d, std=0.1) for _ in range(nc)]
        outs = [torch.empty(L, d, device=dev, dtype=dt) for _ in range(nc)]

        def launch(i):
            xb.op_residual_reuse(cfg.dtype, xs[i % nc], rs[i % nc], outs[i % nc])
        work, unit = 3.0 * L * d * es, "GB/s"
        shape = {"n": L * d}
    else:                                                # gate
        G = cfg.groups[0]
        V, npc = G[0], cfg.frames * G[1] * G[2]
        nc = copies(V * npc * d * es)
        xs = [rnd(V * npc, d) for _ in range(nc)]
        kfp = 32
        rows = torch.tensor([[c * npc + (2 * j + 1) * npc // (2 * kfp) for j in range(kfp)] for c in range(V)],
                            dtype=torch.int32, device=dev)
        phi = rnd(2, V * kfp * d + V * d, dtype=torch.float32)
        pa = torch.zeros(2, 8, device=dev)
        cell = torch.frombuffer(bytearray(bytes(xb.GateCell(0.97, 1, 0, 1, 0))), dtype=torch.uint8).to(dev)
        flag = torch.zeros(1, dtype=torch.uint8, device=dev)
        stats = torch.zeros(3, device=dev)
        ws = torch.zeros(xb.op_gate_workspace_bytes(cfg.dtype, V, npc, d), dtype=torch.uint8, device=dev)
        gp = xb.gate_params(tau_floor=0.9, tau_dev=4.0)
        act = np.array([0.5, -0.4], np.float32)

        def launch(i):
            xb.op_gate(cfg.dtype, V, npc, xs[i % nc], rows, phi, pa, cell, act, 1, 1, gp, flag, stats[0:1],
                       stats[1:2], stats[2:3], ws)
        work, unit = float(V * npc * d * es), "GB/s"
        shape = {"cams": V, "tokens_per_cam": npc, "d": d}
    stream = torch.cuda.current_stream()
    launch(0)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    torch.cuda._sleep(int(2e8))                    # ~0.1 s of device time while the launches are queued
    for i in range(3):
        launch(1 + i)
    e0.record(stream)
    for i in range(args.iters):
        launch(4 + i)
    e1.record(stream)
    e1.synchronize()
    assert xb.op_device_error() == 0
    ms = e0.elapsed_time(e1) / args.iters
    ach = work / (ms * 1e-3) / (1e12 if unit == "TFLOP/s" else 1e9)
    peak = float(peaks["bf16_tflops"] if unit == "TFLOP/s" else peaks["hbm_gbs"])
    print(json.dumps({"op": k, "workload": cfg.name, "shape": shape, "us_per_launch": ms * 1e3, "work": work,
                      unit: ach, "peak": peak, "frac": ach / peak, "iters": args.iters, "input_copies": nc,
                      "timing": "CUDA events around back-to-back launches queued behind a device sleep"}),
          flush=True)


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
    xc = xb.XCache(cfg, X.make_weights_torch(cfg, dev), stream=stream)
    torch.cuda.empty_cache()
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
