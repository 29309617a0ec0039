"""AR rollout driver over the C ABI (Section 2.1 inference loop).

Chunk n: (cross-attention models: xc_set_context with the chunk's condition
tokens) x = eps_n; for t < S: v = xc_chunk_step(x, sigma_t, t); x += (sigma_{t+1}
- sigma_t) v (Euler step, xc_euler_update); then, on a KV-update chunk (every
chunk, or n mod P == P - 1 with kv_period P > 0), the KV-update pass on the
chunk's clean latent at sigma = 0.  Actions are replayed one chunk at a time
(closed-loop protocol, Section 3.1.3).  All arithmetic runs in the CUDA
library; this module only moves buffers and sequences calls.
"""
from __future__ import annotations

import numpy as np
import torch

from .xcache import XCache, GateParams

DEFAULT_SIGMAS = (1.0, 0.75, 0.5, 0.25, 0.0)


def rollout(xc: XCache, traj, n_chunks: int, gate: GateParams, sigmas=DEFAULT_SIGMAS,
            keep_trace: bool = False, replay=None, want_stats: bool = True,
            n_start: int = 0):
    """Runs chunks [n_start, n_start + n_chunks) of ``traj`` (an object with
    noise(n), clean(n), action(n) returning numpy arrays).  ``replay[n][t]`` (bool [B])
    switches on decision-replay for pass t of chunk n.  Returns dict(final
    [n][L, C] numpy, stats [n][t], trace [n][t] numpy [B, L, d] or None)."""
    cfg = xc.cfg
    S, L, C = cfg.n_steps, cfg.tokens, cfg.c_latent
    dev = torch.device("cuda")
    x = torch.empty(L, C, device=dev, dtype=torch.float32)
    v = torch.empty_like(x)
    clean = torch.empty_like(x)
    tr = None
    if keep_trace:
        tdt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
        tr = torch.empty(cfg.n_blocks, L, cfg.d_model, device=dev, dtype=tdt)
        xc.set_trace(tr)
    finals, stats, traces = [], [], []
    try:
        for n in range(n_start, n_start + n_chunks):
            if getattr(cfg, "d_ctx", 0) > 0:
                xc.set_context(traj.context(n))
            x.copy_(torch.from_numpy(np.ascontiguousarray(traj.noise(n), dtype=np.float32)))
            a = traj.action(n)
            st_n, tr_n = [], []
            for t in range(S):
                g = gate
                if replay is not None:
                    g = _with_replay(gate, replay[n - n_start][t])
                st_n.append(xc.chunk_step(x, a, sigmas[t], t, False, g, v_out=v, want_stats=want_stats))
                if keep_trace:
                    tr_n.append(tr.float().cpu().numpy())
                xc.euler(x, v, sigmas[t + 1] - sigmas[t])
            P = int(getattr(cfg, "kv_period", 0))
            if P == 0 or n % P == P - 1:
                clean.copy_(torch.from_numpy(np.ascontiguousarray(traj.clean(n), dtype=np.float32)))
                st_n.append(xc.chunk_step(clean, a, 0.0, S, True, gate, v_out=None, want_stats=want_stats))
            finals.append(x.cpu().numpy().astype(np.float64))
            stats.append(st_n)
            traces.append(tr_n)
    finally:
        if keep_trace:
            xc.set_trace(None)
    return dict(final=finals, stats=stats, trace=traces if keep_trace else None)


def _with_replay(gate: GateParams, skips) -> GateParams:
    import ctypes
    g = GateParams.from_buffer_copy(gate)
    arr = (ctypes.c_uint8 * len(skips))(*[1 if s else 0 for s in skips])
    g._replay_keepalive = arr
    g.replay_skip = ctypes.cast(arr, ctypes.POINTER(ctypes.c_uint8))
    return g
