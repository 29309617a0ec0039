"""Seeded synthetic inputs for the X-Cache chunk step.

This module is the only code shared by the CPU oracle (``oracle/``) and the
GPU path (``paper_2604_20289_gb300``).  It holds model shapes, weights,
latent trajectories and action streams -- never any of the method's
arithmetic (no block, no gate, no fingerprint).

Random numbers come from one counter-based generator so that any tensor (or
any slice of it) can be regenerated independently on any machine:

* SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number
  generators", OOPSLA 2014): state_i = key + (i + 1) * 0x9E3779B97F4A7C15,
  output = mix(state_i) with the published 64-bit finaliser.
* Box-Muller (Box & Muller 1958): z = sqrt(-2 ln u1) * cos(2 pi u2) with u1,
  u2 drawn from counters 2i and 2i+1, each a 53-bit uniform in (0, 1).

The paper's evaluation data (an internal X-World test split of 264-frame,
7-camera clips, Section 3.1.3) is not available; the inputs below stand in
for it with the same structure: a multi-camera latent grid per chunk, latents
that drift slowly from chunk to chunk (AR(1) in the chunk index), and a smooth
2-d action stream (steer, accel) replayed one chunk at a time.
"""
from __future__ import annotations

import dataclasses
import math
import os
from concurrent.futures import ThreadPoolExecutor
from dataclasses import dataclass

import numpy as np

_GAMMA = np.uint64(0x9E3779B97F4A7C15)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def _mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 output function (wrapping uint64 arithmetic)."""
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        return z ^ (z >> np.uint64(31))


def _stream_key(seed: int, name: str) -> np.uint64:
    """64-bit key of a named stream: SplitMix64 of the seed folded with an
    FNV-1a hash of the stream name."""
    h = 0xCBF29CE484222325
    for ch in name.encode():
        h = ((h ^ ch) * 0x100000001B3) & 0xFFFFFFFFFFFFFFFF
    k = np.array([(seed * 0x9E3779B97F4A7C15 + h) & 0xFFFFFFFFFFFFFFFF], dtype=np.uint64)
    return _mix64(k)[0]


def uniform(seed: int, name: str, n: int, offset: int = 0) -> np.ndarray:
    """n uniforms in (0, 1) from counters [offset, offset + n) of a stream."""
    key = _stream_key(seed, name)
    i = np.arange(offset, offset + n, dtype=np.uint64)
    with np.errstate(over="ignore"):
        s = key + (i + np.uint64(1)) * _GAMMA
    bits = _mix64(s) >> np.uint64(11)
    return (bits.astype(np.float64) + 0.5) * (1.0 / 9007199254740992.0)


def normal(seed: int, name: str, n: int, offset: int = 0) -> np.ndarray:
    """n standard normals; normal j uses uniforms 2(offset+j), 2(offset+j)+1.
    Large requests are filled in parallel blocks (numpy releases the GIL);
    the values do not depend on the number of threads."""
    out = np.empty(n, dtype=np.float64)
    step = 1 << 20

    def fill(a: int):
        m = min(step, n - a)
        u = uniform(seed, name, 2 * m, 2 * (offset + a))
        out[a:a + m] = np.sqrt(-2.0 * np.log(u[0::2])) * np.cos(2.0 * math.pi * u[1::2])

    starts = range(0, n, step)
    if n <= 2 * step:
        for a in starts:
            fill(a)
    else:
        with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
            list(ex.map(fill, starts))
    return out


def bf16_representable(a: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bfloat16 value (ties to even) and
    return them as float32, so that both sides see identical weights."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    b = a.view(np.uint32).astype(np.uint64)
    b = (b + np.uint64(0x7FFF) + ((b >> np.uint64(16)) & np.uint64(1))) & np.uint64(0xFFFF0000)
    return b.astype(np.uint32).view(np.float32)


# --------------------------------------------------------------------------
# Model shapes
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class ModelCfg:
    """Shape of the synthetic multi-camera causal DiT.

    A chunk holds ``n_cams * frames * grid_h * grid_w`` tokens, ordered
    (camera, frame, h, w) row-major.  ``kv_window`` counts ring slots
    including the current chunk.

    ``view_groups`` (optional) replaces the single camera grid with groups of
    cameras that share a grid shape: a tuple of (cameras, grid_h, grid_w);
    the groups' tokens follow one another in that order, each group camera by
    camera, and ``n_cams`` is then the total camera count.  ``kv_period`` P
    > 0 makes every P-th chunk (n mod P == P - 1) the one whose clean latent
    feeds the KV-update pass; 0 runs that pass after every chunk.  ``d_ctx``
    > 0 adds a cross-attention layer to every block, attending to up to
    ``max_ctx`` condition tokens of width ``d_ctx`` per chunk."""
    name: str
    n_blocks: int
    d_model: int
    n_heads: int
    head_dim: int
    d_ffn: int
    n_cams: int
    frames: int
    grid_h: int
    grid_w: int
    kv_window: int
    n_chunks: int
    dtype: str = "bf16"          # "f32" or "bf16"
    c_latent: int = 16
    action_dim: int = 2
    n_steps: int = 4
    t_freq: int = 256
    ln_eps: float = 1e-6
    rope_theta: float = 10000.0
    view_groups: tuple = ()
    kv_period: int = 0
    d_ctx: int = 0               # > 0: cross-attention to d_ctx-wide condition tokens
    max_ctx: int = 0             # most condition tokens a chunk may carry

    @property
    def groups(self) -> tuple:
        """((cameras, grid_h, grid_w), ...) of the view groups in token order."""
        if self.view_groups:
            return tuple(tuple(g) for g in self.view_groups)
        return ((self.n_cams, self.grid_h, self.grid_w),)

    @property
    def tokens(self) -> int:
        return sum(c * self.frames * h * w for c, h, w in self.groups)

    def replace(self, **kw) -> "ModelCfg":
        return dataclasses.replace(self, **kw)


# The workloads: a tiny fp32 model, a small 8-block model, a 1.3B-class and a
# 14B-class model on a 6-camera 3x20x36 latent grid, and a 200-chunk stress
# rollout on the 1.3B-class shape.
TINY_F32 = ModelCfg("tiny_f32_2blk_d64", 2, 64, 4, 16, 256, 2, 2, 4, 4, 3, 8, dtype="f32")
SMALL_BF16 = ModelCfg("small_bf16_8blk_d512_6cam", 8, 512, 8, 64, 2048, 6, 3, 16, 28, 4, 16)
DIT_1P3B = ModelCfg("dit1p3b_bf16_30blk_d1536_6cam", 30, 1536, 12, 128, 8960, 6, 3, 20, 36, 3, 32)
DIT_14B = ModelCfg("dit14b_bf16_40blk_d5120_6cam", 40, 5120, 40, 128, 13824, 6, 3, 20, 36, 3, 24)
STRESS_1P3B = DIT_1P3B.replace(name="stress_dit1p3b_200chunks", n_chunks=200)

# Mid-size parity shapes: several GEMM / attention tiles plus ragged tails
# (840 tokens = 6 x 128 + 72; 2520 keys = 19 x 128 + 88).
MID_HD64 = ModelCfg("mid_bf16_3blk_d256_hd64", 3, 256, 4, 64, 1024, 2, 3, 10, 14, 3, 4)
MID_HD128 = ModelCfg("mid_bf16_2blk_d256_hd128", 2, 256, 2, 128, 768, 2, 3, 10, 14, 3, 4)

# View-group parity shapes (grid_h / grid_w repeat group 0's grid): a tiny
# fp32 model with two groups whose cameras are larger than the K = 32 sample
# (232 tokens), and a bf16 model with a front / side / rear layout of 3 + 2 + 2
# cameras (Section 2.3.1; 2196 tokens = 17 x 128 + 20).
GROUPS_F32 = ModelCfg("groups_f32_2blk_d64_3cam", 2, 64, 4, 16, 256, 3, 2, 6, 8, 3, 6, dtype="f32",
                      view_groups=((2, 6, 8), (1, 4, 5)))
GROUPS_BF16 = ModelCfg("groups_bf16_2blk_d256_7cam", 2, 256, 4, 64, 1024, 7, 3, 10, 14, 3, 4,
                       view_groups=((3, 10, 14), (2, 8, 12), (2, 6, 10)))

# Cross-attention parity shapes: condition tokens of width d_ctx, up to
# max_ctx per chunk (count varying from chunk to chunk).
XATTN_F32 = TINY_F32.replace(name="xattn_f32_2blk_d64", d_ctx=32, max_ctx=24)
XATTN_BF16 = MID_HD64.replace(name="xattn_bf16_3blk_d256_hd64", d_ctx=128, max_ctx=300)
XATTN_HD128 = MID_HD128.replace(name="xattn_bf16_2blk_d256_hd128", d_ctx=256, max_ctx=160)

ALL_CFGS = {c.name: c for c in (TINY_F32, SMALL_BF16, DIT_1P3B, DIT_14B, STRESS_1P3B,
                                  MID_HD64, MID_HD128, GROUPS_F32, GROUPS_BF16, XATTN_F32, XATTN_BF16,
                                  XATTN_HD128)}


# --------------------------------------------------------------------------
# Weights (math convention y = x @ W, W stored [in, out])
# --------------------------------------------------------------------------
def weight_shapes(cfg: ModelCfg) -> dict:
    d, F, B, C, A, tf = cfg.d_model, cfg.d_ffn, cfg.n_blocks, cfg.c_latent, cfg.action_dim, cfg.t_freq
    return {
        "pe_w": (C, d), "pe_b": (d,),
        "t_w1": (tf, d), "t_b1": (d,), "t_w2": (d, d), "t_b2": (d,),
        "a_w1": (A, d), "a_b1": (d,), "a_w2": (d, d), "a_b2": (d,),
        "mod_w": (d, 6 * d), "mod_b": (6 * d,),
        "blk_mod": (B, 6, d),
        "qkv_w": (B, d, 3 * d), "qkv_b": (B, 3 * d),
        "o_w": (B, d, d), "o_b": (B, d),
        "f1_w": (B, d, F), "f1_b": (B, F),
        "f2_w": (B, F, d), "f2_b": (B, d),
        "head_w": (d, 2 * d), "head_b": (2 * d,), "head_tab": (2, d),
        "out_w": (d, C), "out_b": (C,),
        **({} if cfg.d_ctx == 0 else {
            "ca_ln_w": (B, d), "ca_ln_b": (B, d),
            "ca_q_w": (B, d, d), "ca_q_b": (B, d),
            "ca_kv_w": (B, cfg.d_ctx, 2 * d), "ca_kv_b": (B, 2 * d),
            "ca_o_w": (B, d, d), "ca_o_b": (B, d)}),
    }


BIAS_STD = 0.05
BIASES = ("pe_b", "t_b1", "t_b2", "a_b1", "a_b2", "mod_b", "qkv_b", "o_b", "f1_b", "f2_b",
          "head_b", "out_b", "ca_ln_b", "ca_q_b", "ca_kv_b", "ca_o_b")
GAINS = ("ca_ln_w",)             # 1 + N(0, BIAS_STD^2)


def _init_std(name: str, shape: tuple) -> float:
    if name in BIASES or name in GAINS:
        return BIAS_STD
    fan_in, fan_out = shape[-2], shape[-1]           # [in, out]; tables [6|2, d]
    return math.sqrt(2.0 / (fan_in + fan_out))        # Xavier-normal


def make_weight(cfg: ModelCfg, name: str, seed: int = 0, block: int | None = None) -> np.ndarray:
    """One weight tensor (float32).  With ``block`` set, only that block's
    slice of a per-block tensor is generated (same values as the full one)."""
    shape = weight_shapes(cfg)[name]
    std = _init_std(name, shape)
    if block is None:
        n = int(np.prod(shape))
        w = normal(seed, cfg.name + "/" + name, n) * std
        out_shape = shape
    else:
        per = int(np.prod(shape[1:]))
        w = normal(seed, cfg.name + "/" + name, per, offset=block * per) * std
        out_shape = shape[1:]
    if name in GAINS:
        w = 1.0 + w
    w = w.astype(np.float32).reshape(out_shape)
    return bf16_representable(w) if cfg.dtype == "bf16" else w


def make_weights(cfg: ModelCfg, seed: int = 0) -> dict:
    return {k: make_weight(cfg, k, seed) for k in weight_shapes(cfg)}


# --------------------------------------------------------------------------
# Rollout inputs: clean latents, noise, actions
# --------------------------------------------------------------------------
@dataclass(frozen=True)
class TrajectoryCfg:
    """Seeded chunk stream.  ``rho`` is the AR(1) chunk-to-chunk correlation of
    clean latents and noise; ``rho_end`` (if set) ramps it linearly; every
    ``jump_every`` chunks each action component jumps by +-``jump``."""
    rho: float = 0.95
    rho_end: float | None = None
    action_step: float = 0.05
    jump_every: int = 0
    jump: float = 0.8
    iid_noise: bool = False


STRESS_TRAJ = TrajectoryCfg(rho=0.95, rho_end=0.5, jump_every=20, jump=0.8)


def _rho_at(traj: TrajectoryCfg, n: int, n_chunks: int) -> float:
    if traj.rho_end is None or n_chunks <= 1:
        return traj.rho
    return traj.rho + (traj.rho_end - traj.rho) * n / (n_chunks - 1)


class Trajectory:
    """Iterates chunks: clean latent x_c[n], noise eps[n] ([L, C] float32) and
    action a[n] ([A] float32).  Chunk n depends only on chunks < n."""

    def __init__(self, cfg: ModelCfg, traj: TrajectoryCfg = TrajectoryCfg(), seed: int = 0,
                 n_chunks: int | None = None):
        self.cfg, self.traj, self.seed = cfg, traj, seed
        self.n_chunks = n_chunks if n_chunks is not None else cfg.n_chunks
        L, C, A = cfg.tokens, cfg.c_latent, cfg.action_dim
        self._clean, self._eps, self._act = [], [], []
        xc = eps = None
        a = None
        for n in range(self.n_chunks):
            rho = _rho_at(traj, n, self.n_chunks)
            z1 = normal(seed, f"{cfg.name}/clean/{n}", L * C).reshape(L, C)
            z2 = normal(seed, f"{cfg.name}/eps/{n}", L * C).reshape(L, C)
            if n == 0:
                xc, eps = z1, z2
                # start from a steady driving state: |a_i| in [0.3, 0.7], random sign
                u = uniform(seed, f"{cfg.name}/a0", 2 * A)
                a = (0.3 + 0.4 * u[:A]) * np.where(u[A:] < 0.5, -1.0, 1.0)
            else:
                s = math.sqrt(1.0 - rho * rho)
                xc = rho * xc + s * z1
                eps = z2 if traj.iid_noise else rho * eps + s * z2
                a = a + traj.action_step * normal(seed, f"{cfg.name}/da/{n}", A)
                if traj.jump_every and n % traj.jump_every == 0:
                    sign = np.where(uniform(seed, f"{cfg.name}/jump/{n}", A) < 0.5, -1.0, 1.0)
                    a = a + traj.jump * sign
                a = np.clip(a, -1.0, 1.0)
            self._clean.append(xc.astype(np.float32))
            self._eps.append(eps.astype(np.float32))
            self._act.append(np.asarray(a, dtype=np.float32).copy())
        # condition tokens (cross-attention): a fixed text part of max_ctx / 2
        # tokens, then object / lane tokens that drift AR(1) from chunk to
        # chunk and whose count varies in [max_ctx / 4, max_ctx / 2]
        self._ctx = []
        if cfg.d_ctx > 0:
            M, D = cfg.max_ctx, cfg.d_ctx
            n_text = M // 2
            text = normal(seed, f"{cfg.name}/ctx_text", n_text * D).reshape(n_text, D)
            obj = None
            for n in range(self.n_chunks):
                rho = _rho_at(traj, n, self.n_chunks)
                z = normal(seed, f"{cfg.name}/ctx_obj/{n}", (M - n_text) * D).reshape(M - n_text, D)
                obj = z if obj is None else rho * obj + math.sqrt(1.0 - rho * rho) * z
                lo = (M - n_text) // 2
                n_obj = lo + int(uniform(seed, f"{cfg.name}/ctx_len/{n}", 1)[0] * (M - n_text - lo + 1))
                n_obj = min(n_obj, M - n_text)
                self._ctx.append(np.concatenate([text, obj[:n_obj]]).astype(np.float32))

    def clean(self, n: int) -> np.ndarray:
        return self._clean[n]

    def noise(self, n: int) -> np.ndarray:
        return self._eps[n]

    def action(self, n: int) -> np.ndarray:
        return self._act[n]

    def context(self, n: int) -> np.ndarray:
        """Condition tokens of chunk n, [n_ctx(n), d_ctx] float32 (models with
        cross-attention only)."""
        return self._ctx[n]


SIGMAS = (1.0, 0.75, 0.5, 0.25, 0.0)   # 4 Euler flow-matching passes, then sigma = 0


def random_tensor(seed: int, name: str, shape: tuple, std: float = 1.0,
                  bf16: bool = False) -> np.ndarray:
    """Generic seeded normal tensor (float32) for kernel-level parity cases."""
    a = (normal(seed, name, int(np.prod(shape))) * std).astype(np.float32).reshape(shape)
    return bf16_representable(a) if bf16 else a


# --------------------------------------------------------------------------
# The same generator on a torch device (large benchmark models)
# --------------------------------------------------------------------------
def _i64(v: int) -> int:
    """A 64-bit pattern as the signed int64 with the same bits."""
    v &= 0xFFFFFFFFFFFFFFFF
    return v - (1 << 64) if v >> 63 else v


def _mix64_t(z):
    """SplitMix64 output function on int64 tensors: wrapping products, logical
    right shifts (arithmetic shift masked to the shifted width)."""
    m1, m2 = _i64(int(_M1)), _i64(int(_M2))
    z = (z ^ ((z >> 30) & ((1 << 34) - 1))) * m1
    z = (z ^ ((z >> 27) & ((1 << 37) - 1))) * m2
    return z ^ ((z >> 31) & ((1 << 33) - 1))


def normal_torch(seed: int, name: str, n: int, device, offset: int = 0, block: int = 1 << 24):
    """``normal`` computed on a torch device (float64): the same counters,
    SplitMix64 stream and Box-Muller transform, so the values agree with the
    numpy ones up to the last bit of the device's log / cos."""
    import torch
    key = _i64(int(_stream_key(seed, name)))
    gamma = _i64(0x9E3779B97F4A7C15)
    out = torch.empty(n, dtype=torch.float64, device=device)
    for a in range(0, n, block):
        m = min(block, n - a)
        i = torch.arange(2 * (offset + a), 2 * (offset + a + m), dtype=torch.int64, device=device)
        s = key + (i + 1) * gamma
        bits = (_mix64_t(s) >> 11) & ((1 << 53) - 1)
        u = (bits.to(torch.float64) + 0.5) * (1.0 / 9007199254740992.0)
        u1, u2 = u[0::2], u[1::2]
        out[a:a + m] = torch.sqrt(-2.0 * torch.log(u1)) * torch.cos(2.0 * math.pi * u2)
    return out


def make_weight_torch(cfg: ModelCfg, name: str, device, seed: int = 0):
    """``make_weight`` generated on a torch device (float32 tensor)."""
    import torch
    shape = weight_shapes(cfg)[name]
    std = _init_std(name, shape)
    n = int(np.prod(shape))
    out = torch.empty(n, dtype=torch.float32, device=device)
    step = 1 << 26
    for a in range(0, n, step):
        m = min(step, n - a)
        w = normal_torch(seed, cfg.name + "/" + name, m, device, offset=a) * std
        if name in GAINS:
            w = 1.0 + w
        w = w.to(torch.float32)
        if cfg.dtype == "bf16":
            w = w.to(torch.bfloat16).to(torch.float32)
        out[a:a + m] = w
    return out.reshape(shape)


def make_weights_torch(cfg: ModelCfg, device, seed: int = 0) -> dict:
    return {k: make_weight_torch(cfg, k, device, seed) for k in weight_shapes(cfg)}
