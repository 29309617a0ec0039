"""X-Cache chunk step, CPU oracle (TEST INFRASTRUCTURE ONLY; see package doc).

Every function names the passage of the paper it follows (X-Cache,
arXiv 2604.20289).  Where the paper is silent the reading taken is stated in
the docstring.  Arithmetic is fp64.  For bf16 models every tensor that a BF16
forward pass stores (Section 3.1.1: all DiT forward passes run in BF16) is
rounded to bf16 at the operator's output; fp32 models are left in fp64.

Parity status: primitives, fingerprint geometry and its global channel, the
gate equations, the conditioning MLPs, the output head and both fingerprint
refresh rules are pinned by tests/test_oracle_pins.py; the composition of a
whole DiT block is pinned
only by brute-force loops on tiny shapes and structural invariants (the
paper's X-World weights are not available), and the paper's 71% skip rate is
X-World-specific -- parity unpinned against the paper for those two.
"""
from __future__ import annotations

import math
from dataclasses import dataclass
from enum import IntEnum

import numpy as np


# ---------------------------------------------------------------------------
# Storage precision
# ---------------------------------------------------------------------------
def to_bf16(x) -> np.ndarray:
    """Round to the nearest bfloat16 value, ties to even, returned as fp64.
    fp64 -> fp32 (IEEE round to nearest) -> bf16 (keep the top 16 bits of the
    fp32 pattern after adding 0x7FFF plus the lowest kept bit)."""
    f = np.asarray(x, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    keep_lsb = (u >> np.uint64(16)) & np.uint64(1)
    r = ((u + np.uint64(0x7FFF) + keep_lsb) & np.uint64(0xFFFF0000)).astype(np.uint32)
    out = r.view(np.float32).astype(np.float64)
    return np.where(np.isnan(f), np.nan, out)


# ---------------------------------------------------------------------------
# Primitives of the DiT block (reading c16 of the block internals: pre-norm,
# adaLN-Zero modulation (Section 1: actions enter every block via adaLN-Zero),
# biased linears, GELU-tanh FFN, RoPE self-attention)
# ---------------------------------------------------------------------------
def layer_norm(x: np.ndarray, eps: float) -> np.ndarray:
    """LayerNorm over the last axis without affine: (x - mean) / sqrt(var + eps),
    population variance."""
    x = np.asarray(x, dtype=np.float64)
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps)


def silu(x: np.ndarray) -> np.ndarray:
    """SiLU(x) = x * sigmoid(x)."""
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x: np.ndarray) -> np.ndarray:
    """GELU, tanh form: 0.5 x (1 + tanh(sqrt(2/pi) (x + 0.044715 x^3)))."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * x ** 3)))


def timestep_embedding(sigma: float, dim: int) -> np.ndarray:
    """Sinusoidal embedding of the flow time 1000*sigma (the timestep part of
    the conditioning c_t in Eq. 1): [cos(s f_i), sin(s f_i)], f_i = 10000^(-i/half)."""
    half = dim // 2
    f = np.exp(-math.log(10000.0) * np.arange(half, dtype=np.float64) / half)
    s = 1000.0 * float(sigma)
    return np.concatenate([np.cos(s * f), np.sin(s * f)])


def rope_pair_table(head_dim: int, theta: float):
    """RoPE over the 4 axes (camera, absolute frame, h, w).  Reading c17: the
    head dimension is split hd/8 : 3hd/8 : hd/4 : hd/4 between the axes, each
    axis owns consecutive interleaved pairs (2p, 2p+1), and pair j of an axis
    with D dims rotates at frequency theta^(-2j/D).
    Returns (axis_of_pair [hd/2] int, freq_of_pair [hd/2] float64)."""
    assert head_dim % 16 == 0
    dims = [head_dim // 8, 3 * head_dim // 8, head_dim // 4, head_dim // 4]
    axis, freq = [], []
    for a, D in enumerate(dims):
        for j in range(D // 2):
            axis.append(a)
            freq.append(theta ** (-2.0 * j / D))
    return np.array(axis), np.array(freq, dtype=np.float64)


def token_positions(n_cams: int, frames: int, gh: int, gw: int, chunk: int) -> np.ndarray:
    """[L, 4] (camera, absolute frame chunk*frames + f, h, w) for tokens in
    (camera, frame, h, w) row-major order."""
    c, f, h, w = np.meshgrid(np.arange(n_cams), np.arange(frames), np.arange(gh), np.arange(gw),
                             indexing="ij")
    pos = np.stack([c.ravel(), f.ravel() + chunk * frames, h.ravel(), w.ravel()], axis=1)
    return pos.astype(np.float64)


def group_token_positions(groups, frames: int, chunk: int) -> np.ndarray:
    """[L, 4] positions of a chunk made of view groups ((cameras, gh, gw), ...)
    whose tokens follow one another: within a group as token_positions, the
    camera coordinate counting on across groups (one camera index per
    physical camera)."""
    out, cam0 = [], 0
    for V, gh, gw in groups:
        pos = token_positions(V, frames, gh, gw, chunk)
        pos[:, 0] += cam0
        out.append(pos)
        cam0 += V
    return np.concatenate(out, axis=0)


def apply_rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotate interleaved pairs of x [L, H, hd] by angle pos[axis(p)] * freq(p):
    (x0, x1) -> (x0 cos - x1 sin, x0 sin + x1 cos)."""
    L, H, hd = x.shape
    axis, freq = rope_pair_table(hd, theta)
    ang = pos[:, axis] * freq[None, :]                      # [L, hd/2]
    c, s = np.cos(ang)[:, None, :], np.sin(ang)[:, None, :]
    x0, x1 = x[..., 0::2], x[..., 1::2]
    out = np.empty_like(x, dtype=np.float64)
    out[..., 0::2] = x0 * c - x1 * s
    out[..., 1::2] = x0 * s + x1 * c
    return out


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, qblock: int = 1024) -> np.ndarray:
    """softmax(q k^T / sqrt(hd)) v per head with an explicit, materialised score
    row per query (max-subtracted exp, normalised).  q [Lq, H, hd], k/v [Lk, H, hd].
    No mask: every query sees every resident key (reading c18)."""
    Lq, H, hd = q.shape
    out = np.empty((Lq, H, hd), dtype=np.float64)
    scale = 1.0 / math.sqrt(hd)
    for h in range(H):
        kh, vh = k[:, h, :], v[:, h, :]
        for a in range(0, Lq, qblock):
            s = (q[a:a + qblock, h, :] @ kh.T) * scale
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p /= p.sum(axis=1, keepdims=True)
            out[a:a + qblock, h, :] = p @ vh
    return out


# ---------------------------------------------------------------------------
# Fingerprint geometry (Section 2.3.1)
# ---------------------------------------------------------------------------
def grid_allocation(Fg: int, Hg: int, Wg: int, K: int):
    """Token budget per axis.  Reading c6: k_a = clamp(floor(c * dim_a), 1, dim_a)
    with c = (K / (Fg Hg Wg))^(1/3), so k_F : k_H : k_W ~ Fg : Hg : Wg and the
    product is about K.  floor(c * dim) is taken exactly as the largest integer
    k with k^3 * (Fg Hg Wg) <= K * dim^3."""
    N = Fg * Hg * Wg
    out = []
    for dim in (Fg, Hg, Wg):
        k = 0
        while (k + 1) <= dim and (k + 1) ** 3 * N <= K * dim ** 3:
            k += 1
        out.append(min(max(k, 1), dim))
    return tuple(out)


def axis_indices(dim: int, k: int) -> np.ndarray:
    """k uniformly spaced, cell-centred indices on an axis of length dim
    (reading c7): floor((2j + 1) dim / (2k)), j = 0..k-1."""
    j = np.arange(k)
    return ((2 * j + 1) * dim) // (2 * k)


def fingerprint_rows(n_cams: int, frames: int, gh: int, gw: int, K: int) -> np.ndarray:
    """Token rows of the spatial fingerprint phi(x) [V, k_F k_H k_W]: the
    Cartesian product of the per-axis indices, per camera of the (single) view
    group.  A camera with <= K tokens keeps all of them (Section 2.3.1)."""
    npc = frames * gh * gw
    rows = []
    for c in range(n_cams):
        if npc <= K:
            rows.append(c * npc + np.arange(npc))
            continue
        kF, kH, kW = grid_allocation(frames, gh, gw, K)
        cam = []
        for f in axis_indices(frames, kF):
            for h in axis_indices(gh, kH):
                for w in axis_indices(gw, kW):
                    cam.append(c * npc + (f * gh + h) * gw + w)
        rows.append(np.array(cam))
    return np.stack(rows)


def linear_rows(n_tok: int, K: int) -> np.ndarray:
    """1-D fallback of Section 2.3.1 (grid shape unavailable): K uniformly
    spaced, cell-centred indices along a camera's token axis of length n_tok,
    floor((2j + 1) n_tok / (2K)) (reading c7 applied to one axis); all tokens
    when n_tok <= K."""
    if n_tok <= K:
        return np.arange(n_tok)
    return axis_indices(n_tok, K)


def group_fingerprint_rows(groups, frames: int, K: int, linear: bool = False) -> list:
    """Spatial-sample rows of every view group (Section 2.3.1: one fingerprint
    per group, its cameras stacked along V): a list with one [V_g, k_g] array
    of chunk token indices per group.  ``linear`` takes the 1-D fallback
    instead of the 3-D grid sample."""
    out, tok0 = [], 0
    for V, gh, gw in groups:
        npc = frames * gh * gw
        if linear:
            loc = linear_rows(npc, K)
            rows = np.stack([c * npc + loc for c in range(V)])
        else:
            rows = fingerprint_rows(V, frames, gh, gw, K)
        out.append(rows + tok0)
        tok0 += V * npc
    return out


# ---------------------------------------------------------------------------
# Gate metrics (Eq. 5 - 9)
# ---------------------------------------------------------------------------
def cosine(a: np.ndarray, b: np.ndarray) -> float:
    """Eq. 5 on one flattened fingerprint entry.  Reading c10: both norms
    < 1e-12 -> 1, exactly one -> 0, NaN -> 0."""
    a = np.asarray(a, dtype=np.float64).ravel()
    b = np.asarray(b, dtype=np.float64).ravel()
    na, nb = math.sqrt(float(a @ a)), math.sqrt(float(b @ b))
    dot = float(a @ b)
    if math.isnan(na) or math.isnan(nb) or math.isnan(dot):
        return 0.0
    if na < 1e-12 and nb < 1e-12:
        return 1.0
    if na < 1e-12 or nb < 1e-12:
        return 0.0
    return dot / (na * nb)


def max_token_deviation(cur: np.ndarray, prev: np.ndarray, eps: float) -> float:
    """Eq. 6: max |phi_n - phi_prev| / (mean |phi_prev| + eps) over one spatial
    entry.  NaN -> +inf (forces recompute)."""
    cur = np.asarray(cur, dtype=np.float64).ravel()
    prev = np.asarray(prev, dtype=np.float64).ravel()
    d = float(np.max(np.abs(cur - prev))) / (float(np.mean(np.abs(prev))) + eps)
    return math.inf if math.isnan(d) else d


def gate_metrics(phi, cached, eps: float):
    """Eq. 5 - 6 over a fingerprint with one spatial and one global entry per
    view group plus the action entry: s_cos = min of the cosines of all
    entries (Eq. 5); d_max = max over the groups' spatial entries of Eq. 6
    (reading c24: every group's sample must pass the deviation test).
    ``phi`` and ``cached`` are (spatial list, global list, action)."""
    sp, gl, ac = phi
    csp, cgl, cac = cached
    s = min([cosine(a, c) for a, c in zip(sp, csp)]
            + [cosine(a, c) for a, c in zip(gl, cgl)]
            + [cosine(ac, cac)])
    dmax = max(max_token_deviation(a, c, eps) for a, c in zip(sp, csp))
    return s, dmax


@dataclass
class GateParams:
    """Gate knobs; defaults are the paper's Table 1 (tau_floor 0.97 per Table 1
    and the ablation's default row, reading c1; step-0 protection off, c2) and
    K = 32 fingerprint tokens (Section 2.3.1)."""
    enabled: bool = True
    tau_floor: float = 0.97
    margin: float = 0.02
    alpha: float = 0.30
    tau_dev: float = 2.0
    eps_dev: float = 1e-6
    front_anchors: int = 1
    back_anchors: int = 0
    warmup_chunks: int = 1
    max_skips: int = 0           # 0 = off
    protect_step0: bool = False
    step0_strict_tau: float = 0.0   # 0 = off, else e.g. 0.999
    fp_tokens: int = 32
    fp_refresh: int = 0          # 0 = refresh on compute, 1 = on every evaluation
    fp_linear: bool = False      # 1-D fallback sample instead of the 3-D grid
    chain: bool = False          # lazy residual chaining over runs of skipped blocks (reading c27)


class Decision(IntEnum):
    FORCED = 0      # computed without evaluating the gate
    COMPUTE = 1     # gate evaluated, recompute
    SKIP = 2        # gate evaluated, reuse cached residual (Eq. 4)


@dataclass
class GateCell:
    """Per-(t, b) cache: residual r_hat (Eq. 3), cached fingerprint entries
    (spatial and global entry of every view group, the action), EMA of the
    cosine (Eq. 8), consecutive-skip counter (max staleness)."""
    valid: bool = False
    r_hat: np.ndarray | None = None
    phi_sp: list | None = None
    phi_gl: list | None = None
    phi_act: np.ndarray | None = None
    ema: float = 0.0
    has_hist: bool = False
    stale: int = 0


def gate_decide(cell: GateCell, s: float, dmax: float, step: int, p: GateParams,
                replay: bool | None = None):
    """Skip test of one evaluated (t, b) cell; updates the cell's EMA and
    consecutive-skip counter and returns (skip, tau_cos).

    * tau_cos = max(tau_floor, ema - m) (Eq. 9), from the EMA before this
      evaluation; the first evaluation of a cell uses tau_floor and seeds the
      EMA with s (reading c12).
    * Optional strict step-0 threshold (Section 2.5 (1), reading c15).
    * skip = (s >= tau_cos) and (d_max < tau_dev) (Eq. 7).
    * At most M consecutive skips per cell (Section 2.5 (4), reading c13).
    * EMA <- alpha s + (1 - alpha) EMA on every evaluation (Eq. 8).
    ``replay`` (decision-replay mode) replaces the decision."""
    tau = max(p.tau_floor, cell.ema - p.margin) if cell.has_hist else p.tau_floor
    if p.step0_strict_tau > 0.0 and step == 0:
        tau = max(tau, p.step0_strict_tau)
    skip = (s >= tau) and (dmax < p.tau_dev)
    if p.max_skips > 0 and cell.stale >= p.max_skips:
        skip = False
    if replay is not None:
        skip = replay
    cell.ema = p.alpha * s + (1.0 - p.alpha) * cell.ema if cell.has_hist else s
    cell.has_hist = True
    cell.stale = cell.stale + 1 if skip else 0
    return skip, tau


# ---------------------------------------------------------------------------
# The DiT (Eq. 1 - 2)
# ---------------------------------------------------------------------------
class OracleModel:
    """Multi-block causal DiT of Section 2.1 with the block internals of
    reading c16.  Weights use the convention y = x @ W."""

    def __init__(self, cfg, weights: dict):
        self.cfg = cfg
        self.w = {k: np.asarray(v, dtype=np.float64) for k, v in weights.items()}
        self.R = to_bf16 if cfg.dtype == "bf16" else (lambda a: np.asarray(a, dtype=np.float64))

    def cond(self, sigma: float, action: np.ndarray):
        """Conditioning c_t: e = MLP_t(sinusoid(1000 sigma)) + MLP_a(action);
        shared projection SiLU(e) W_m + b_m plus a per-block table gives the
        six adaLN-Zero vectors (shift1, scale1, gate1, shift2, scale2, gate2)
        of every block; a separate projection gives the head's (shift, scale)."""
        w, d = self.w, self.cfg.d_model
        te = timestep_embedding(sigma, self.cfg.t_freq)
        e_t = silu(te @ w["t_w1"] + w["t_b1"]) @ w["t_w2"] + w["t_b2"]
        e_a = silu(np.asarray(action, np.float64) @ w["a_w1"] + w["a_b1"]) @ w["a_w2"] + w["a_b2"]
        e = e_t + e_a
        m = (silu(e) @ w["mod_w"] + w["mod_b"]).reshape(6, d)
        mods = m[None, :, :] + w["blk_mod"]                      # [B, 6, d]
        hm = (silu(e) @ w["head_w"] + w["head_b"]).reshape(2, d) + w["head_tab"]
        return mods, hm

    def patch_embed(self, latent: np.ndarray) -> np.ndarray:
        """x_{t,0}: linear patch embedding of the [L, 16] latent."""
        return self.R(np.asarray(latent, np.float64) @ self.w["pe_w"] + self.w["pe_b"])

    def ln_mod(self, x, shift, scale):
        return self.R(layer_norm(x, self.cfg.ln_eps) * (1.0 + scale) + shift)

    def context_kv(self, b: int, context: np.ndarray):
        """Keys and values of block b's cross-attention over the chunk's
        condition tokens (objects, lanes, text; Section 2.1 and 2.5): the
        tokens [n_ctx, d_ctx] (rounded to the storage type) times W_kv plus
        bias, split into k and v [n_ctx, H, hd].  No RoPE."""
        cfg, w, R = self.cfg, self.w, self.R
        n, d, H, hd = context.shape[0], cfg.d_model, cfg.n_heads, cfg.head_dim
        kv = R(R(np.asarray(context, np.float64)) @ w["ca_kv_w"][b] + w["ca_kv_b"][b])
        return kv[:, :d].reshape(n, H, hd), kv[:, d:].reshape(n, H, hd)

    def cross_attention(self, b: int, x1: np.ndarray, ctx_kv):
        """Cross-attention layer of block b (reading c26): x1 + (attention of
        LN(x1) gamma + beta projected by W_q, over the condition keys and
        values) W_o + b_o.  No modulation and no gate."""
        cfg, w, R = self.cfg, self.w, self.R
        L, d, H, hd = x1.shape[0], cfg.d_model, cfg.n_heads, cfg.head_dim
        h = R(layer_norm(x1, cfg.ln_eps) * w["ca_ln_w"][b] + w["ca_ln_b"][b])
        q = R(h @ w["ca_q_w"][b] + w["ca_q_b"][b]).reshape(L, H, hd)
        kc, vc = ctx_kv
        o = R(attention(q, kc, vc).reshape(L, d))
        return R(x1 + (o @ w["ca_o_w"][b] + w["ca_o_b"][b]))

    def block(self, b: int, x_in: np.ndarray, mod: np.ndarray, past_k: list, past_v: list,
              pos: np.ndarray, ctx_kv=None, rows=None):
        """x_{t,b} = x_{t,b-1} + f_b(x_{t,b-1}; c_t) (Eq. 1).  Returns the block
        output and this pass's (k, v) of the current chunk [L, H, hd].  With
        ``ctx_kv`` (this block's condition keys / values) the cross-attention
        layer sits between the self-attention and the FFN.  With ``rows``
        (token indices) only those rows of the output are computed and
        returned (keys and values still come from every token): every step
        after the K/V projection acts on one token row at a time."""
        cfg, w, R = self.cfg, self.w, self.R
        L, d, H, hd = x_in.shape[0], cfg.d_model, cfg.n_heads, cfg.head_dim
        sh1, sc1, g1, sh2, sc2, g2 = mod
        h = self.ln_mod(x_in, sh1, sc1)
        qkv = h @ w["qkv_w"][b] + w["qkv_b"][b]
        q = qkv[:, :d].reshape(L, H, hd)
        k = qkv[:, d:2 * d].reshape(L, H, hd)
        v = qkv[:, 2 * d:].reshape(L, H, hd)
        q = R(apply_rope(q, pos, cfg.rope_theta))
        k = R(apply_rope(k, pos, cfg.rope_theta))
        v = R(v)
        if rows is not None:
            rows = np.asarray(rows)
            q, x_in, L = q[rows], x_in[rows], len(rows)
        keys = np.concatenate(past_k + [k], axis=0)
        vals = np.concatenate(past_v + [v], axis=0)
        o = R(attention(q, keys, vals).reshape(L, d))
        x1 = R(x_in + g1 * (o @ w["o_w"][b] + w["o_b"][b]))
        if ctx_kv is not None:
            x1 = self.cross_attention(b, x1, ctx_kv)
        h2 = self.ln_mod(x1, sh2, sc2)
        u = R(gelu_tanh(h2 @ w["f1_w"][b] + w["f1_b"][b]))
        x2 = R(x1 + g2 * (u @ w["f2_w"][b] + w["f2_b"][b]))
        return x2, k, v

    def head(self, x: np.ndarray, hm: np.ndarray) -> np.ndarray:
        """Velocity v = (LN(x)(1 + scale) + shift) W_out + b_out, kept fp64."""
        hf = self.ln_mod(x, hm[0], hm[1])
        return hf @ self.w["out_w"] + self.w["out_b"]


# ---------------------------------------------------------------------------
# Rolling KV cache + X-Cache state + one chunk step
# ---------------------------------------------------------------------------
class OracleXCache:
    """The AR chunk step of Section 2.1 with the cross-chunk residual cache
    (Section 2.2), dual-metric gate (2.3), adaptive threshold (2.4) and safety
    mechanisms (2.5).

    Rolling KV cache: per block a FIFO of the clean (k, v) of the last
    kv_window - 1 KV-update chunks, written by the KV-update pass (Section
    2.1) with the oldest chunk evicted; every pass attends to those plus the
    current chunk's own (k, v) (reading c18).

    KV-update chunks (Section 2.5 (3), reading c23): with kv_period P = 0
    every chunk ends with the KV-update pass and only that pass is forced
    full.  With P > 0 only chunks n with n mod P == P - 1 have one; their
    denoising passes run in force-compute mode (every block computes, the
    gate is not evaluated, the residual and fingerprint caches are
    refreshed), and a chunk without one ends after its last denoising pass."""

    def __init__(self, cfg, weights: dict):
        self.cfg = cfg
        self.model = OracleModel(cfg, weights)
        self._fp_rows = {}
        self.reset()

    def reset(self):
        cfg = self.cfg
        self.n = 0                      # generation step (chunk index)
        self.next_step = 0
        self.ring_k = [[] for _ in range(cfg.n_blocks)]
        self.ring_v = [[] for _ in range(cfg.n_blocks)]
        self.cells = [[GateCell() for _ in range(cfg.n_blocks)] for _ in range(cfg.n_steps)]
        self.ctx_kv = None

    def set_context(self, context: np.ndarray):
        """Condition tokens for the following passes (models with
        cross-attention): every block's keys and values over them."""
        self.ctx_kv = [self.model.context_kv(b, context) for b in range(self.cfg.n_blocks)]

    def is_kv_chunk(self, n: int) -> bool:
        P = getattr(self.cfg, "kv_period", 0)
        return P == 0 or n % P == P - 1

    def fp_rows(self, K: int, linear: bool = False) -> list:
        key = (K, bool(linear))
        if key not in self._fp_rows:
            c = self.cfg
            self._fp_rows[key] = group_fingerprint_rows(c.groups, c.frames, K, linear)
        return self._fp_rows[key]

    def fingerprint(self, x: np.ndarray, action: np.ndarray, K: int, linear: bool = False):
        """phi(x), per view group (Section 2.3.1): spatial entry [V_g, k_g, d]
        and global channel = per-camera token mean [V_g, d]; condition channel
        = the action (2.3.2).  Returns (spatial list, global list, action)."""
        sp, gl, tok0 = [], [], 0
        for (V, gh, gw), rows in zip(self.cfg.groups, self.fp_rows(K, linear)):
            npc = self.cfg.frames * gh * gw
            sp.append(x[rows].copy())                                        # [V_g, k_g, d]
            gl.append(x[tok0:tok0 + V * npc].reshape(V, npc, -1).mean(axis=1))   # [V_g, d]
            tok0 += V * npc
        return sp, gl, np.asarray(action, np.float64).copy()

    def chain_sum(self, base: np.ndarray, pending: list) -> np.ndarray:
        """Reading c27: the block input after a run of skipped blocks, base +
        r_hat_j + ... + r_hat_{b-1} (Eq. 4 applied over the run), accumulated
        in float32 in block order and rounded once to the storage type."""
        acc = np.asarray(base, np.float64).astype(np.float32)
        for r in pending:
            acc = acc + np.asarray(r, np.float64).astype(np.float32)
        return self.model.R(acc.astype(np.float64))

    def chained_fingerprint(self, base: np.ndarray, pending: list, action, K: int, linear: bool = False):
        """phi of the lazily chained block input (reading c27): the spatial
        entry is the chained sum on the sampled rows only; the global channel
        is the per-camera mean of the last materialised input plus the
        per-camera means of the pending cached residuals."""
        sp, gl, tok0 = [], [], 0
        for (V, gh, gw), rows in zip(self.cfg.groups, self.fp_rows(K, linear)):
            npc = self.cfg.frames * gh * gw
            sp.append(self.chain_sum(base[rows], [r[rows] for r in pending]))
            m = np.asarray(base[tok0:tok0 + V * npc], np.float64).reshape(V, npc, -1).mean(axis=1)
            for r in pending:
                m = m + np.asarray(r[tok0:tok0 + V * npc], np.float64).reshape(V, npc, -1).mean(axis=1)
            gl.append(m)
            tok0 += V * npc
        return sp, gl, np.asarray(action, np.float64).copy()

    def chunk_step(self, latent, action, sigma: float, step: int, is_kv_update: bool,
                   p: GateParams, replay=None, trace: list | None = None):
        """One forward pass over all B blocks.  Returns (v [L, C], stats) where
        stats = dict(decision [B] int, s_cos [B], d_max [B], tau [B]); metrics
        are NaN where the gate was not evaluated.  ``replay`` (bool [B]) replaces
        the skip decision of evaluated blocks (decision-replay mode)."""
        cfg, M = self.cfg, self.model
        B = cfg.n_blocks
        S = cfg.n_steps
        n = self.n
        kv_chunk = self.is_kv_chunk(n)
        if is_kv_update:
            if self.next_step not in (0, S):
                raise RuntimeError("KV-update pass out of order")
            if not kv_chunk:
                raise RuntimeError("KV-update pass on a chunk without one")
        elif step != self.next_step or step >= S:
            raise RuntimeError("denoising step out of order")
        forced_chunk = getattr(cfg, "kv_period", 0) > 0 and kv_chunk
        xattn = getattr(cfg, "d_ctx", 0) > 0
        if xattn and self.ctx_kv is None:
            raise RuntimeError("cross-attention model without condition tokens")
        mods, hm = M.cond(sigma, action)
        pos = group_token_positions(cfg.groups, cfg.frames, n)
        x = M.patch_embed(latent)
        kv_new = {}
        stats = dict(decision=np.zeros(B, np.int64), s_cos=np.full(B, np.nan),
                     d_max=np.full(B, np.nan), tau=np.full(B, np.nan))
        # Lazy residual chaining (reading c27): x is the last materialised
        # block input; `pending` the cached residuals of the skipped blocks
        # after it, added only when a block computes (or before the head).
        chain = bool(getattr(p, "chain", False)) and not is_kv_update
        pending = []
        for b in range(B):
            gated_block = (p.enabled and not is_kv_update
                           and p.front_anchors <= b < B - p.back_anchors)
            skip = False
            phi = None
            if gated_block:
                cell = self.cells[step][b]
                if chain and pending:
                    phi = self.chained_fingerprint(x, pending, action, p.fp_tokens, p.fp_linear)
                else:
                    phi = self.fingerprint(x, action, p.fp_tokens, p.fp_linear)
                eligible = (n >= p.warmup_chunks and not (p.protect_step0 and step == 0)
                            and not forced_chunk and cell.valid)
                if eligible:
                    s, dmax = gate_metrics(phi, (cell.phi_sp, cell.phi_gl, cell.phi_act),
                                           p.eps_dev)                        # Eq. 5 - 6
                    skip, tau = gate_decide(cell, s, dmax, step, p,
                                            None if replay is None else bool(replay[b]))
                    stats["s_cos"][b], stats["d_max"][b], stats["tau"][b] = s, dmax, tau
                    stats["decision"][b] = Decision.SKIP if skip else Decision.COMPUTE
            if skip and chain:
                cell = self.cells[step][b]
                pending.append(cell.r_hat)                                   # Eq. 4, deferred
                if p.fp_refresh == 1:
                    cell.phi_sp, cell.phi_gl, cell.phi_act = phi
                if trace is not None:
                    trace.append(self.chain_sum(x, pending))
                continue
            if skip:
                cell = self.cells[step][b]
                x_out = M.R(x + cell.r_hat)                                  # Eq. 4
                if p.fp_refresh == 1:
                    cell.phi_sp, cell.phi_gl, cell.phi_act = phi
            else:
                if pending:                                                  # materialise the run
                    x = self.chain_sum(x, pending)
                    pending = []
                x_out, k, v = M.block(b, x, mods[b], self.ring_k[b], self.ring_v[b], pos,
                                      self.ctx_kv[b] if xattn else None)
                if is_kv_update:
                    kv_new[b] = (k, v)
                elif gated_block:
                    cell = self.cells[step][b]
                    cell.r_hat = M.R(x_out - x)                              # Eq. 2 - 3
                    cell.phi_sp, cell.phi_gl, cell.phi_act = phi
                    cell.valid = True
            if trace is not None:
                trace.append(x_out)
            x = x_out
        if pending:
            x = self.chain_sum(x, pending)
        v = M.head(x, hm)
        if is_kv_update:
            for b in range(B):                                               # FIFO append
                k, vv = kv_new[b]
                self.ring_k[b].append(k)
                self.ring_v[b].append(vv)
                while len(self.ring_k[b]) > cfg.kv_window - 1:
                    self.ring_k[b].pop(0)
                    self.ring_v[b].pop(0)
            self.n += 1
            self.next_step = 0
        elif step == S - 1 and not kv_chunk:
            self.n += 1                     # chunk without a KV-update pass
            self.next_step = 0
        else:
            self.next_step = step + 1
        return v, stats


# ---------------------------------------------------------------------------
# AR rollout (Section 2.1; closed-loop protocol of Section 3.1.3)
# ---------------------------------------------------------------------------
SIGMAS = (1.0, 0.75, 0.5, 0.25, 0.0)


def rollout(cfg, weights, traj, params: GateParams, n_chunks: int, replay=None,
            keep_trace: bool = False):
    """Chunk n: (cross-attention models: set the chunk's condition tokens)
    x = eps_n; for t < S: v = step(x, sigma_t); x += (sigma_{t+1} -
    sigma_t) v (Euler, flow matching); then, on a KV-update chunk, the
    KV-update pass on the chunk's clean latent x_c[n] at sigma = 0
    (teacher-forced, reading c22).
    Returns dict(final [n][L, C], stats [n][t] (t = S is the KV pass, absent
    on chunks without one), trace)."""
    oc = OracleXCache(cfg, weights)
    S = cfg.n_steps
    finals, stats, traces = [], [], []
    for n in range(n_chunks):
        x = np.asarray(traj.noise(n), np.float64)
        a = traj.action(n)
        if getattr(cfg, "d_ctx", 0) > 0:
            oc.set_context(traj.context(n))
        st_n, tr_n = [], []
        for t in range(S):
            tr = [] if keep_trace else None
            rp = None if replay is None else replay[n][t]
            v, st = oc.chunk_step(x, a, SIGMAS[t], t, False, params, replay=rp, trace=tr)
            x = x + (SIGMAS[t + 1] - SIGMAS[t]) * v
            st_n.append(st)
            tr_n.append(tr)
        if oc.is_kv_chunk(n):
            _, st = oc.chunk_step(traj.clean(n), a, 0.0, S, True, params)
            st_n.append(st)
        finals.append(x)
        stats.append(st_n)
        traces.append(tr_n)
    return dict(final=finals, stats=stats, trace=traces, state=oc)
