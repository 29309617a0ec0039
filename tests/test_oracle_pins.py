"""Pins of the CPU oracle against things other than itself: library routines
for textbook special cases, closed forms, invariants, hand-worked values and
brute force on tiny inputs.  CPU only."""
import json
import math
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as F

import oracle as O
import xc_inputs as X

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
rng = np.random.default_rng(1234)


# ---------------------------------------------------------------- bf16 storage
def test_bf16_round_matches_torch_and_hand_values():
    x = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000),
                        [0.0, -0.0, 1.0, 65504.0, 3.0e38]])
    ref = torch.tensor(x, dtype=torch.float32).to(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.to_bf16(x), ref)
    # ties to even: 1 + 2^-8 is halfway between 1 and 1 + 2^-7 -> 1;
    # 1 + 3*2^-8 is halfway between 1 + 2^-7 and 1 + 2^-6 -> 1 + 2^-6
    assert O.to_bf16(1 + 2 ** -8) == 1.0
    assert O.to_bf16(1 + 3 * 2 ** -8) == 1 + 2 ** -6
    assert np.isnan(O.to_bf16(np.nan))


# ----------------------------------------------------------------- primitives
def test_layer_norm_textbook():
    x = rng.standard_normal((7, 96)) * 3 + 1.5
    y = O.layer_norm(x, 1e-6)
    np.testing.assert_allclose(y.mean(-1), 0.0, atol=1e-12)
    v = x.var(-1)
    np.testing.assert_allclose(y.var(-1), v / (v + 1e-6), rtol=1e-12)
    ref = F.layer_norm(torch.tensor(x), (96,), eps=1e-6).numpy()
    np.testing.assert_allclose(y, ref, rtol=1e-12, atol=1e-12)


def test_gelu_silu_library():
    x = np.linspace(-8, 8, 1001)
    np.testing.assert_allclose(O.gelu_tanh(x), F.gelu(torch.tensor(x), approximate="tanh").numpy(),
                               rtol=1e-12, atol=1e-14)
    np.testing.assert_allclose(O.silu(x), F.silu(torch.tensor(x)).numpy(), rtol=1e-12, atol=1e-14)
    assert O.gelu_tanh(np.array([0.0]))[0] == 0.0


def test_timestep_embedding_closed_form():
    e0 = O.timestep_embedding(0.0, 256)
    np.testing.assert_array_equal(e0, np.r_[np.ones(128), np.zeros(128)])
    e = O.timestep_embedding(0.75, 256)
    assert e[0] == pytest.approx(math.cos(750.0)) and e[128] == pytest.approx(math.sin(750.0))
    # the last frequency is 10000^(-127/128)
    f = 10000.0 ** (-127 / 128)
    assert e[127] == pytest.approx(math.cos(750.0 * f)) and e[255] == pytest.approx(math.sin(750.0 * f))


def test_rope_pair_table_hand_values():
    axis, freq = O.rope_pair_table(16, 10000.0)
    np.testing.assert_array_equal(axis, [0, 1, 1, 1, 2, 2, 3, 3])
    np.testing.assert_allclose(freq, [1.0, 1.0, 10000 ** (-1 / 3), 10000 ** (-2 / 3),
                                      1.0, 10000 ** -0.5, 1.0, 10000 ** -0.5], rtol=1e-15)
    for hd, dims in ((64, (8, 24, 16, 16)), (128, (16, 48, 32, 32))):
        axis, _ = O.rope_pair_table(hd, 10000.0)
        assert [int((axis == a).sum()) * 2 for a in range(4)] == list(dims)


def test_rope_complex_rotation_norm_and_relative_position():
    L, H, hd = 5, 3, 64
    x = rng.standard_normal((L, H, hd))
    pos = rng.integers(0, 40, (L, 4)).astype(np.float64)
    y = O.apply_rope(x, pos, 10000.0)
    # complex form: (x0 + i x1) * exp(i angle)
    axis, freq = O.rope_pair_table(hd, 10000.0)
    z = (x[..., 0::2] + 1j * x[..., 1::2]) * np.exp(1j * pos[:, axis] * freq)[:, None, :]
    np.testing.assert_allclose(y[..., 0::2], z.real, atol=1e-12)
    np.testing.assert_allclose(y[..., 1::2], z.imag, atol=1e-12)
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-12)
    np.testing.assert_array_equal(O.apply_rope(x, np.zeros((L, 4)), 10000.0), x)
    # <R_p q, R_p' k> depends only on p - p' (shift both by the same offset)
    q, k = rng.standard_normal((1, 1, hd)), rng.standard_normal((1, 1, hd))
    p1, p2, sh = rng.integers(0, 30, 4), rng.integers(0, 30, 4), rng.integers(0, 30, 4)
    d1 = np.sum(O.apply_rope(q, p1[None] * 1.0, 1e4) * O.apply_rope(k, p2[None] * 1.0, 1e4))
    d2 = np.sum(O.apply_rope(q, (p1 + sh)[None] * 1.0, 1e4) * O.apply_rope(k, (p2 + sh)[None] * 1.0, 1e4))
    assert d1 == pytest.approx(d2, rel=1e-10, abs=1e-12)


def test_token_positions_order():
    pos = O.token_positions(2, 3, 4, 5, chunk=7)
    assert pos.shape == (120, 4)
    r = ((1 * 3 + 2) * 4 + 3) * 5 + 4          # camera 1, frame 2, h 3, w 4
    np.testing.assert_array_equal(pos[r], [1, 7 * 3 + 2, 3, 4])


def test_attention_special_cases_and_library():
    hd = 32
    q = rng.standard_normal((6, 2, hd))
    v = rng.standard_normal((1, 2, hd))
    k = rng.standard_normal((1, 2, hd))
    np.testing.assert_allclose(O.attention(q, k, v), np.broadcast_to(v, (6, 2, hd)), atol=1e-14)
    kk = np.repeat(rng.standard_normal((1, 2, hd)), 9, axis=0)
    vv = rng.standard_normal((9, 2, hd))
    np.testing.assert_allclose(O.attention(q, kk, vv), np.broadcast_to(vv.mean(0), (6, 2, hd)),
                               atol=1e-12)
    k = rng.standard_normal((50, 2, hd)) * 2
    v = rng.standard_normal((50, 2, hd))
    ref = F.scaled_dot_product_attention(torch.tensor(q).permute(1, 0, 2), torch.tensor(k).permute(1, 0, 2),
                                         torch.tensor(v).permute(1, 0, 2)).permute(1, 0, 2).numpy()
    np.testing.assert_allclose(O.attention(q, k, v, qblock=4), ref, rtol=1e-10, atol=1e-12)


# ------------------------------------------------------ fingerprint (Sec 2.3.1)
def test_grid_allocation_paper_grids():
    # k_F : k_H : k_W ~ F : H : W with product ~ K = 32
    assert O.grid_allocation(3, 16, 28, 32) == (1, 4, 8)
    assert O.grid_allocation(3, 20, 36, 32) == (1, 4, 8)
    assert O.grid_allocation(8, 8, 8, 64) == (4, 4, 4)            # exact cube root
    assert O.grid_allocation(2, 4, 4, 4) == (1, 2, 2)             # c = 1/2 exactly


def test_grid_allocation_brute_force_float():
    r = np.random.default_rng(5)
    checked = 0
    for _ in range(3000):
        dims = r.integers(1, 60, 3)
        K = int(r.integers(4, 200))
        N = int(np.prod(dims))
        c = (K / N) ** (1.0 / 3.0)
        exact = [c * d for d in dims]
        if any(abs(e - round(e)) < 1e-9 for e in exact):
            continue
        want = tuple(int(min(max(math.floor(e), 1), d)) for e, d in zip(exact, dims))
        assert O.grid_allocation(*map(int, dims), K) == want
        checked += 1
    assert checked > 2500


def test_axis_indices_hand_values():
    np.testing.assert_array_equal(O.axis_indices(3, 1), [1])
    np.testing.assert_array_equal(O.axis_indices(16, 4), [2, 6, 10, 14])
    np.testing.assert_array_equal(O.axis_indices(28, 8), [1, 5, 8, 12, 15, 19, 22, 26])
    np.testing.assert_array_equal(O.axis_indices(7, 7), np.arange(7))


def test_fingerprint_rows_enumeration():
    V, Fr, gh, gw = 3, 3, 16, 28
    rows = O.fingerprint_rows(V, Fr, gh, gw, 32)
    assert rows.shape == (V, 32)
    npc = Fr * gh * gw
    for c in range(V):
        got = set()
        for r in rows[c]:
            cc, rem = divmod(int(r), npc)
            f, rem = divmod(rem, gh * gw)
            h, w = divmod(rem, gw)
            assert cc == c and f == 1 and h in (2, 6, 10, 14) and w in (1, 5, 8, 12, 15, 19, 22, 26)
            got.add((f, h, w))
        assert len(got) == 32
    # a camera with <= K tokens keeps all of them
    np.testing.assert_array_equal(O.fingerprint_rows(2, 2, 4, 4, 32), np.arange(64).reshape(2, 32))


# --------------------------------------------------------- gate metrics Eq. 5-6
def test_cosine_closed_forms_and_library():
    from scipy.spatial.distance import cosine as sp_cos_dist
    a = rng.standard_normal(300)
    assert O.cosine(a, 2 * a) == pytest.approx(1.0, abs=1e-14)
    assert O.cosine(a, -a) == pytest.approx(-1.0, abs=1e-14)
    assert O.cosine([1.0, 0.0], [0.0, 3.0]) == 0.0
    b = rng.standard_normal(300)
    assert O.cosine(a, b) == pytest.approx(1.0 - sp_cos_dist(a, b), abs=1e-13)
    assert O.cosine(np.zeros(4), np.zeros(4)) == 1.0
    assert O.cosine(np.zeros(4), np.ones(4)) == 0.0
    assert O.cosine(np.r_[np.nan, 1.0], np.ones(2)) == 0.0


def test_max_token_deviation_closed_form():
    p = rng.standard_normal((6, 32, 16))
    d = O.max_token_deviation(2 * p, p, 1e-6)
    assert d == pytest.approx(np.abs(p).max() / (np.abs(p).mean() + 1e-6), rel=1e-13)
    assert O.max_token_deviation(p, p, 1e-6) == 0.0
    assert O.max_token_deviation(p * np.nan, p, 1e-6) == math.inf


# -------------------------------------------------- Eq. 7-9 and staleness rule
def test_table1_defaults_fixture():
    g = json.load(open(os.path.join(GOLDEN, "table1_defaults.json")))
    p = O.GateParams()
    for k in ("front_anchors", "back_anchors", "warmup_chunks", "tau_floor", "margin", "alpha",
              "tau_dev", "fp_tokens"):
        assert getattr(p, k) == g[k], k
    assert (p.max_skips == 0) == (g["max_skips"] == "off")
    assert p.protect_step0 == (g["step0_protection"] == "on")
    assert p.enabled


def test_ema_threshold_closed_form():
    p = O.GateParams(tau_floor=0.9, margin=0.02, alpha=0.3, tau_dev=10.0)
    cell = O.GateCell(valid=True)
    seq = [0.99, 0.995, 0.97, 0.999, 0.93, 0.998, 0.996]
    for k, s in enumerate(seq):
        skip, tau = O.gate_decide(cell, s, 0.5, 1, p)
        if k == 0:
            assert tau == 0.9
        else:
            ema_prev = (1 - 0.3) ** (k - 1) * seq[0] + sum(
                0.3 * (1 - 0.3) ** (k - 1 - i) * seq[i] for i in range(1, k))
            assert tau == pytest.approx(max(0.9, ema_prev - 0.02), abs=1e-14)
        assert tau >= p.tau_floor
        assert skip == (s >= tau)
        ema_now = (1 - 0.3) ** k * seq[0] + sum(0.3 * (1 - 0.3) ** (k - i) * seq[i] for i in range(1, k + 1))
        assert cell.ema == pytest.approx(ema_now, abs=1e-14)


def test_deviation_gate_and_strict_step0_and_staleness():
    p = O.GateParams(tau_floor=0.5, tau_dev=2.0)
    c = O.GateCell(valid=True)
    assert O.gate_decide(c, 0.99, 1.999, 1, p)[0] is True
    assert O.gate_decide(c, 0.99, 2.0, 1, p)[0] is False           # strict < tau_dev (Eq. 7)
    ps = O.GateParams(tau_floor=0.5, step0_strict_tau=0.999)
    assert O.gate_decide(O.GateCell(valid=True), 0.998, 0.0, 0, ps) == (False, 0.999)
    assert O.gate_decide(O.GateCell(valid=True), 0.998, 0.0, 1, ps) == (True, 0.5)
    pm = O.GateParams(tau_floor=0.5, max_skips=2)
    c = O.GateCell(valid=True)
    got = [O.gate_decide(c, 0.99, 0.0, 1, pm)[0] for _ in range(7)]
    assert got == [True, True, False, True, True, False, True]


# ---------------------------------------------------- block: brute-force loops
def _bruteforce_block(cfg, w, b, x, mod, keys_past, vals_past, pos):
    """Element-by-element loops (fp64, fp32 model so no rounding)."""
    L, d, H, hd = x.shape[0], cfg.d_model, cfg.n_heads, cfg.head_dim
    eps = cfg.ln_eps

    def ln_mod(xx, sh, sc):
        out = np.zeros_like(xx)
        for i in range(L):
            mu = sum(xx[i]) / d
            var = sum((xx[i, j] - mu) ** 2 for j in range(d)) / d
            for j in range(d):
                out[i, j] = (xx[i, j] - mu) / math.sqrt(var + eps) * (1 + sc[j]) + sh[j]
        return out

    def linear(xx, W, bias):
        out = np.zeros((xx.shape[0], W.shape[1]))
        for i in range(xx.shape[0]):
            for j in range(W.shape[1]):
                out[i, j] = sum(xx[i, kk] * W[kk, j] for kk in range(W.shape[0])) + bias[j]
        return out

    def rope(row, p):
        axis, freq = O.rope_pair_table(hd, cfg.rope_theta)
        out = row.copy()
        for h in range(H):
            for pp in range(hd // 2):
                a = p[axis[pp]] * freq[pp]
                x0, x1 = row[h * hd + 2 * pp], row[h * hd + 2 * pp + 1]
                out[h * hd + 2 * pp] = x0 * math.cos(a) - x1 * math.sin(a)
                out[h * hd + 2 * pp + 1] = x0 * math.sin(a) + x1 * math.cos(a)
        return out

    sh1, sc1, g1, sh2, sc2, g2 = mod
    hN = ln_mod(x, sh1, sc1)
    qkv = linear(hN, w["qkv_w"][b], w["qkv_b"][b])
    q = np.array([rope(qkv[i, :d], pos[i]) for i in range(L)])
    k = np.array([rope(qkv[i, d:2 * d], pos[i]) for i in range(L)])
    v = qkv[:, 2 * d:]
    K = np.concatenate([kp.reshape(-1, d) for kp in keys_past] + [k])
    Vv = np.concatenate([vp.reshape(-1, d) for vp in vals_past] + [v])
    o = np.zeros((L, d))
    for h in range(H):
        sl = slice(h * hd, (h + 1) * hd)
        for i in range(L):
            sc = [sum(q[i, sl] * K[j, sl]) / math.sqrt(hd) for j in range(K.shape[0])]
            m = max(sc)
            e = [math.exp(s - m) for s in sc]
            z = sum(e)
            for c in range(hd):
                o[i, h * hd + c] = sum(e[j] * Vv[j, h * hd + c] for j in range(K.shape[0])) / z
    x1 = x + g1 * linear(o, w["o_w"][b], w["o_b"][b])
    h2 = ln_mod(x1, sh2, sc2)
    u = linear(h2, w["f1_w"][b], w["f1_b"][b])
    u = np.array([[0.5 * t * (1 + math.tanh(math.sqrt(2 / math.pi) * (t + 0.044715 * t ** 3)))
                   for t in row] for row in u])
    return x1 + g2 * linear(u, w["f2_w"][b], w["f2_b"][b])


TINY_BF = X.ModelCfg("pin_tiny", 2, 32, 2, 16, 48, 1, 1, 2, 3, 3, 2, dtype="f32")


def test_block_matches_bruteforce_loops():
    cfg = TINY_BF
    w = {k: v.astype(np.float64) for k, v in X.make_weights(cfg).items()}
    m = O.OracleModel(cfg, w)
    mods, _ = m.cond(0.5, np.array([0.2, -0.1]))
    x = rng.standard_normal((cfg.tokens, cfg.d_model))
    pos = O.token_positions(1, 1, 2, 3, chunk=2)
    kp = [rng.standard_normal((cfg.tokens, 2, 16))]
    vp = [rng.standard_normal((cfg.tokens, 2, 16))]
    got, _, _ = m.block(1, x, mods[1], kp, vp, pos)
    want = _bruteforce_block(cfg, w, 1, x, mods[1], kp, vp, pos)
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-12)


def test_block_adaln_zero_identity():
    """gate1 = gate2 = 0 makes f_b == 0, so x_{t,b} = x_{t,b-1} (Eq. 1)."""
    cfg = TINY_BF
    w = X.make_weights(cfg)
    m = O.OracleModel(cfg, w)
    mods, _ = m.cond(0.25, np.array([0.3, 0.3]))
    mods[0, 2] = 0.0
    mods[0, 5] = 0.0
    x = rng.standard_normal((cfg.tokens, cfg.d_model))
    got, _, _ = m.block(0, x, mods[0], [], [], O.token_positions(1, 1, 2, 3, 0))
    np.testing.assert_array_equal(got, x)


# ------------------------------------------------ rollout invariants
def _run(cfg, params, n_chunks, keep_trace=False, traj=None):
    w = X.make_weights(cfg)
    tr = traj or X.Trajectory(cfg, n_chunks=n_chunks)
    return O.rollout(cfg, w, tr, params, n_chunks, keep_trace=keep_trace), w, tr


FORCE_RECOMPUTE = dict(tau_floor=2.0)
FORCE_REUSE = dict(tau_floor=-2.0, margin=10.0, tau_dev=1e30)


def test_force_recompute_equals_no_cache_bitwise():
    cfg = X.TINY_F32
    r_off, _, _ = _run(cfg, O.GateParams(enabled=False), 5)
    r_fc, _, _ = _run(cfg, O.GateParams(**FORCE_RECOMPUTE), 5)
    for a, b in zip(r_off["final"], r_fc["final"]):
        np.testing.assert_array_equal(a, b)
    dec = np.array([[s["decision"] for s in ch] for ch in r_fc["stats"]])
    assert not (dec == O.Decision.SKIP).any()
    assert (dec[1:, :4, 1:] == O.Decision.COMPUTE).all()     # evaluated after warmup


@pytest.mark.parametrize("cfg", [X.TINY_F32, X.TINY_F32.replace(name="tiny_bf16_pin", dtype="bf16")])
def test_force_reuse_output_is_input_plus_cached_residual(cfg):
    r, w, tr = _run(cfg, O.GateParams(**FORCE_REUSE), 4, keep_trace=True)
    S, B = cfg.n_steps, cfg.n_blocks
    R = O.to_bf16 if cfg.dtype == "bf16" else (lambda a: a)
    m = O.OracleModel(cfg, w)
    for n in range(1, 4):
        for t in range(S):
            st = r["stats"][n][t]
            for b in range(B):
                if b < 1:
                    assert st["decision"][b] == O.Decision.FORCED
                    continue
                assert st["decision"][b] == O.Decision.SKIP
                x_in = r["trace"][n][t][b - 1]
                # r_hat(t, b) is the residual of chunk 0 (the last computing chunk)
                r_hat = R(r["trace"][0][t][b] - r["trace"][0][t][b - 1])
                np.testing.assert_array_equal(r["trace"][n][t][b], R(x_in + r_hat))
    del m


def test_safety_rules_counts():
    cfg = X.MID_HD64.replace(name="pin_mid_small", grid_h=4, grid_w=6, n_chunks=6)
    p = O.GateParams(tau_floor=0.0, margin=1.0, tau_dev=1e9, back_anchors=1, max_skips=2,
                     protect_step0=True)
    r, _, _ = _run(cfg, p, 6)
    dec = np.array([[s["decision"] for s in ch] for ch in r["stats"]])   # [n, S+1, B]
    assert (dec[:, 4, :] == O.Decision.FORCED).all()      # KV-update passes: every block computes
    assert (dec[0] == O.Decision.FORCED).all()            # warmup chunk
    assert (dec[:, :, 0] != O.Decision.SKIP).all()        # front anchor
    assert (dec[:, :, -1] != O.Decision.SKIP).all()       # back anchor
    assert (dec[:, 0, :] != O.Decision.SKIP).all()        # step-0 protection
    sk = dec[:, :4, 1] == O.Decision.SKIP
    assert sk.any()
    for t in range(1, 4):                                 # at most M = 2 consecutive skips
        run = 0
        for n in range(6):
            run = run + 1 if sk[n, t] else 0
            assert run <= 2


def test_ring_is_fifo_over_window():
    """Chunk n attends the clean K/V of chunks n-W+1..n-1 only (W = 3).  One
    block, so a chunk's K/V depend on that chunk's clean latent alone."""
    cfg = X.TINY_F32.replace(name="pin_tiny_1blk", n_blocks=1)
    base = X.Trajectory(cfg, n_chunks=4)

    class Pert:
        def __init__(self, which):
            self.which = which

        def noise(self, n):
            return base.noise(n)

        def action(self, n):
            return base.action(n)

        def clean(self, n):
            c = base.clean(n)
            return c + 0.5 if n == self.which else c

    p = O.GateParams(enabled=False)
    w = X.make_weights(cfg)
    ref = O.rollout(cfg, w, base, p, 4)["final"][3]
    far = O.rollout(cfg, w, Pert(0), p, 4)["final"][3]     # evicted by chunk 3
    near = O.rollout(cfg, w, Pert(1), p, 4)["final"][3]    # still resident
    np.testing.assert_array_equal(far, ref)
    assert np.abs(near - ref).max() > 1e-6


# ------------------------------------------------ view groups (Section 2.3.1)
def test_group_token_positions_brute_force():
    groups, Fr, chunk = ((2, 2, 3), (1, 4, 5)), 2, 3
    want = []
    cam = 0
    for V, gh, gw in groups:                      # explicit loops in token order
        for c in range(V):
            for f in range(Fr):
                for h in range(gh):
                    for w in range(gw):
                        want.append((cam + c, chunk * Fr + f, h, w))
        cam += V
    np.testing.assert_array_equal(O.group_token_positions(groups, Fr, chunk), np.array(want, float))


def test_linear_rows_hand_values():
    # 1344 tokens, K = 32: floor((2j + 1) * 1344 / 64) = 21 (2j + 1)
    np.testing.assert_array_equal(O.linear_rows(1344, 32), 21 * (2 * np.arange(32) + 1))
    np.testing.assert_array_equal(O.linear_rows(100, 3), [16, 50, 83])
    np.testing.assert_array_equal(O.linear_rows(20, 32), np.arange(20))


def test_group_fingerprint_rows_enumeration():
    groups, Fr = ((2, 16, 28), (1, 4, 4)), 3
    rows = O.group_fingerprint_rows(groups, Fr, 32)
    assert [r.shape for r in rows] == [(2, 32), (1, 18)]
    # group 0 starts at token 0: the single-group sample
    np.testing.assert_array_equal(rows[0], O.fingerprint_rows(2, 3, 16, 28, 32))
    # group 1 (3 x 4 x 4 = 48 > 32 tokens) starts after 2 x 1344 tokens; its
    # allocation is (2, 3, 3): f in {0, 2}, h and w in {0, 2, 3}
    got = set()
    for r in rows[1][0]:
        rem = int(r) - 2688
        f, rem = divmod(rem, 16)
        h, w = divmod(rem, 4)
        assert f in (0, 2) and h in (0, 2, 3) and w in (0, 2, 3)
        got.add((f, h, w))
    assert len(got) == 18
    # 1-D fallback: per camera, linear_rows along its own token axis
    lin = O.group_fingerprint_rows(groups, Fr, 32, linear=True)
    np.testing.assert_array_equal(lin[0][1], 1344 + 21 * (2 * np.arange(32) + 1))
    np.testing.assert_array_equal(lin[1][0], 2688 + O.linear_rows(48, 32))


def test_gate_metrics_over_groups_closed_forms():
    sp = [rng.standard_normal((2, 32, 8)), rng.standard_normal((1, 18, 8))]
    gl = [rng.standard_normal((2, 8)), rng.standard_normal((1, 8))]
    ac = rng.standard_normal(2)
    twice = ([2 * a for a in sp], [2 * a for a in gl], 2 * ac)
    s, d = O.gate_metrics(twice, (sp, gl, ac), 1e-6)
    assert s == pytest.approx(1.0, abs=1e-13)
    # d over the groups: max|2a - a| / (mean|a| + eps), the larger of the two
    want = max(np.abs(a).max() / (np.abs(a).mean() + 1e-6) for a in sp)
    assert d == pytest.approx(want, rel=1e-12)
    # one group's spatial sample flipped: that entry's cosine -1 is the minimum
    flip = ([sp[0], -sp[1]], gl, ac)
    s, d = O.gate_metrics(flip, (sp, gl, ac), 1e-6)
    assert s == pytest.approx(-1.0, abs=1e-13)
    assert d == pytest.approx(2 * np.abs(sp[1]).max() / (np.abs(sp[1]).mean() + 1e-6), rel=1e-12)
    # one group's global entry orthogonalised: cosine 0 is the minimum
    g1 = gl[1].ravel()
    o = rng.standard_normal(g1.size)
    o -= (o @ g1) / (g1 @ g1) * g1
    s, _ = O.gate_metrics((sp, [gl[0], o.reshape(gl[1].shape)], ac), (sp, gl, ac), 1e-6)
    assert s == pytest.approx(0.0, abs=1e-12)


def test_single_view_group_equals_plain_grid():
    cfg = X.TINY_F32.replace(name="pin_tiny_groups", n_chunks=3)
    grp = cfg.replace(view_groups=((cfg.n_cams, cfg.grid_h, cfg.grid_w),))
    p = O.GateParams(tau_floor=0.5, margin=0.02, tau_dev=10.0)
    w = X.make_weights(cfg)
    a = O.rollout(cfg, w, X.Trajectory(cfg, n_chunks=3), p, 3)
    b = O.rollout(grp, w, X.Trajectory(grp, n_chunks=3), p, 3)
    for n in range(3):
        np.testing.assert_array_equal(a["final"][n], b["final"][n])


# ----------------------------------- KV-update chunks (Section 2.5 (3), c23)
def test_kv_period_one_is_all_blocks():
    """P = 1: every chunk is a KV-update chunk, so every denoising pass runs
    in force-compute mode: no skip, outputs equal to the gate switched off."""
    cfg = X.TINY_F32.replace(name="pin_tiny_p1", n_chunks=4, kv_period=1)
    w = X.make_weights(cfg)
    lax = O.GateParams(tau_floor=0.0, margin=1.0, tau_dev=1e9)
    r = O.rollout(cfg, w, X.Trajectory(cfg, n_chunks=4), lax, 4)
    off = O.rollout(cfg.replace(kv_period=0), w, X.Trajectory(cfg, n_chunks=4),
                    O.GateParams(enabled=False), 4)
    for n in range(4):
        np.testing.assert_array_equal(r["final"][n], off["final"][n])
        assert all((st["decision"] == O.Decision.FORCED).all() for st in r["stats"][n])


def test_kv_period_forced_chunks_and_skip_bound():
    P, N = 3, 7
    cfg = X.TINY_F32.replace(name="pin_tiny_p3", n_chunks=N, kv_period=P)
    lax = O.GateParams(tau_floor=0.0, margin=1.0, tau_dev=1e9)
    r = O.rollout(cfg, X.make_weights(cfg), X.Trajectory(cfg, n_chunks=N), lax, N)
    S, B = cfg.n_steps, cfg.n_blocks
    gated = skipped = 0
    for n, st_n in enumerate(r["stats"]):
        kv = n % P == P - 1
        assert len(st_n) == S + (1 if kv else 0)          # KV pass on KV chunks only
        dec = np.array([s["decision"] for s in st_n])
        if kv or n < lax.warmup_chunks:
            assert (dec == O.Decision.FORCED).all()
        else:                                            # lax thresholds: every gated block skips
            assert (dec[:, 1:] == O.Decision.SKIP).all()
        if n >= lax.warmup_chunks:
            gated += S * (B - 1)
            skipped += int((dec[:S, 1:] == O.Decision.SKIP).sum())
    # each forced chunk takes its share: skip rate <= (P - 1) / P
    assert skipped / gated <= (P - 1) / P


def test_kv_period_ring_holds_kv_chunks_only():
    """P = 2, W = 3: the ring holds the clean K/V of the last two KV-update
    chunks (n = 1, 3, 5, ...).  One block, so a chunk's K/V depend on its own
    clean latent alone."""
    cfg = X.TINY_F32.replace(name="pin_tiny_p2", n_blocks=1, kv_period=2)
    base = X.Trajectory(cfg, n_chunks=7)

    class Pert:
        def __init__(self, which):
            self.which = which

        def noise(self, n):
            return base.noise(n)

        def action(self, n):
            return base.action(n)

        def clean(self, n):
            c = base.clean(n)
            return c + 0.5 if n == self.which else c

    p = O.GateParams(enabled=False)
    w = X.make_weights(cfg)
    ref = O.rollout(cfg, w, base, p, 7)["final"]
    not_kv = O.rollout(cfg, w, Pert(0), p, 7)["final"]     # chunk 0 has no KV pass
    kv1 = O.rollout(cfg, w, Pert(1), p, 7)["final"]        # written after chunk 1
    for n in range(7):
        np.testing.assert_array_equal(not_kv[n], ref[n])
    for n in (0, 1):
        np.testing.assert_array_equal(kv1[n], ref[n])
    for n in (2, 3, 4, 5):                                  # resident: (1), (1, 3)
        assert np.abs(kv1[n] - ref[n]).max() > 1e-6
    np.testing.assert_array_equal(kv1[6], ref[6])          # ring (3, 5): chunk 1 evicted


# --------------------------------------- cross-attention conditioning (c26)
def _xattn_model():
    cfg = X.XATTN_F32
    return cfg, O.OracleModel(cfg, X.make_weights(cfg))


def test_cross_attention_brute_force():
    """Explicit loops over queries, heads and condition tokens."""
    cfg, m = _xattn_model()
    d, H, hd, b = cfg.d_model, cfg.n_heads, cfg.head_dim, 1
    x1 = rng.standard_normal((5, d))
    ctx = rng.standard_normal((3, cfg.d_ctx))
    w = m.w
    got = m.cross_attention(b, x1, m.context_kv(b, ctx))
    want = np.empty_like(x1)
    for i in range(x1.shape[0]):
        mu = sum(x1[i]) / d
        var = sum((x1[i] - mu) ** 2) / d
        h = (x1[i] - mu) / math.sqrt(var + cfg.ln_eps) * w["ca_ln_w"][b] + w["ca_ln_b"][b]
        q = h @ w["ca_q_w"][b] + w["ca_q_b"][b]
        o = np.zeros(d)
        for hh in range(H):
            sl = slice(hh * hd, (hh + 1) * hd)
            scores = []
            for j in range(ctx.shape[0]):
                kv = ctx[j] @ w["ca_kv_w"][b] + w["ca_kv_b"][b]
                scores.append((float(q[sl] @ kv[:d][sl]) / math.sqrt(hd), kv[d:][sl]))
            mx = max(s for s, _ in scores)
            den = sum(math.exp(s - mx) for s, _ in scores)
            for s, v in scores:
                o[sl] += math.exp(s - mx) / den * v
        want[i] = x1[i] + o @ w["ca_o_w"][b] + w["ca_o_b"][b]
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-10)


def test_cross_attention_token_invariances():
    """No positional encoding on condition tokens: permuting them changes
    nothing; repeating every token m times changes nothing (softmax over
    identical keys); one token gives its value to every query."""
    cfg, m = _xattn_model()
    x1 = rng.standard_normal((7, cfg.d_model))
    ctx = rng.standard_normal((4, cfg.d_ctx))
    base = m.cross_attention(0, x1, m.context_kv(0, ctx))
    perm = m.cross_attention(0, x1, m.context_kv(0, ctx[[2, 0, 3, 1]]))
    np.testing.assert_allclose(perm, base, rtol=1e-12, atol=1e-12)
    rep = m.cross_attention(0, x1, m.context_kv(0, np.repeat(ctx, 3, axis=0)))
    np.testing.assert_allclose(rep, base, rtol=1e-12, atol=1e-12)
    k1, v1 = m.context_kv(0, ctx[:1])
    one = m.cross_attention(0, x1, (k1, v1))
    v = v1.reshape(1, -1)
    np.testing.assert_allclose(one - x1, np.broadcast_to(v @ m.w["ca_o_w"][0] + m.w["ca_o_b"][0], x1.shape),
                               rtol=1e-12, atol=1e-12)


def test_cross_attention_with_zero_output_is_plain_block():
    cfg, m = _xattn_model()
    m.w["ca_o_w"][:] = 0.0
    m.w["ca_o_b"][:] = 0.0
    x = rng.standard_normal((cfg.tokens, cfg.d_model))
    mods, _ = m.cond(0.5, np.array([0.3, -0.4]))
    pos = O.token_positions(cfg.n_cams, cfg.frames, cfg.grid_h, cfg.grid_w, 0)
    ctx = rng.standard_normal((5, cfg.d_ctx))
    a, _, _ = m.block(0, x, mods[0], [], [], pos, m.context_kv(0, ctx))
    b, _, _ = m.block(0, x, mods[0], [], [], pos)
    np.testing.assert_array_equal(a, b)


def test_block_rows_subset_equals_full_block():
    """A block evaluated on sampled rows gives those rows of the full block."""
    for cfg in (X.TINY_F32, X.XATTN_F32):
        m = O.OracleModel(cfg, X.make_weights(cfg))
        x = rng.standard_normal((cfg.tokens, cfg.d_model))
        mods, _ = m.cond(0.75, np.array([0.2, -0.1]))
        pos = O.token_positions(cfg.n_cams, cfg.frames, cfg.grid_h, cfg.grid_w, 1)
        past_k = [rng.standard_normal((cfg.tokens, cfg.n_heads, cfg.head_dim))]
        past_v = [rng.standard_normal((cfg.tokens, cfg.n_heads, cfg.head_dim))]
        ctx = m.context_kv(1, rng.standard_normal((5, cfg.d_ctx))) if cfg.d_ctx else None
        full, k, v = m.block(1, x, mods[1], past_k, past_v, pos, ctx)
        rows = np.array([0, 7, 33, cfg.tokens - 1])
        sub, k2, v2 = m.block(1, x, mods[1], past_k, past_v, pos, ctx, rows=rows)
        np.testing.assert_allclose(sub, full[rows], rtol=1e-12, atol=1e-12)
        np.testing.assert_array_equal(k2, k)


# ------------------------------- fingerprint global channel (Section 2.3.2)
def test_fingerprint_global_channel_explicit_camera_loops():
    """Global entry of every view group = per-camera token mean, summed by
    explicit loops over each camera's own token slice (two groups of unequal
    grids, so the camera slices are ragged); shifting one camera's tokens by a
    constant moves that camera's mean by the constant and nothing else."""
    cfg = X.GROUPS_F32
    oc = O.OracleXCache(cfg, X.make_weights(cfg))
    L, d = cfg.tokens, cfg.d_model
    x = rng.standard_normal((L, d))
    act = np.array([0.3, -0.2])
    _, gl, ac = oc.fingerprint(x, act, 32)
    want, tok = [], 0
    for V, gh, gw in cfg.groups:
        npc = cfg.frames * gh * gw
        means = np.zeros((V, d))
        for c in range(V):
            for j in range(d):
                s = 0.0
                for i in range(tok + c * npc, tok + (c + 1) * npc):
                    s += x[i, j]
                means[c, j] = s / npc
        want.append(means)
        tok += V * npc
    assert [g.shape for g in gl] == [w.shape for w in want] == [(2, d), (1, d)]
    for g, w in zip(gl, want):
        np.testing.assert_allclose(g, w, rtol=1e-12, atol=1e-13)
    np.testing.assert_array_equal(ac, act)
    # camera 1 of group 0 occupies tokens [96, 192): shift it by 0.75
    xs = x.copy()
    npc0 = cfg.frames * 6 * 8
    xs[npc0:2 * npc0] += 0.75
    _, gl2, _ = oc.fingerprint(xs, act, 32)
    np.testing.assert_allclose(gl2[0][0], gl[0][0], rtol=0, atol=1e-13)
    np.testing.assert_allclose(gl2[0][1], gl[0][1] + 0.75, rtol=0, atol=1e-12)
    np.testing.assert_allclose(gl2[1], gl[1], rtol=0, atol=1e-13)


# ------------------------------------- conditioning (adaLN-Zero, Section 1)
COND_CFG = X.ModelCfg("pin_cond_d8", 3, 8, 1, 8, 16, 1, 1, 1, 1, 2, 1, dtype="f32", t_freq=6)


def test_cond_with_zero_projections_is_bias_plus_block_table():
    """Every matrix zero: SiLU(e) W_m vanishes, so the six vectors of block b
    are b_m (split as shift1, scale1, gate1, shift2, scale2, gate2) plus the
    block's own table row, and the head's (shift, scale) are b_h + its table."""
    cfg = COND_CFG
    w = {k: v.astype(np.float64) for k, v in X.make_weights(cfg).items()}
    for k in ("t_w1", "t_w2", "a_w1", "a_w2", "mod_w", "head_w"):
        w[k] = np.zeros_like(w[k])
    mods, hm = O.OracleModel(cfg, w).cond(0.6, np.array([0.4, -0.7]))
    d = cfg.d_model
    for b in range(cfg.n_blocks):
        for s in range(6):
            for c in range(d):
                assert mods[b, s, c] == w["mod_b"][s * d + c] + w["blk_mod"][b, s, c]
    for s in range(2):
        for c in range(d):
            assert hm[s, c] == w["head_b"][s * d + c] + w["head_tab"][s, c]


def test_cond_scalar_loops():
    """The two conditioning MLPs, the shared modulation projection and the
    head projection as scalar loops (d = 8, 6 sinusoid features):
      te = [cos(1000 sigma f_i), sin(1000 sigma f_i)], f_i = 10000^(-i/3)
      e  = (SiLU(te W_t1 + b_t1) W_t2 + b_t2) + (SiLU(a W_a1 + b_a1) W_a2 + b_a2)
      mods[b][s][c] = sum_k SiLU(e_k) W_m[k][s d + c] + b_m[s d + c] + table[b][s][c]
      hm[s][c]      = sum_k SiLU(e_k) W_h[k][s d + c] + b_h[s d + c] + table_h[s][c]."""
    cfg = COND_CFG
    w = {k: v.astype(np.float64) for k, v in X.make_weights(cfg).items()}
    for k in w:                       # random biases and tables too
        if k.endswith("_b") or k in ("blk_mod", "head_tab"):
            w[k] = rng.standard_normal(w[k].shape) * 0.3
    sigma, a = 0.35, [0.45, -0.8]
    mods, hm = O.OracleModel(cfg, w).cond(sigma, np.array(a))
    d, tf = cfg.d_model, cfg.t_freq

    def silu(v):
        return v / (1.0 + math.exp(-v))

    half = tf // 2
    te = [math.cos(1000 * sigma * 10000 ** (-i / half)) for i in range(half)] + \
         [math.sin(1000 * sigma * 10000 ** (-i / half)) for i in range(half)]
    ht = [silu(sum(te[i] * w["t_w1"][i, j] for i in range(tf)) + w["t_b1"][j]) for j in range(d)]
    ha = [silu(sum(a[i] * w["a_w1"][i, j] for i in range(2)) + w["a_b1"][j]) for j in range(d)]
    e = [sum(ht[k] * w["t_w2"][k, j] for k in range(d)) + w["t_b2"][j]
         + sum(ha[k] * w["a_w2"][k, j] for k in range(d)) + w["a_b2"][j] for j in range(d)]
    se = [silu(v) for v in e]
    for b in range(cfg.n_blocks):
        for s in range(6):
            for c in range(d):
                want = sum(se[k] * w["mod_w"][k, s * d + c] for k in range(d)) + w["mod_b"][s * d + c] \
                    + w["blk_mod"][b, s, c]
                assert mods[b, s, c] == pytest.approx(want, rel=1e-12, abs=1e-13)
    for s in range(2):
        for c in range(d):
            want = sum(se[k] * w["head_w"][k, s * d + c] for k in range(d)) + w["head_b"][s * d + c] \
                + w["head_tab"][s, c]
            assert hm[s, c] == pytest.approx(want, rel=1e-12, abs=1e-13)


# ------------------------------------------------------------ output head
@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_head_element_loops(dtype):
    """v[i][c] = sum_j h[i][j] W_out[j][c] + b_out[c] with
    h[i][j] = LN(x_i)_j (1 + scale_j) + shift_j, (shift, scale) = hm; the
    bf16 model rounds h (the stored modulated activation) and keeps v fp64."""
    cfg = COND_CFG.replace(name=f"pin_head_{dtype}", dtype=dtype)
    w = X.make_weights(cfg)
    m = O.OracleModel(cfg, w)
    W, bo = m.w["out_w"], m.w["out_b"]
    x = rng.standard_normal((5, cfg.d_model)) * 2.0 + 0.5
    hm = rng.standard_normal((2, cfg.d_model))
    got = m.head(x, hm)
    d, C = cfg.d_model, cfg.c_latent
    rnd = (lambda t: float(O.to_bf16(t))) if dtype == "bf16" else (lambda t: t)
    assert got.shape == (5, C)
    for i in range(5):
        mu = sum(x[i]) / d
        var = sum((x[i, j] - mu) ** 2 for j in range(d)) / d
        h = [rnd((x[i, j] - mu) / math.sqrt(var + cfg.ln_eps) * (1 + hm[1, j]) + hm[0, j]) for j in range(d)]
        for c in range(C):
            want = sum(h[j] * W[j, c] for j in range(d)) + bo[c]
            assert got[i, c] == pytest.approx(want, rel=1e-12, abs=1e-12)


# --------------------------- fingerprint refresh on every evaluation (c5)
@pytest.mark.parametrize("refresh", [0, 1])
def test_fingerprint_refresh_after_skip(refresh):
    """fp_refresh = 1 (literal "previous generation" of Eq. 5-6): after an
    evaluated skip the cell holds the fingerprint of that pass's block input
    (its sampled rows, per-camera means and the chunk's action).  fp_refresh
    = 0: a skip leaves the cached fingerprint (the input that produced r_hat)
    untouched."""
    cfg = X.TINY_F32.replace(name="pin_refresh", n_chunks=4)
    w = X.make_weights(cfg)
    traj = X.Trajectory(cfg, n_chunks=4)
    p = O.GateParams(tau_floor=0.0, margin=1.0, tau_dev=1e9, fp_refresh=refresh)
    oc = O.OracleXCache(cfg, w)
    rows = O.fingerprint_rows(cfg.n_cams, cfg.frames, cfg.grid_h, cfg.grid_w, 32)
    npc = cfg.frames * cfg.grid_h * cfg.grid_w
    S = cfg.n_steps
    n_skips = 0
    for n in range(4):
        x = np.asarray(traj.noise(n), np.float64)
        a = traj.action(n)
        for t in range(S):
            before = [(c.phi_sp, c.phi_gl, c.phi_act) for c in oc.cells[t]]
            tr = []
            v, st = oc.chunk_step(x, a, O.SIGMAS[t], t, False, p, trace=tr)
            x_in0 = oc.model.patch_embed(x)
            for b in range(cfg.n_blocks):
                if st["decision"][b] != O.Decision.SKIP:
                    continue
                n_skips += 1
                cell = oc.cells[t][b]
                if refresh == 0:
                    assert cell.phi_sp is before[b][0] and cell.phi_gl is before[b][1]
                    continue
                xin = x_in0 if b == 0 else tr[b - 1]
                np.testing.assert_array_equal(cell.phi_sp[0], np.stack([xin[r] for r in rows]))
                means = np.stack([xin[c * npc:(c + 1) * npc].sum(axis=0) / npc for c in range(cfg.n_cams)])
                np.testing.assert_allclose(cell.phi_gl[0], means, rtol=1e-12, atol=1e-14)
                np.testing.assert_array_equal(cell.phi_act, a)
            x = x + (O.SIGMAS[t + 1] - O.SIGMAS[t]) * v
        oc.chunk_step(traj.clean(n), a, 0.0, S, True, p)
    assert n_skips > 0


# ------------------------------- lazy residual chaining (NEXT-2, reading c27)
def test_chained_fingerprint_explicit_loops():
    """Fingerprint of a chained input: sampled rows of base + r1 + r2 summed
    in float32 left to right and rounded once; global channel = per-camera
    mean of base plus the per-camera means of r1 and r2 (explicit loops)."""
    cfg = X.GROUPS_F32.replace(name="pin_chain_groups", dtype="bf16")
    oc = O.OracleXCache(cfg, X.make_weights(cfg))
    L, d = cfg.tokens, cfg.d_model
    base = O.to_bf16(rng.standard_normal((L, d)))
    rs = [O.to_bf16(0.1 * rng.standard_normal((L, d))) for _ in range(2)]
    sp, gl, _ = oc.chained_fingerprint(base, rs, np.array([0.1, 0.2]), 32)
    rows = O.group_fingerprint_rows(cfg.groups, cfg.frames, 32)
    for g, (V, gh, gw) in enumerate(cfg.groups):
        for c in range(V):
            for i, row in enumerate(rows[g][c]):
                for j in range(0, d, 7):
                    a = np.float32(base[row, j])
                    a = np.float32(a + np.float32(rs[0][row, j]))
                    a = np.float32(a + np.float32(rs[1][row, j]))
                    assert sp[g][c, i, j] == O.to_bf16(float(a))
    tok = 0
    for g, (V, gh, gw) in enumerate(cfg.groups):
        npc = cfg.frames * gh * gw
        for c in range(V):
            sl = slice(tok + c * npc, tok + (c + 1) * npc)
            for j in range(0, d, 5):
                want = sum(base[sl, j]) / npc + sum(rs[0][sl, j]) / npc + sum(rs[1][sl, j]) / npc
                assert gl[g][c, j] == pytest.approx(want, rel=1e-12, abs=1e-14)
        tok += V * npc


def test_chain_with_forced_recompute_is_the_plain_path():
    """No block ever skips, so nothing is chained: bitwise the same rollout."""
    cfg = X.TINY_F32
    a, _, _ = _run(cfg, O.GateParams(**FORCE_RECOMPUTE), 4)
    b, _, _ = _run(cfg, O.GateParams(chain=True, **FORCE_RECOMPUTE), 4)
    for x, y in zip(a["final"], b["final"]):
        np.testing.assert_array_equal(x, y)


def test_chain_fp32_matches_plain_reuse_closely():
    """fp32 model: chaining only changes the summation (float32 left to
    right instead of one block at a time in fp64) and the global channel
    (sum of means instead of mean of the sum, equal in exact arithmetic), so
    decisions agree and final latents agree to float32 rounding."""
    cfg = X.TINY_F32.replace(name="pin_chain_f32", n_chunks=5, n_blocks=4)
    # the back anchor computes after a run of skipped blocks: its input is
    # materialised from the chain
    kw = dict(tau_floor=0.5, margin=1.0, tau_dev=100.0, front_anchors=0, back_anchors=1)
    a, _, _ = _run(cfg, O.GateParams(**kw), 5)
    b, _, _ = _run(cfg, O.GateParams(chain=True, **kw), 5)
    da = np.array([[s["decision"] for s in ch] for ch in a["stats"]])
    db = np.array([[s["decision"] for s in ch] for ch in b["stats"]])
    np.testing.assert_array_equal(da, db)
    assert (da == O.Decision.SKIP).sum() >= 4
    for x, y in zip(a["final"], b["final"]):
        np.testing.assert_allclose(y, x, rtol=1e-5, atol=1e-5 * np.abs(x).max())


def test_chain_force_reuse_input_of_head_is_one_rounded_sum():
    """bf16, every gated block skipped after the warmup chunk: the head sees
    round(x_0 + r_hat_1 + ... + r_hat_{B-1}) summed in float32 block by
    block (the anchor block 0 computes), checked through the trace's last
    entry against an explicit loop over the cached residuals."""
    cfg = X.TINY_F32.replace(name="pin_chain_bf16", dtype="bf16", n_blocks=4)
    w = X.make_weights(cfg)
    traj = X.Trajectory(cfg, n_chunks=2)
    p = O.GateParams(chain=True, **FORCE_REUSE)
    oc = O.OracleXCache(cfg, w)
    S = cfg.n_steps
    for n in range(2):
        x = np.asarray(traj.noise(n), np.float64)
        for t in range(S):
            tr = []
            v, st = oc.chunk_step(x, traj.action(n), O.SIGMAS[t], t, False, p, trace=tr)
            if n == 1:
                assert list(st["decision"][1:]) == [O.Decision.SKIP] * (cfg.n_blocks - 1)
                acc = np.asarray(tr[0], np.float32)
                for b in range(1, cfg.n_blocks):
                    acc = (acc + np.asarray(oc.cells[t][b].r_hat, np.float32)).astype(np.float32)
                np.testing.assert_array_equal(tr[-1], O.to_bf16(acc.astype(np.float64)))
                # ... and the velocity is the head applied to that chained input
                _, hm = oc.model.cond(O.SIGMAS[t], traj.action(n))
                np.testing.assert_array_equal(v, oc.model.head(tr[-1], hm))
            x = x + (O.SIGMAS[t + 1] - O.SIGMAS[t]) * v
        oc.chunk_step(traj.clean(n), traj.action(n), 0.0, S, True, p)


def test_chain_sum_accumulates_in_float32():
    """1 + 2^-8 + 2^-24 + 2^-24 added left to right in float32: each 2^-24 is
    half a float32 ulp and is lost (ties to even), the sum stays on the bf16
    tie 1 + 2^-8 and rounds to even, 1.0.  The exact sum 1 + 2^-8 + 2^-23 is
    a float32 value above the tie and rounds up to 1 + 2^-7."""
    cfg = X.TINY_F32.replace(name="pin_chain_sum", dtype="bf16")
    oc = O.OracleXCache(cfg, X.make_weights(cfg))
    got = oc.chain_sum(np.array([1.0]), [np.array([2.0 ** -8]), np.array([2.0 ** -24]), np.array([2.0 ** -24])])
    assert got[0] == 1.0
    assert O.to_bf16(1.0 + 2.0 ** -8 + 2.0 ** -23) == 1.0 + 2.0 ** -7
