"""Gate kernel parity (xc_op_gate through the C ABI) against the oracle's
fingerprint, Eq. 5-6 metrics and Eq. 7-9 decision on seeded inputs.

Tolerances: the spatial sample is copied exactly (bf16 / fp32 values are
exact in fp32); per-camera means differ only by fp32 vs fp64 summation
(rel 1e-6); cosines and d_max are reduced in fp64 from fp32 partials
(abs 1e-6 / rel 1e-6); the threshold is computed in fp64 on both sides from
the same fp32 knobs, so it matches to 1e-12."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

import oracle as O  # noqa: E402
import xc_inputs as X  # noqa: E402

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2604_20289_gb300 import xcache as xb  # noqa: E402

DEV = torch.device("cuda")
f32 = lambda v: float(np.float32(v))  # noqa: E731


class GateCase:
    """A block input x and a cached fingerprint taken from a correlated x_prev."""

    def __init__(self, cfg, rho, seed=11, act_delta=0.02):
        self.cfg = cfg
        V, npc, d = cfg.n_cams, cfg.frames * cfg.grid_h * cfg.grid_w, cfg.d_model
        L = V * npc
        bf = cfg.dtype == "bf16"
        xp = X.random_tensor(seed, "gx_prev", (L, d), std=1.5).astype(np.float64) + 0.3
        nz = X.random_tensor(seed, "gx_noise", (L, d), std=1.5).astype(np.float64)
        x = rho * xp + np.sqrt(1 - rho * rho) * nz
        R = (lambda a: O.to_bf16(a)) if bf else (lambda a: a.astype(np.float32).astype(np.float64))
        self.x, self.x_prev = R(x), R(xp)
        self.rows = O.fingerprint_rows(V, cfg.frames, cfg.grid_h, cfg.grid_w, 32)
        self.kfp = self.rows.shape[1]
        self.V, self.npc, self.d = V, npc, d
        self.act_prev = np.array([0.5, -0.4], np.float32)
        self.act = (self.act_prev + act_delta).astype(np.float32)

    def fingerprint(self, x, act):
        sp = x[self.rows]
        gl = x.reshape(self.V, self.npc, -1).mean(axis=1)
        return sp, gl, act.astype(np.float64)

    def device_state(self, cell_kw):
        sp, gl, _ = self.fingerprint(self.x_prev, self.act_prev)
        n_all = sp.size + gl.size
        phi = np.zeros((2, n_all), np.float32)
        active = cell_kw.get("active", 0)
        phi[active] = np.concatenate([sp.ravel(), gl.ravel()]).astype(np.float32)
        pa = np.zeros((2, 8), np.float32)
        pa[active, :2] = self.act_prev
        cell = xb.GateCell(cell_kw.get("ema", 0.0), cell_kw.get("has_hist", 0), cell_kw.get("stale", 0),
                           cell_kw.get("valid", 1), active)
        cell_t = torch.frombuffer(bytearray(bytes(cell)), dtype=torch.uint8).to(DEV)
        dt = torch.bfloat16 if self.cfg.dtype == "bf16" else torch.float32
        return dict(x=torch.from_numpy(self.x.astype(np.float32)).to(DEV).to(dt),
                    rows=torch.from_numpy(self.rows.astype(np.int32)).to(DEV),
                    phi=torch.from_numpy(phi).to(DEV), phi_act=torch.from_numpy(pa).to(DEV), cell=cell_t,
                    flag=torch.zeros(1, dtype=torch.uint8, device=DEV),
                    stats=torch.full((3,), float("nan"), device=DEV))


def run_gate(case, st, mode, step, gp, ws=None, x=None):
    if ws is None:
        nb = xb.op_gate_workspace_bytes(case.cfg.dtype, case.V, case.npc, case.d)
        ws = torch.zeros(nb, dtype=torch.uint8, device=DEV)
    xb.op_gate(case.cfg.dtype, case.V, case.npc, st["x"] if x is None else x, st["rows"], st["phi"],
               st["phi_act"], st["cell"], case.act, mode, step, gp, st["flag"], st["stats"][0:1],
               st["stats"][1:2], st["stats"][2:3], ws)
    torch.cuda.synchronize()
    assert xb.op_device_error() == 0
    return ws


def read_cell(st):
    return xb.GateCell.from_buffer_copy(bytes(st["cell"].cpu().numpy().tobytes()))


def oracle_eval(case, cell_kw, p, step):
    sp, gl, ac = case.fingerprint(case.x, case.act)
    psp, pgl, pac = case.fingerprint(case.x_prev, case.act_prev)
    s = min(O.cosine(sp, psp.astype(np.float32)), O.cosine(gl, pgl.astype(np.float32)),
            O.cosine(ac, pac))
    d = O.max_token_deviation(sp, psp, p.eps_dev)
    cell = O.GateCell(valid=True, ema=cell_kw.get("ema", 0.0), has_hist=bool(cell_kw.get("has_hist", 0)),
                      stale=cell_kw.get("stale", 0))
    skip, tau = O.gate_decide(cell, s, d, step, p)
    return s, d, tau, skip, cell


# small model (8 column slices x 6 cameras, rows split over the SMs), tiny fp32
# model (one CTA per camera), 1.3B and 14B block inputs (d 1536 and 5120)
CASES = [(X.SMALL_BF16, 0.97), (X.TINY_F32, 0.95), (X.DIT_1P3B.replace(n_blocks=1), 0.96),
         (X.DIT_14B.replace(n_blocks=1), 0.96)]


@pytest.mark.parametrize("cfg,rho", CASES, ids=lambda v: getattr(v, "name", str(v)))
@pytest.mark.parametrize("cell_kw", [dict(), dict(has_hist=1, ema=0.99, stale=1),
                                     dict(has_hist=1, ema=0.90, stale=2, active=1)],
                         ids=["first", "ema_high", "ema_low_stale"])
def test_gate_eval_matches_oracle(cfg, rho, cell_kw):
    case = GateCase(cfg, rho)
    kw = dict(tau_floor=f32(0.93), margin=f32(0.02), alpha=f32(0.3), tau_dev=f32(4.0), max_skips=2)
    p = O.GateParams(**kw)
    st = case.device_state(cell_kw)
    run_gate(case, st, 1, 1, xb.gate_params(**kw))
    s, d, tau, skip, ocell = oracle_eval(case, cell_kw, p, 1)
    g_s, g_d, g_tau = st["stats"].cpu().numpy().astype(np.float64)
    assert abs(g_s - s) <= 1e-6, (g_s, s)
    assert abs(g_d - d) <= 1e-6 * d, (g_d, d)
    assert abs(g_tau - tau) <= 1e-6, (g_tau, tau)
    if abs(s - tau) > 1e-3 * tau and abs(d - p.tau_dev) > 1e-3 * p.tau_dev:
        assert int(st["flag"].item()) == (xb.XC_DEC_SKIP if skip else xb.XC_DEC_COMPUTE)
    c = read_cell(st)
    assert abs(c.ema - ocell.ema) <= 1e-6 and c.has_hist == 1 and c.stale == ocell.stale
    active0 = cell_kw.get("active", 0)
    assert c.active == (active0 if skip else active0 ^ 1)
    # the current fingerprint went to the inactive half
    sp, gl, _ = case.fingerprint(case.x, case.act)
    cur = st["phi"][active0 ^ 1].cpu().numpy().astype(np.float64)
    np.testing.assert_array_equal(cur[:sp.size], sp.ravel())
    np.testing.assert_allclose(cur[sp.size:], gl.ravel(), rtol=1e-5, atol=1e-6)
    np.testing.assert_array_equal(st["phi_act"][active0 ^ 1, :2].cpu().numpy(), case.act)


@pytest.mark.parametrize("cfg,rho", CASES[:2], ids=lambda v: getattr(v, "name", str(v)))
def test_gate_refresh_and_replay_and_reuse_of_workspace(cfg, rho):
    case = GateCase(cfg, rho)
    p = xb.gate_params(tau_floor=f32(0.5), tau_dev=f32(100.0))
    st = case.device_state(dict(valid=0))
    ws = run_gate(case, st, 1, 0, p)                       # invalid cache: forced, refreshed
    c = read_cell(st)
    assert int(st["flag"].item()) == xb.XC_DEC_FORCED and c.valid == 1 and c.active == 1
    assert np.isnan(st["stats"].cpu().numpy()).all()
    run_gate(case, st, 1, 2, p, ws=ws)                     # same input again: cos 1, d 0 -> skip
    assert int(st["flag"].item()) == xb.XC_DEC_SKIP
    assert st["stats"][0].item() == pytest.approx(1.0, abs=1e-6) and st["stats"][1].item() == 0.0
    rp = xb.gate_params(tau_floor=f32(0.5), tau_dev=f32(100.0), replay_skip=[0])
    run_gate(case, st, 1, 2, rp, ws=ws)                    # decision replay overrides the test
    assert int(st["flag"].item()) == xb.XC_DEC_COMPUTE
    run_gate(case, st, 0, 1, p, ws=ws)                     # refresh-only mode
    assert int(st["flag"].item()) == xb.XC_DEC_FORCED


def test_gate_workspace_too_small_is_rejected():
    case = GateCase(X.TINY_F32, 0.9)
    st = case.device_state({})
    nb = xb.op_gate_workspace_bytes("f32", case.V, case.npc, case.d)
    with pytest.raises(xb.XCacheError) as e:
        run_gate(case, st, 1, 1, None, ws=torch.zeros(nb - 1, dtype=torch.uint8, device=DEV))
    assert e.value.status == xb.XC_EINVAL
