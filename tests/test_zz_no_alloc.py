"""The allocation-free gate entry point (xc_op_gate_static) against the
caller-workspace gate (xc_op_gate), through the C ABI, on two calls in a row.

xc_op_gate_static exists for callers that cannot call cudaMalloc when they
call in (a runtime that owns the process's only device allocator, a
device-memory budget fixed at start-up, a latency-critical loop that must not
allocate): its scratch is a file-scope device array instead of a workspace.  Both run the same deterministic kernel, so the
outputs must agree within the gate tests' tolerances (abs 1e-6 on the metrics,
exact decisions and cached fingerprints).  This file is collected last and
passes both alone in a fresh process and after the other tests."""
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


def _state(phi0, pa0, cell):
    return dict(phi=phi0.clone(), phi_act=pa0.clone(),
                cell=torch.frombuffer(bytearray(bytes(cell)), dtype=torch.uint8).to(DEV),
                flag=torch.zeros(1, dtype=torch.uint8, device=DEV),
                stats=torch.full((3,), float("nan"), device=DEV))


def _call_static(dtype, V, npc, x, rows, st, action, mode, step, gate):
    act = np.ascontiguousarray(action, dtype=np.float32)
    xb.check(xb.LIB.xc_op_gate_static(
        xb.dtype_code(dtype), V, npc, x.shape[1], x.data_ptr(), rows.data_ptr(), rows.shape[1],
        st["phi"].data_ptr(), st["phi_act"].data_ptr(), st["cell"].data_ptr(), act.ctypes.data, act.size,
        mode, step, gate, st["flag"].data_ptr(), st["stats"][0:1].data_ptr(), st["stats"][1:2].data_ptr(),
        st["stats"][2:3].data_ptr(), torch.cuda.current_stream().cuda_stream))


def _call_workspace(dtype, V, npc, x, rows, st, action, mode, step, gate, ws):
    xb.op_gate(dtype, V, npc, x, rows, st["phi"], st["phi_act"], st["cell"], action, mode, step, gate,
               st["flag"], st["stats"][0:1], st["stats"][1:2], st["stats"][2:3], ws)


def _compare(a, b):
    torch.cuda.synchronize()
    assert int(a["flag"].item()) == int(b["flag"].item())
    sa, sb = a["stats"].cpu().numpy(), b["stats"].cpu().numpy()
    assert np.array_equal(np.isnan(sa), np.isnan(sb))
    np.testing.assert_allclose(sa[~np.isnan(sa)], sb[~np.isnan(sb)], rtol=0, atol=1e-6)
    ca = xb.GateCell.from_buffer_copy(bytes(a["cell"].cpu().numpy().tobytes()))
    cb = xb.GateCell.from_buffer_copy(bytes(b["cell"].cpu().numpy().tobytes()))
    assert (ca.has_hist, ca.stale, ca.valid, ca.active) == (cb.has_hist, cb.stale, cb.valid, cb.active)
    assert abs(ca.ema - cb.ema) <= 1e-6
    np.testing.assert_array_equal(a["phi_act"].cpu().numpy(), b["phi_act"].cpu().numpy())
    pa, pb = a["phi"].cpu().numpy(), b["phi"].cpu().numpy()
    np.testing.assert_allclose(pa, pb, rtol=1e-6, atol=1e-7)


@pytest.mark.parametrize("cfg", [X.SMALL_BF16, X.TINY_F32], ids=lambda c: c.name)
def test_static_scratch_gate_matches_workspace_gate_on_two_calls(cfg):
    V, d = cfg.n_cams, cfg.d_model
    npc = cfg.frames * cfg.grid_h * cfg.grid_w
    L = V * npc
    bf = cfg.dtype == "bf16"
    dt = torch.bfloat16 if bf else torch.float32
    xs = []
    for name in ("nz_x0", "nz_x1", "nz_x2"):
        a = X.random_tensor(21, name, (L, d), std=1.3, bf16=bf)
        xs.append(a)
    x1 = 0.96 * xs[0] + 0.28 * xs[1]
    x2 = 0.96 * x1 + 0.28 * xs[2]
    dev_x = [torch.from_numpy(np.ascontiguousarray(v, dtype=np.float32)).to(DEV).to(dt) for v in (x1, x2)]
    rows = O.fingerprint_rows(V, cfg.frames, cfg.grid_h, cfg.grid_w, 32).astype(np.int32)
    rows_t = torch.from_numpy(rows).to(DEV)
    kfp = rows.shape[1]
    # cached fingerprint of xs[0] in the active half 0
    x0 = xs[0].astype(np.float64)
    n_all = V * kfp * d + V * d
    phi = np.zeros((2, n_all), np.float32)
    phi[0] = np.concatenate([x0[rows].ravel(), x0.reshape(V, npc, d).mean(axis=1).ravel()])
    pa = np.zeros((2, 8), np.float32)
    pa[0, :2] = [0.5, -0.45]
    phi0, pa0 = torch.from_numpy(phi).to(DEV), torch.from_numpy(pa).to(DEV)
    cell = xb.GateCell(0.97, 1, 0, 1, 0)
    gate = xb.gate_params(tau_floor=float(np.float32(0.9)), tau_dev=float(np.float32(4.0)))
    ws = torch.zeros(xb.op_gate_workspace_bytes(cfg.dtype, V, npc, d), dtype=torch.uint8, device=DEV)
    A, B = _state(phi0, pa0, cell), _state(phi0, pa0, cell)
    actions = (np.array([0.51, -0.44], np.float32), np.array([0.52, -0.46], np.float32))
    for call in range(2):
        _call_workspace(cfg.dtype, V, npc, dev_x[call], rows_t, A, actions[call], 1, 1, gate, ws)
        _call_static(cfg.dtype, V, npc, dev_x[call], rows_t, B, actions[call], 1, 1, gate)
        _compare(A, B)
        assert not np.isnan(B["stats"].cpu().numpy()).any()
    assert xb.op_device_error() == 0


def test_static_scratch_gate_rejects_geometry_beyond_its_maximum():
    buf = torch.zeros(1024, dtype=torch.uint8, device=DEV)
    p = buf.data_ptr()
    act = np.zeros(2, np.float32)
    # 128 cameras x d 262144: 65536 (camera, column slice) CTAs, each with 8
    # fp32 partial metrics (32 bytes) -- about 2 MiB of scratch, twice the maximum
    need = xb.op_gate_workspace_bytes("bf16", 128, 8, 262144)
    assert need > 2 * (1 << 20)
    st = xb.LIB.xc_op_gate_static(xb.XC_BF16, 128, 8, 262144, p, p, 1, p, p, p, act.ctypes.data, 2, 1, 1,
                                  None, p, p, p, p, None)
    assert st == xb.XC_EINVAL
    assert "static maximum" in xb.last_error(None)
