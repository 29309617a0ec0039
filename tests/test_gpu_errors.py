"""Error paths of the C ABI on a GPU: injected device-allocation failures in
xc_init (every allocation in turn) report XC_ENOMEM, leak nothing, and leave
the library usable."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

import xc_inputs as X  # noqa: E402

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2604_20289_gb300 import xcache as xb  # noqa: E402


def test_injected_allocation_failures_in_init():
    cfg = X.MID_HD64
    w = X.make_weights(cfg)
    traj = X.Trajectory(cfg, n_chunks=1)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info()[0]
    failures = 0
    try:
        for n in range(1, 101):
            xb.LIB.xc_debug_fail_alloc(n)
            try:
                xc = xb.XCache(cfg, w)
            except xb.XCacheError as e:
                assert e.status == xb.XC_ENOMEM, str(e)
                assert "injected" in str(e)
                failures += 1
            else:
                xc.close()
    finally:
        xb.LIB.xc_debug_fail_alloc(0)
    assert failures >= 20                       # the weights, ring, caches, scratch: every one in turn
    torch.cuda.synchronize()
    assert free0 - torch.cuda.mem_get_info()[0] <= 16 << 20, "device memory leaked by failed inits"
    # the library still works: a full context and one pass
    xc = xb.XCache(cfg, w)
    x = torch.tensor(traj.noise(0), device="cuda")
    v = torch.empty_like(x)
    st = xc.chunk_step(x, traj.action(0), 1.0, 0, False, xb.gate_params(), v_out=v)
    xc.sync()
    assert np.isfinite(v.cpu().numpy()).all() and st["chunk"] == 0
    xc.close()


def test_expired_device_wait_is_reported_and_the_context_stays_usable():
    """A bounded wait that runs out (nothing completes the barrier phase it
    waits for) records its bit in the error word: xc_sync reports
    XC_ETIMEOUT once, and the same context then runs a pass that gives the
    same velocity as before."""
    cfg = X.TINY_F32
    w = X.make_weights(cfg)
    traj = X.Trajectory(cfg, n_chunks=1)
    xc = xb.XCache(cfg, w)
    x = torch.tensor(traj.noise(0), device="cuda")
    v0, v1 = torch.empty_like(x), torch.empty_like(x)
    xc.chunk_step(x, traj.action(0), 1.0, 0, False, xb.gate_params(), v_out=v0)
    xc.reset()
    assert xb.LIB.xc_debug_expire_wait(xc.ctx) == xb.XC_OK
    with pytest.raises(xb.XCacheError) as e:
        xc.sync()
    assert e.value.status == xb.XC_ETIMEOUT
    xc.sync()                                   # reported once, then cleared
    xc.chunk_step(x, traj.action(0), 1.0, 0, False, xb.gate_params(), v_out=v1)
    xc.sync()
    assert torch.equal(v0, v1)
    xc.close()
    # the operator entry points' error word
    assert xb.op_device_error() == 0
    assert xb.LIB.xc_debug_expire_wait(None) == xb.XC_OK
    assert xb.op_device_error() != 0
    assert xb.op_device_error() == 0
