"""C-ABI library: loads, exports every declared symbol, host-side validation.
No GPU needed (no compute call is made)."""
import ctypes
import json
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LIB = os.path.join(ROOT, "paper_2604_20289_gb300", "libxcache.so")


@pytest.fixture(scope="module")
def xb():
    if not os.path.exists(LIB):
        from paper_2604_20289_gb300 import build
        build.build()
    from paper_2604_20289_gb300 import xcache
    return xcache


def declared_functions():
    names = []
    for h in ("xcache.h", "xcache_ops.h"):
        src = open(os.path.join(ROOT, "include", h)).read()
        src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
        names += re.findall(r"\b(xc_[a-z_0-9]+)\s*\(", src)
    return sorted(set(names))


def test_every_declared_symbol_is_exported(xb):
    lib = ctypes.CDLL(LIB)
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(xb.SIGNATURES), set(names) ^ set(xb.SIGNATURES)


def test_gate_defaults_are_table1(xb):
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "table1_defaults.json")))
    p = xb.gate_params()
    assert p.enabled == 1 and not p.replay_skip
    for k in ("front_anchors", "back_anchors", "warmup_chunks", "fp_tokens"):
        assert getattr(p, k) == g[k]
    for k in ("tau_floor", "margin", "alpha", "tau_dev"):
        assert getattr(p, k) == pytest.approx(g[k], rel=1e-7)
    assert p.max_skips == 0 and p.protect_step0 == 0


def test_host_validation_without_gpu(xb):
    # NULL context: state error, message available
    st = xb.LIB.xc_chunk_step(None, None, None, 1.0, 0, 0, None, None, None)
    assert st == xb.XC_ESTATE
    assert "NULL" in xb.last_error(None)
    # invalid model cfg is rejected before any CUDA call
    cfg = xb.ModelCfg(n_blocks=0, d_model=64, n_heads=4, head_dim=16, d_ffn=256, c_latent=16,
                      action_dim=2, n_cams=1, frames=1, grid_h=2, grid_w=2, kv_window_chunks=2,
                      n_denoise_steps=4, dtype=0, t_freq_dim=256, ln_eps=1e-6, rope_theta=1e4)
    w = xb.Weights()
    ctx = ctypes.c_void_p()
    assert xb.LIB.xc_init(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(ctx)) == xb.XC_EINVAL
    assert "n_blocks" in xb.last_error(None)
    cfg.n_blocks = 2
    cfg.dtype = 1            # bf16 with head_dim 16 is not supported
    assert xb.LIB.xc_init(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(ctx)) == xb.XC_EINVAL
    cfg.dtype = 0
    # NULL weights
    assert xb.LIB.xc_init(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(ctx)) == xb.XC_EINVAL
    assert "weight" in xb.last_error(None)
    # operator argument checks happen before any launch
    assert xb.LIB.xc_op_linear(1, 0, 0, 256, 64, None, None, None, None, None, None, None, None,
                               None) == xb.XC_EINVAL
    assert xb.LIB.xc_op_attention(1, 0, 1, 1, 64, None, None, None, None, None, 0, None) == xb.XC_EINVAL


def _cfg(xb, **kw):
    base = dict(n_blocks=2, d_model=64, n_heads=4, head_dim=16, d_ffn=256, c_latent=16, action_dim=2,
                n_cams=3, frames=2, grid_h=4, grid_w=4, kv_window_chunks=2, n_denoise_steps=4, dtype=0,
                t_freq_dim=256, ln_eps=1e-6, rope_theta=1e4)
    groups = kw.pop("groups", ())
    base.update(kw)
    c = xb.ModelCfg(**base)
    c.n_groups = len(groups)
    for i, (v, h, w) in enumerate(groups[:xb.XC_MAX_GROUPS]):
        c.group_cams[i], c.group_h[i], c.group_w[i] = v, h, w
    return c


@pytest.mark.parametrize("kw,msg", [
    (dict(groups=((2, 4, 4), (2, 2, 2))), "n_cams"),                  # 4 cameras in groups, n_cams 3
    (dict(groups=((3, 4, 4), (0, 2, 2))), "empty view group"),
    (dict(groups=((1, 1, 1),) * 5, n_cams=5), "n_groups"),              # more than XC_MAX_GROUPS
    (dict(kv_period=-1), "kv_period"),
    (dict(d_ctx=24, max_ctx=8), "d_ctx"),                              # not a multiple of 16
    (dict(d_ctx=32, max_ctx=0), "max_ctx"),
    (dict(dtype=1, head_dim=64, n_heads=4, d_model=256, d_ffn=256, d_ctx=32, max_ctx=8), "d_ctx"),
])
def test_model_cfg_validation_of_groups_kv_period_and_context(xb, kw, msg):
    """Rejected before any CUDA call (no GPU needed)."""
    cfg = _cfg(xb, **kw)
    w = xb.Weights()
    ctx = ctypes.c_void_p()
    assert xb.LIB.xc_init(ctypes.byref(cfg), ctypes.byref(w), None, ctypes.byref(ctx)) == xb.XC_EINVAL
    assert msg in xb.last_error(None), xb.last_error(None)


def test_set_context_without_context(xb):
    assert xb.LIB.xc_set_context(None, None, 1) == xb.XC_ESTATE
    assert "NULL" in xb.last_error(None)
