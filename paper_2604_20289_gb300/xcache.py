"""ctypes binding of libxcache.so (include/xcache.h, include/xcache_ops.h).

Argument marshalling only: every step of the chunk step runs in the CUDA
library.  Device buffers are torch CUDA tensors (passed by data_ptr());
streams are torch streams.  Importing this module loads the library and
raises if it is missing -- there is no fallback path.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libxcache.so")

XC_OK, XC_EINVAL, XC_ESTATE, XC_ENOMEM, XC_ECUDA, XC_ENUMERIC, XC_ETIMEOUT = range(7)
XC_F32, XC_BF16 = 0, 1
XC_DEC_FORCED, XC_DEC_COMPUTE, XC_DEC_SKIP = 0, 1, 2
XC_EPI_BIAS, XC_EPI_GELU, XC_EPI_RESID_GATE, XC_EPI_RESID_CACHE = 0, 1, 2, 3
XC_MAX_BLOCKS = 64
XC_MAX_GROUPS = 4
STATUS_NAMES = {0: "XC_OK", 1: "XC_EINVAL", 2: "XC_ESTATE", 3: "XC_ENOMEM", 4: "XC_ECUDA",
                5: "XC_ENUMERIC", 6: "XC_ETIMEOUT"}


class XCacheError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {msg}")
        self.status = status


class ModelCfg(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int) for n in (
        "n_blocks", "d_model", "n_heads", "head_dim", "d_ffn", "c_latent", "action_dim",
        "n_cams", "frames", "grid_h", "grid_w", "kv_window_chunks", "n_denoise_steps", "dtype",
        "t_freq_dim")] + [("ln_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                          ("kv_period", ctypes.c_int), ("n_groups", ctypes.c_int),
                          ("group_cams", ctypes.c_int * XC_MAX_GROUPS),
                          ("group_h", ctypes.c_int * XC_MAX_GROUPS),
                          ("group_w", ctypes.c_int * XC_MAX_GROUPS),
                          ("d_ctx", ctypes.c_int), ("max_ctx", ctypes.c_int)]


WEIGHT_NAMES = ("pe_w", "pe_b", "t_w1", "t_b1", "t_w2", "t_b2", "a_w1", "a_b1", "a_w2", "a_b2",
                "mod_w", "mod_b", "blk_mod", "qkv_w", "qkv_b", "o_w", "o_b", "f1_w", "f1_b",
                "f2_w", "f2_b", "head_w", "head_b", "head_tab", "out_w", "out_b",
                "ca_ln_w", "ca_ln_b", "ca_q_w", "ca_q_b", "ca_kv_w", "ca_kv_b", "ca_o_w", "ca_o_b")


class Weights(ctypes.Structure):
    _fields_ = [(n, ctypes.POINTER(ctypes.c_float)) for n in WEIGHT_NAMES]


class GateParams(ctypes.Structure):
    _fields_ = [("enabled", ctypes.c_int), ("tau_floor", ctypes.c_float), ("margin", ctypes.c_float),
                ("alpha", ctypes.c_float), ("tau_dev", ctypes.c_float), ("eps_dev", ctypes.c_float),
                ("front_anchors", ctypes.c_int), ("back_anchors", ctypes.c_int),
                ("warmup_chunks", ctypes.c_int), ("max_skips", ctypes.c_int),
                ("protect_step0", ctypes.c_int), ("step0_strict_tau", ctypes.c_float),
                ("fp_tokens", ctypes.c_int), ("fp_refresh", ctypes.c_int), ("fp_linear", ctypes.c_int),
                ("chain", ctypes.c_int),
                ("replay_skip", ctypes.POINTER(ctypes.c_uint8)),
                ("replay_table", ctypes.c_void_p)]


class StepStats(ctypes.Structure):
    _fields_ = [("n_blocks", ctypes.c_int), ("chunk_index", ctypes.c_int),
                ("decision", ctypes.c_uint8 * XC_MAX_BLOCKS),
                ("s_cos", ctypes.c_float * XC_MAX_BLOCKS),
                ("d_max", ctypes.c_float * XC_MAX_BLOCKS),
                ("tau_cos", ctypes.c_float * XC_MAX_BLOCKS)]


class ProfileRec(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int), ("block", ctypes.c_int), ("pass_seq", ctypes.c_int),
                ("decision", ctypes.c_int), ("chunk", ctypes.c_int), ("n_keys", ctypes.c_int),
                ("ms", ctypes.c_float)]


KERNEL_KINDS = ("cond", "embed", "gate", "ln", "qkv", "attn", "oproj", "ffn1", "ffn2", "reuse", "head",
                "xattn", "chain")

_P = ctypes.c_void_p
_I = ctypes.c_int
_F = ctypes.c_float
_L = ctypes.c_long
SIGNATURES = {
    "xc_gate_params_default": (None, [ctypes.POINTER(GateParams)]),
    "xc_init": (_I, [ctypes.POINTER(ModelCfg), ctypes.POINTER(Weights), _P, ctypes.POINTER(_P)]),
    "xc_chunk_step": (_I, [_P, _P, _P, _F, _I, _I, ctypes.POINTER(GateParams), _P,
                           ctypes.POINTER(StepStats)]),
    "xc_reset": (_I, [_P]),
    "xc_set_context": (_I, [_P, _P, _I]),
    "xc_destroy": (None, [_P]),
    "xc_last_error": (ctypes.c_char_p, [_P]),
    "xc_euler_update": (_I, [_P, _P, _P, _F, _L]),
    "xc_set_block_trace": (_I, [_P, _P]),
    "xc_sync": (_I, [_P]),
    "xc_chunk_index": (_I, [_P]),
    "xc_debug_fail_alloc": (None, [_I]),
    "xc_debug_expire_wait": (_I, [_P]),
    "xc_launch_count": (ctypes.c_longlong, [_P]),
    "xc_profile_start": (_I, [_P, ctypes.c_uint, _I]),
    "xc_profile_stop": (_I, [_P, ctypes.POINTER(ProfileRec), _I, ctypes.POINTER(_I)]),
    "xc_op_linear": (_I, [_I, _I, _I, _I, _I, _P, _P, _P, _P, _P, _P, _P, _P, _P]),
    "xc_op_qkv_rope": (_I, [_I, _I, _I, _I, _I, _I, _I, _I, _F, _P, _P, _P, _P, _P, _P, _P]),
    "xc_op_attention_workspace_bytes": (ctypes.c_size_t, [_I, _I]),
    "xc_op_attention": (_I, [_I, _I, _I, _I, _I, _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "xc_op_ln_mod": (_I, [_I, _I, _I, _F, _P, _P, _P, _P, _P]),
    "xc_op_residual_reuse": (_I, [_I, _L, _P, _P, _P, _P]),
    "xc_op_device_error": (_I, []),
    "xc_op_gate_workspace_bytes": (ctypes.c_size_t, [_I, _I, _I, _I]),
    "xc_op_gate": (_I, [_I, _I, _I, _I, _P, _P, _I, _P, _P, _P, _P, _I, _I, _I, ctypes.POINTER(GateParams),
                        _P, _P, _P, _P, _P, ctypes.c_size_t, _P]),
    "xc_op_gate_static": (_I, [_I, _I, _I, _I, _P, _P, _I, _P, _P, _P, _P, _I, _I, _I,
                               ctypes.POINTER(GateParams), _P, _P, _P, _P, _P]),
}


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"{LIB_PATH} is missing: build it with "
                          "`python -m paper_2604_20289_gb300.build` (no fallback path exists)")
    lib = ctypes.CDLL(LIB_PATH)
    for name, (res, args) in SIGNATURES.items():
        f = getattr(lib, name)
        f.restype = res
        f.argtypes = args
    return lib


LIB = _load()


def last_error(ctx=None) -> str:
    return LIB.xc_last_error(ctx).decode(errors="replace")


def check(status: int, ctx=None):
    if status != XC_OK:
        raise XCacheError(status, last_error(ctx))


def _ptr(t) -> int | None:
    """Device pointer of a torch tensor, host pointer of a numpy array, None."""
    if t is None:
        return None
    if isinstance(t, np.ndarray):
        return t.ctypes.data
    return t.data_ptr()


def _stream(stream) -> int | None:
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    return getattr(stream, "cuda_stream", stream)


def dtype_code(dtype) -> int:
    return {"f32": XC_F32, "bf16": XC_BF16, XC_F32: XC_F32, XC_BF16: XC_BF16}[dtype]


def model_cfg(cfg) -> ModelCfg:
    """ModelCfg from any object with the shape attributes (e.g. xc_inputs.ModelCfg);
    optional ``view_groups`` ((cameras, grid_h, grid_w), ...) and ``kv_period``."""
    m = ModelCfg(cfg.n_blocks, cfg.d_model, cfg.n_heads, cfg.head_dim, cfg.d_ffn, cfg.c_latent,
                 cfg.action_dim, cfg.n_cams, cfg.frames, cfg.grid_h, cfg.grid_w, cfg.kv_window,
                 cfg.n_steps, dtype_code(cfg.dtype), cfg.t_freq, cfg.ln_eps, cfg.rope_theta)
    m.kv_period = int(getattr(cfg, "kv_period", 0))
    groups = tuple(getattr(cfg, "view_groups", ()))
    if len(groups) > XC_MAX_GROUPS:
        raise ValueError(f"at most {XC_MAX_GROUPS} view groups")
    m.n_groups = len(groups)
    for i, (c, h, w) in enumerate(groups):
        m.group_cams[i], m.group_h[i], m.group_w[i] = c, h, w
    m.d_ctx = int(getattr(cfg, "d_ctx", 0))
    m.max_ctx = int(getattr(cfg, "max_ctx", 0))
    return m


def gate_params(**kw) -> GateParams:
    """Table 1 defaults, overridden by keyword (replay_skip: sequence of 0/1;
    replay_table: torch CUDA uint8 tensor [n_denoise_steps, n_blocks], kept
    alive by the caller)."""
    p = GateParams()
    LIB.xc_gate_params_default(ctypes.byref(p))
    replay = kw.pop("replay_skip", None)
    table = kw.pop("replay_table", None)
    if table is not None:
        p.replay_table = table.data_ptr()
    for k, v in kw.items():
        if not hasattr(p, k):
            raise KeyError(k)
        setattr(p, k, int(v) if isinstance(getattr(p, k), int) else float(v))
    if replay is not None:
        arr = (ctypes.c_uint8 * len(replay))(*[1 if r else 0 for r in replay])
        p._replay_keepalive = arr
        p.replay_skip = ctypes.cast(arr, ctypes.POINTER(ctypes.c_uint8))
    return p


class XCache:
    """One X-Cache context (xc_init .. xc_destroy) on the current CUDA device."""

    def __init__(self, cfg, weights: dict, stream=None):
        self.cfg = cfg
        self._c_cfg = model_cfg(cfg)
        # numpy arrays (host) or contiguous float32 torch CUDA tensors (device)
        keep = {k: (weights[k] if hasattr(weights[k], "data_ptr") else
                    np.ascontiguousarray(weights[k], dtype=np.float32))
                for k in WEIGHT_NAMES if k in weights}
        w = Weights(*[ctypes.cast(_ptr(keep[k]), ctypes.POINTER(ctypes.c_float)) if k in keep else None
                      for k in WEIGHT_NAMES])
        ctx = ctypes.c_void_p()
        self._stream = _stream(stream)
        check(LIB.xc_init(ctypes.byref(self._c_cfg), ctypes.byref(w), self._stream, ctypes.byref(ctx)))
        self.ctx = ctx

    def close(self):
        if getattr(self, "ctx", None):
            LIB.xc_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def chunk_step(self, latent, action, sigma: float, step: int, is_kv_update: bool = False,
                   gate: GateParams | None = None, v_out=None, want_stats: bool = True):
        """latent / v_out: torch CUDA tensors or numpy float32 host arrays."""
        act = np.ascontiguousarray(action, dtype=np.float32)
        st = StepStats() if want_stats else None
        check(LIB.xc_chunk_step(self.ctx, _ptr(latent), act.ctypes.data, float(sigma), int(step),
                                int(bool(is_kv_update)), ctypes.byref(gate) if gate is not None else None,
                                _ptr(v_out), ctypes.byref(st) if st is not None else None), self.ctx)
        if st is None:
            return None
        B = st.n_blocks
        return dict(chunk=st.chunk_index,
                    decision=np.array(st.decision[:B], dtype=np.int64),
                    s_cos=np.array(st.s_cos[:B], dtype=np.float64),
                    d_max=np.array(st.d_max[:B], dtype=np.float64),
                    tau=np.array(st.tau_cos[:B], dtype=np.float64))

    def reset(self):
        check(LIB.xc_reset(self.ctx), self.ctx)

    def set_context(self, tokens):
        """Condition tokens [n_ctx, d_ctx] (torch CUDA tensor or numpy float32)."""
        if isinstance(tokens, np.ndarray):
            tokens = np.ascontiguousarray(tokens, dtype=np.float32)
        check(LIB.xc_set_context(self.ctx, _ptr(tokens), int(tokens.shape[0])), self.ctx)

    def euler(self, x, v, dsigma: float):
        check(LIB.xc_euler_update(self.ctx, _ptr(x), _ptr(v), float(dsigma), x.numel()), self.ctx)

    def set_trace(self, buf):
        check(LIB.xc_set_block_trace(self.ctx, _ptr(buf)), self.ctx)

    def sync(self):
        check(LIB.xc_sync(self.ctx), self.ctx)

    @property
    def chunk_index(self) -> int:
        return LIB.xc_chunk_index(self.ctx)

    @property
    def launch_count(self) -> int:
        return LIB.xc_launch_count(self.ctx)

    def profile_start(self, kinds=KERNEL_KINDS, capacity: int = 65536):
        mask = 0
        for k in kinds:
            mask |= 1 << KERNEL_KINDS.index(k)
        self._prof_cap = capacity
        check(LIB.xc_profile_start(self.ctx, mask, capacity), self.ctx)

    def profile_stop(self) -> list:
        """Synchronises; returns dicts (kind, block, pass_seq, decision, chunk, n_keys, ms)."""
        cap = getattr(self, "_prof_cap", 65536)
        recs = (ProfileRec * cap)()
        n = ctypes.c_int()
        check(LIB.xc_profile_stop(self.ctx, recs, cap, ctypes.byref(n)), self.ctx)
        return [dict(kind=KERNEL_KINDS[r.kind], block=r.block, pass_seq=r.pass_seq,
                     decision=r.decision, chunk=r.chunk, n_keys=r.n_keys, ms=r.ms)
                for r in recs[:min(n.value, cap)]]


# --------------------------------------------------------------- operators
def op_linear(dtype, epilogue, A, Wt, bias, out, gate=None, resid=None, xin=None, rhat=None,
              stream=None):
    M, K = A.shape
    N = Wt.shape[0]
    check(LIB.xc_op_linear(dtype_code(dtype), epilogue, M, N, K, _ptr(A), _ptr(Wt), _ptr(bias),
                           _ptr(gate), _ptr(resid), _ptr(xin), _ptr(out), _ptr(rhat),
                           _stream(stream)))


def op_qkv_rope(dtype, n_cams, frames, gh, gw, chunk, head_dim, theta, A, Wt, bias, q, k, v,
                stream=None):
    d = A.shape[1]
    check(LIB.xc_op_qkv_rope(dtype_code(dtype), n_cams, frames, gh, gw, chunk, d, head_dim,
                             float(theta), _ptr(A), _ptr(Wt), _ptr(bias), _ptr(q), _ptr(k), _ptr(v),
                             _stream(stream)))


def op_attention_workspace_bytes(dtype, head_dim):
    return LIB.xc_op_attention_workspace_bytes(dtype_code(dtype), head_dim)


def op_attention(dtype, n_heads, head_dim, q, k, v, o, workspace=None, stream=None):
    """workspace: None (one SM per unit), "auto" (a device buffer of
    op_attention_workspace_bytes is allocated for the call) or a device
    tensor of at least that many bytes."""
    if isinstance(workspace, str) and workspace == "auto":
        import torch
        nb = op_attention_workspace_bytes(dtype, head_dim)
        workspace = torch.empty(max(nb, 1), dtype=torch.uint8, device=q.device) if nb else None
    ws_ptr = _ptr(workspace) if workspace is not None else None
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    check(LIB.xc_op_attention(dtype_code(dtype), q.shape[0], k.shape[0], n_heads, head_dim, _ptr(q),
                              _ptr(k), _ptr(v), _ptr(o), ws_ptr, ws_bytes, _stream(stream)))


def op_ln_mod(dtype, x, shift, scale, out, eps=1e-6, stream=None):
    M, d = x.shape
    check(LIB.xc_op_ln_mod(dtype_code(dtype), M, d, float(eps), _ptr(x), _ptr(shift), _ptr(scale),
                           _ptr(out), _stream(stream)))


def op_residual_reuse(dtype, x, rhat, out, stream=None):
    check(LIB.xc_op_residual_reuse(dtype_code(dtype), x.numel(), _ptr(x), _ptr(rhat), _ptr(out),
                                   _stream(stream)))


def op_device_error() -> int:
    return LIB.xc_op_device_error()


class GateCell(ctypes.Structure):
    """xc_gate_cell: per-(t, b) gate state (32 bytes)."""
    _fields_ = [("ema", ctypes.c_double), ("has_hist", ctypes.c_int), ("stale", ctypes.c_int),
                ("valid", ctypes.c_int), ("active", ctypes.c_int), ("pad", ctypes.c_int * 2)]


def op_gate_workspace_bytes(dtype, n_cams, tokens_per_cam, d) -> int:
    return LIB.xc_op_gate_workspace_bytes(dtype_code(dtype), n_cams, tokens_per_cam, d)


def op_gate(dtype, n_cams, tokens_per_cam, x, fp_rows, phi, phi_act, cell, action, mode, step,
            gate, flag, s_cos, d_max, tau, workspace, stream=None):
    """x, fp_rows [n_cams, kfp] int32, phi, phi_act, cell (uint8 tensor of 32 bytes), flag,
    s_cos, d_max, tau, workspace: torch CUDA tensors; action: numpy float32."""
    act = np.ascontiguousarray(action, dtype=np.float32)
    check(LIB.xc_op_gate(dtype_code(dtype), n_cams, tokens_per_cam, x.shape[1], _ptr(x), _ptr(fp_rows),
            fp_rows.shape[1], _ptr(phi), _ptr(phi_act), _ptr(cell), act.ctypes.data, act.size, mode,
            step, ctypes.byref(gate) if gate is not None else None, _ptr(flag), _ptr(s_cos),
            _ptr(d_max), _ptr(tau), _ptr(workspace), workspace.numel() * workspace.element_size(),
            _stream(stream)))
