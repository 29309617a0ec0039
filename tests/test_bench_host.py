"""Host logic of bench.py, on the CPU: the roofline peak chosen by the timed
region's clocks, the algorithmic work per kernel kind, the traffic record's
source-hash check, the oracle cost fit, the predicted speedup and the KV-pass
schedule."""
import hashlib
import json
import os
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2604_20289_gb300 import xcache as xb  # noqa: E402

PEAKS = {"hbm_gbs": 6675.5, "bf16_tflops": 1953.3, "bf16_tflops_sustained": 1741.5}


def test_peak_follows_the_clocks():
    full = {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": []}
    capped = {"sm_mhz": 1867.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"]}
    low = {"sm_mhz": 1500.0, "sm_max_mhz": 2070.0, "reasons": []}      # held low with no reason given
    assert bench.choose_peak(PEAKS, full) == (1953.3, "bf16_tflops")
    assert bench.choose_peak(PEAKS, capped) == (1741.5, "bf16_tflops_sustained")
    assert bench.choose_peak(PEAKS, low) == (1741.5, "bf16_tflops_sustained")
    # within 3 % of the maximum counts as holding it
    assert bench.choose_peak(PEAKS, {"sm_mhz": 2025.0, "sm_max_mhz": 2070.0, "reasons": []})[1] == "bf16_tflops"


def test_algorithmic_work_of_the_14b_block():
    cfg = bench.WORKLOADS["14b"]
    L, d, F, keys = 12960, 5120, 13824, 38880
    assert (cfg.tokens, cfg.d_model, cfg.d_ffn, cfg.kv_window * cfg.tokens) == (L, d, F, keys)
    assert bench.kernel_work(cfg, "attn", keys) == ("tensor", 4.0 * L * keys * d)   # QK^T and PV, 2 FLOP each
    assert bench.kernel_work(cfg, "attn", keys)[1] == pytest.approx(1.0319560704e13)
    assert bench.kernel_work(cfg, "qkv", keys) == ("tensor", 2.0 * L * 3 * d * d)
    assert bench.kernel_work(cfg, "oproj", keys) == ("tensor", 2.0 * L * d * d)
    assert bench.kernel_work(cfg, "ffn1", keys) == ("tensor", 2.0 * L * d * F)
    assert bench.kernel_work(cfg, "ffn2", keys) == ("tensor", 2.0 * L * d * F)
    x = L * d * 2                                                       # one bf16 activation
    assert bench.kernel_work(cfg, "gate", keys) == ("hbm", x)
    assert bench.kernel_work(cfg, "reuse", keys) == ("hbm", 3 * x)
    assert bench.kernel_work(cfg, "ln", keys) == ("hbm", 2 * x)
    assert bench.kernel_work(cfg, "embed", keys) == ("hbm", L * 16 * 4 + 16 * d * 4 + x)
    assert bench.kernel_work(cfg, "head", keys) == ("hbm", x + d * 16 * 4 + L * 16 * 4)
    # conditioning: the fp32 MLP weights (t_freq x d, A x d, 2 d^2, 6 d^2, 2 d^2) and the per-block tables
    B, tf, A = cfg.n_blocks, cfg.t_freq, cfg.action_dim
    w = 4 * (tf * d + A * d + 10 * d * d)
    assert bench.kernel_work(cfg, "cond", keys) == ("hbm", w + 8 * B * 6 * d)
    assert bench.kernel_work(cfg, "head", keys)[1] < bench.kernel_work(cfg, "reuse", keys)[1]
    assert bench.kernel_work(cfg, "euler", keys) == ("", 0.0)


def test_traffic_record_follows_the_source_hash(tmp_path, monkeypatch):
    src_dir = tmp_path / "paper_2604_20289_gb300" / "csrc"
    src_dir.mkdir(parents=True)
    (tmp_path / "profiles").mkdir()
    src = src_dir / "k_demo.cu"
    src.write_text("// kernel v1\n")
    sha = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    rec = {"bytes_per_launch": 123, "source": "k_demo.cu", "sha": sha}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps({"demo<1>": rec}))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.traffic_record("demo<1>")["bytes_per_launch"] == 123
    assert bench.traffic_record("other") is None
    src.write_text("// kernel v2\n")                                   # the kernel changed since the capture
    assert bench.traffic_record("demo<1>") is None


def test_oracle_cost_fit_recovers_fixed_and_per_row():
    fixed, per_row, L = 6.5, 0.0125, 12960
    samples = {32: [fixed + 32 * per_row] * 2, 256: [fixed + 256 * per_row - 1e-3, fixed + 256 * per_row + 1e-3]}
    f = bench.fit_block(samples, L)
    assert f["rows"] == [32, 256]
    assert f["per_row_s"] == pytest.approx(per_row)
    assert f["fixed_s"] == pytest.approx(fixed)
    assert f["block_s"] == pytest.approx(fixed + L * per_row)
    # a noisy sample that would give a negative slope is clamped: no negative costs
    g = bench.fit_block({32: [2.0], 256: [1.9]}, L)
    assert g["per_row_s"] == 0.0 and g["fixed_s"] == pytest.approx(2.0)


def _rec(kind, ps, block, ms, dec=xb.XC_DEC_COMPUTE):
    return {"kind": kind, "pass_seq": ps, "block": block, "ms": ms, "decision": dec}


def test_predicted_speedup_by_hand():
    # all-blocks arm: one chunk, one pass (t = 0), two blocks of 10 ms each
    recs_all = [_rec(k, 0, b, ms) for b in (0, 1) for k, ms in
                (("ln", 0.5), ("qkv", 2.0), ("attn", 4.0), ("oproj", 1.0), ("ln", 0.5), ("ffn1", 1.0), ("ffn2", 1.0))]
    # X-Cache arm: block 0 gated and computed, block 1 gated and skipped (gate 1 ms, reuse 0.5 ms),
    # a forced (KV-pass) gate that does not count
    recs = [_rec("gate", 0, 0, 1.0), _rec("gate", 0, 1, 1.0, xb.XC_DEC_SKIP),
            _rec("reuse", 0, 1, 0.5, xb.XC_DEC_SKIP), _rec("gate", 1, 0, 1.0, xb.XC_DEC_FORCED)]
    t_all = 20.0
    got = bench.predicted_speedup(recs, recs_all, t_all, [0, 1], [0], 1, 1)
    # saved = T_block(1) - gate - reuse = 10 - 1 - 0.5; gated = 1 + 1
    assert got == pytest.approx(t_all / (t_all - 8.5 + 2.0))


def test_kv_pass_schedule():
    cfg = bench.WORKLOADS["small"]
    assert all(bench.has_kv_pass(cfg.replace(kv_period=0), n) for n in range(6))
    assert [bench.has_kv_pass(cfg.replace(kv_period=3), n) for n in range(7)] == \
        [False, False, True, False, False, True, False]
