"""More chunk-step parity against the CPU oracle through xc_chunk_step:
rollouts whose decisions the deviation metric (Eq. 6-7) takes part in,
the every-evaluation fingerprint refresh and the 1-D fallback sample on a
bf16 model, the device decision-replay table, and a benchmark-size block
after the KV ring has filled and wrapped.

Tolerances as in test_gpu_chunk_step: bf16 per-block rel-L2 <= 1e-2, final
latent <= 3e-2, decisions identical except within 1e-3 relative of a
threshold; full-size sampled rows <= 1e-2 per row and 5e-3 together."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu

import oracle as O  # noqa: E402
import xc_inputs as X  # noqa: E402

if not torch.cuda.is_available():
    pytest.skip("needs a CUDA GPU", allow_module_level=True)

from paper_2604_20289_gb300 import xcache as xb  # noqa: E402
from paper_2604_20289_gb300.rollout import rollout as gpu_rollout  # noqa: E402
from test_gpu_chunk_step import (compare_decisions, decisions, model, params, rel_l2,  # noqa: E402
                                 replay_of)


def _per_block_parity(cfg, op, gp, ref):
    w, xc = model(cfg)
    traj = X.Trajectory(cfg)
    rep = gpu_rollout(xc, traj, cfg.n_chunks, gp, replay=replay_of(ref["stats"]), keep_trace=True)
    np.testing.assert_array_equal(decisions(rep["stats"]), decisions(ref["stats"]))
    for n in range(cfg.n_chunks):
        for t in range(cfg.n_steps):
            for b in range(cfg.n_blocks):
                e = rel_l2(rep["trace"][n][t][b], ref["trace"][n][t][b])
                assert e <= 1e-2, (n, t, b, e)
        assert rel_l2(rep["final"][n], ref["final"][n]) <= 3e-2
    xc.reset()
    free = gpu_rollout(xc, traj, cfg.n_chunks, gp)
    compare_decisions(ref["stats"], free["stats"], op)


def _deviation_decided(stats, p):
    """Evaluated decisions where the cosine passed its threshold and the
    deviation test alone decided (s >= tau, d_max >= tau_dev)."""
    n = 0
    for ch in stats:
        for st in ch:
            for b in range(len(st["decision"])):
                if st["decision"][b] == O.Decision.COMPUTE and st["s_cos"][b] >= st["tau"][b] \
                        and st["d_max"][b] >= p.tau_dev:
                    n += 1
    return n


@pytest.mark.parametrize("cfg,tau_dev", [(X.MID_HD64, 2.0), (X.GROUPS_BF16, 2.2)],
                         ids=["mid_bf16", "view_groups_bf16"])
def test_deviation_metric_decides_rollout(cfg, tau_dev):
    """tau_dev inside the range of the d_max values of these rollouts, so
    that Eq. 6's deviation decides some decisions (not just the cosine)."""
    op, gp = params(tau_floor=0.92, tau_dev=tau_dev)
    w, _ = model(cfg)
    ref = O.rollout(cfg, w, X.Trajectory(cfg), op, cfg.n_chunks, keep_trace=True)
    assert _deviation_decided(ref["stats"], op) >= 1
    assert (decisions(ref["stats"]) == O.Decision.SKIP).any()
    _per_block_parity(cfg, op, gp, ref)


@pytest.mark.parametrize("kw", [dict(fp_refresh=1), dict(fp_linear=True), dict(fp_refresh=1, fp_tokens=20)],
                         ids=["refresh_every_eval", "linear_sample", "refresh_k20"])
def test_fingerprint_options_bf16_rollout(kw):
    cfg = X.MID_HD64
    op, gp = params(tau_floor=0.92, tau_dev=2.6, **kw)
    w, _ = model(cfg)
    ref = O.rollout(cfg, w, X.Trajectory(cfg), op, cfg.n_chunks, keep_trace=True)
    assert (decisions(ref["stats"]) == O.Decision.SKIP).any()
    _per_block_parity(cfg, op, gp, ref)


def test_device_replay_table_equals_host_replay():
    """Decision replay from a device [S][B] table gives the decisions and
    outputs of the host per-pass replay (the oracle's decisions)."""
    cfg = X.MID_HD64
    op, gp = params(tau_floor=0.92, tau_dev=10.0)
    w, xc = model(cfg)
    traj = X.Trajectory(cfg)
    ref = O.rollout(cfg, w, traj, op, cfg.n_chunks)
    rp = replay_of(ref["stats"])
    host = gpu_rollout(xc, traj, cfg.n_chunks, gp, replay=rp)
    xc.reset()
    S = cfg.n_steps
    finals, stats = [], []
    x = torch.empty(cfg.tokens, cfg.c_latent, device="cuda")
    v = torch.empty_like(x)
    for n in range(cfg.n_chunks):
        table = torch.tensor(np.array(rp[n], np.uint8), device="cuda")          # [S][B]
        g = xb.gate_params(tau_floor=float(np.float32(0.92)), tau_dev=10.0, replay_table=table)
        x.copy_(torch.from_numpy(traj.noise(n)))
        st_n = []
        for t in range(S):
            st_n.append(xc.chunk_step(x, traj.action(n), O.SIGMAS[t], t, False, g, v_out=v))
            xc.euler(x, v, O.SIGMAS[t + 1] - O.SIGMAS[t])
        xc.chunk_step(torch.from_numpy(traj.clean(n)).cuda(), traj.action(n), 0.0, S, True, g)
        torch.cuda.synchronize()
        del table
        finals.append(x.cpu().numpy())
        stats.append(st_n)
    np.testing.assert_array_equal(decisions(stats), decisions([ch[:S] for ch in host["stats"]]))
    for a, b in zip(finals, host["final"]):
        np.testing.assert_array_equal(a, b)


@pytest.mark.parametrize("cfg", [X.SMALL_BF16, X.DIT_14B.replace(name="dit14b_shape_2blk", n_blocks=2)],
                         ids=["small_bf16", "dit14b_block_shape"])
def test_full_ring_wrapped_block_sampled_rows(cfg):
    """After W_kv full chunks the ring is full and the next chunk's K/V go to
    slot 0 again (slot arithmetic, FIFO eviction).  Block 0 of pass 0 of that
    chunk, on sampled token rows, against the oracle, whose ring holds block
    0's clean K/V of the last W_kv - 1 chunks -- each computed by the oracle
    from that chunk's clean latent at sigma = 0 (block 0's keys and values
    depend on its own input only).  Benchmark launch configuration: split
    attention over a full ring, persistent GEMMs, CUDA-graph replay."""
    w, xc = model(cfg)
    N, W, S = cfg.kv_window, cfg.kv_window, cfg.n_steps
    traj = X.Trajectory(cfg, n_chunks=N + 1)
    L, d = cfg.tokens, cfg.d_model
    _, g = params(tau_floor=2.0)                                  # every gated block recomputes
    x = torch.empty(L, cfg.c_latent, device="cuda")
    v = torch.empty_like(x)
    for n in range(N):
        x.copy_(torch.from_numpy(traj.noise(n)))
        for t in range(S):
            xc.chunk_step(x, traj.action(n), O.SIGMAS[t], t, False, g, v_out=v, want_stats=False)
            xc.euler(x, v, O.SIGMAS[t + 1] - O.SIGMAS[t])
        xc.chunk_step(torch.from_numpy(traj.clean(n)).cuda(), traj.action(n), 0.0, S, True, g, want_stats=False)
    tr = torch.empty(cfg.n_blocks, L, d, device="cuda", dtype=torch.bfloat16)
    xc.set_trace(tr)
    try:
        x.copy_(torch.from_numpy(traj.noise(N)))
        xc.chunk_step(x, traj.action(N), 1.0, 0, False, g, v_out=v, want_stats=False)
        xc.sync()
    finally:
        xc.set_trace(None)
    got = tr[0].float().cpu().numpy()
    del tr
    M = O.OracleModel(cfg, w)
    ring_k, ring_v = [], []
    for n in range(N - W + 1, N):                                 # resident: the last W - 1 KV-update chunks
        mods, _ = M.cond(0.0, traj.action(n))
        pos = O.group_token_positions(cfg.groups, cfg.frames, n)
        _, k, vv = M.block(0, M.patch_embed(traj.clean(n)), mods[0], [], [], pos, rows=np.array([0]))
        ring_k.append(k)
        ring_v.append(vv)
    mods, _ = M.cond(1.0, traj.action(N))
    pos = O.group_token_positions(cfg.groups, cfg.frames, N)
    rows = np.unique(np.r_[0, 1, 127, 128, 255, 256, L // 2, L - 129, L - 128, L - 1,
                           np.random.default_rng(9).choice(L, 22, replace=False)])
    want, _, _ = M.block(0, M.patch_embed(traj.noise(N)), mods[0], ring_k, ring_v, pos, rows=rows)
    for i, r in enumerate(rows):
        assert rel_l2(got[r], want[i]) <= 1e-2, (r, rel_l2(got[r], want[i]))
    assert rel_l2(got[rows], want) <= 5e-3
    xc.close()
    _MODELS_drop(cfg)


def _MODELS_drop(cfg):
    import test_gpu_chunk_step as T
    T._MODELS.pop(cfg.name, None)


# ----------------------------------------- lazy residual chaining (reading c27)
@pytest.mark.parametrize("cfg,kw", [
    (X.TINY_F32.replace(name="chain_tiny_f32_4blk", n_blocks=4), dict(tau_floor=0.5, margin=1.0, tau_dev=100.0,
                                                                       front_anchors=0, back_anchors=1)),
    (X.MID_HD64.replace(name="chain_mid_bf16_5blk", n_blocks=5), dict(tau_floor=0.9, tau_dev=3.0, back_anchors=1)),
    (X.GROUPS_BF16.replace(name="chain_groups_bf16_4blk", n_blocks=4), dict(tau_floor=0.9, tau_dev=3.0,
                                                                            back_anchors=1))],
    ids=["tiny_f32", "mid_bf16", "view_groups_bf16"])
def test_chained_rollout_parity(cfg, kw):
    """Runs of skipped blocks are chained (no per-block reuse writes; the
    next gate's fingerprint from the sampled rows and the residual means;
    the input written before the next computed block or the head) and
    compared with the oracle's chained mode: numerics in decision-replay
    mode (fp32: max |err| <= 1e-4 RMS; bf16: final latent rel-L2 <= 3e-2),
    decisions free-running."""
    op, gp = params(chain=True, **kw)
    w, xc = model(cfg)
    traj = X.Trajectory(cfg)
    ref = O.rollout(cfg, w, traj, op, cfg.n_chunks)
    dec = decisions(ref["stats"])
    # at least one run of two or more skipped blocks followed by a computed block or the head
    assert any((dec[n, t, b] == O.Decision.SKIP and dec[n, t, b + 1] == O.Decision.SKIP)
               for n in range(dec.shape[0]) for t in range(cfg.n_steps) for b in range(cfg.n_blocks - 1))
    rep = gpu_rollout(xc, traj, cfg.n_chunks, gp, replay=replay_of(ref["stats"]))
    np.testing.assert_array_equal(decisions(rep["stats"]), dec)
    for n in range(cfg.n_chunks):
        want, got = ref["final"][n], rep["final"][n]
        if cfg.dtype == "f32":
            rms = np.sqrt(np.mean(want ** 2))
            assert np.max(np.abs(got - want)) <= 1e-4 * rms, (n, np.max(np.abs(got - want)) / rms)
        else:
            assert rel_l2(got, want) <= 3e-2, (n, rel_l2(got, want))
    xc.reset()
    free = gpu_rollout(xc, traj, cfg.n_chunks, gp)
    compare_decisions(ref["stats"], free["stats"], op)
    xc.close()
    _MODELS_drop(cfg)


def test_chained_small_model_matches_per_block_reuse_decisions():
    """Benchmark-size model: chaining changes only roundings, so the metrics
    of the chained rollout stay close to those of per-block reuse on the same
    decisions (replayed from the per-block run), and its outputs stay close."""
    cfg = X.SMALL_BF16
    w, xc = model(cfg)
    traj = X.Trajectory(cfg, n_chunks=4)
    _, gp = params(tau_floor=0.9, tau_dev=3.0)
    plain = gpu_rollout(xc, traj, 4, gp)
    rp = replay_of(plain["stats"])
    assert sum(int(s) for ch in rp for t in ch for s in t) >= 10
    xc.reset()
    _, gc = params(tau_floor=0.9, tau_dev=3.0, chain=True)
    ch = gpu_rollout(xc, traj, 4, gc, replay=rp)
    for a, b in zip(plain["final"], ch["final"]):
        assert rel_l2(b, a) <= 1e-2
    for ca, cb in zip(plain["stats"], ch["stats"]):
        for sa, sb in zip(ca, cb):
            ok = ~np.isnan(sa["s_cos"])
            np.testing.assert_allclose(sb["s_cos"][ok], sa["s_cos"][ok], rtol=0, atol=5e-3)


def test_all_method_options_together_bf16():
    """View groups (front / side / rear cameras), cross-attention to a
    varying number of condition tokens, a KV-update pass every second chunk
    (force-compute chunks) and lazy chaining, on one bf16 model: decisions
    and final latents against the oracle (decision replay) and free-running
    decisions."""
    cfg = X.GROUPS_BF16.replace(name="all_options_bf16_4blk", n_blocks=4, d_ctx=128, max_ctx=64, kv_period=2,
                                n_chunks=5)
    op, gp = params(tau_floor=0.9, tau_dev=3.0, back_anchors=1, chain=True)
    w, xc = model(cfg)
    traj = X.Trajectory(cfg, n_chunks=cfg.n_chunks)
    ref = O.rollout(cfg, w, traj, op, cfg.n_chunks)
    dec = decisions([ch[:cfg.n_steps] for ch in ref["stats"]])
    assert (dec == O.Decision.SKIP).any()
    rep = gpu_rollout(xc, traj, cfg.n_chunks, gp, replay=replay_of(ref["stats"]))
    np.testing.assert_array_equal(decisions([ch[:cfg.n_steps] for ch in rep["stats"]]), dec)
    for n in range(cfg.n_chunks):
        assert rel_l2(rep["final"][n], ref["final"][n]) <= 3e-2, (n, rel_l2(rep["final"][n], ref["final"][n]))
    xc.reset()
    free = gpu_rollout(xc, traj, cfg.n_chunks, gp)
    compare_decisions(ref["stats"], free["stats"], op)
    xc.close()
    _MODELS_drop(cfg)
