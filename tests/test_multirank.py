"""The N > 1 benchmark path on CPU: replicas (one rollout per GPU, no
data-path collective) joined by one max-over-ranks all-reduce of the timed
region; world size 2 over gloo on 127.0.0.1."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    r, w, local = bench.dist_env()
    dist.init_process_group("gloo", rank=r, world_size=w)
    try:
        # each replica times its own steps; the job's time is the slowest one
        local_ms = 100.0 + 50.0 * rank
        ms = bench.max_over_ranks(local_ms, w)
        rate = bench.whole_job_rate(8, w, ms * 1e-3)
        dist.barrier()
        out.put((r, w, local, ms, rate))
    finally:
        dist.destroy_process_group()


def test_two_replicas_take_the_slowest_time():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    out = ctx.SimpleQueue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(out.get() for _ in range(world))
    for r, (rank, w, local, ms, rate) in enumerate(got):
        assert (rank, w, local) == (r, world, r)
        assert ms == 150.0                       # max over the ranks' 100 and 150 ms
        assert rate == pytest.approx(2 * 8 / 0.150)


def test_single_rank_is_unreduced():
    import bench
    assert bench.max_over_ranks(123.5, 1) == 123.5
    assert bench.whole_job_rate(8, 1, 0.5) == 16.0
