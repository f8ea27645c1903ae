"""The N > 1 path of bench.py on CPU: two gloo ranks. Each GPU runs its own replica of the
step (no data-path collective), so the only cross-rank step is the timing reduction: the job
time is the slowest rank's and the value counts every rank's bytes. Under torchrun the
reference arm runs on rank 0 only."""
import contextlib
import io
import os
import socket

import pytest
import torch.multiprocessing as tmp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, times, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        assert bench.dist_env() == (world, rank, rank)
        q.put((rank,) + bench.whole_job(times[rank], world, 1_000_000, 10))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_count_both_replicas():
    world, times = 2, [10.0, 25.0]
    ctx = tmp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, times, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(world))
    for rank, ms, gbs in got:
        assert ms == 25.0                                   # max over ranks
        assert gbs == pytest.approx(2 * 1e6 * 10 / 0.025 / 1e9)   # both replicas' bytes


def test_single_rank_needs_no_process_group():
    assert bench.whole_job(8.0, 1, 2_000_000, 4) == (8.0, pytest.approx(4 * 2e6 / 0.008 / 1e9))


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    class A:
        steps, warmup, gpus = 1, 0, 2
    out = io.StringIO()
    with contextlib.redirect_stdout(out):
        assert bench.reference_arm(A()) is None
    assert out.getvalue() == ""

