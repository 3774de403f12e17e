"""The N > 1 path of bench.py on CPU: two gloo ranks, each encoding its own
layer, report the whole-job value from the slowest rank's time (weak scaling,
no collective on the data path)."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    local_seconds = 1.0 + rank            # rank 1 is the slowest
    t = bench.max_over_ranks(local_seconds)
    q.put((rank, t, bench.rank_layer(rank), bench.job_value(1000, world, 5, t)))
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_report_the_slowest_time_and_whole_job_value():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [2.0, 2.0]          # both see the max
    assert [r[2] for r in res] == [0, 1]              # distinct layers per rank
    assert res[0][3] == pytest.approx(2 * 1000 * 5 / 2.0)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    class A:  # noqa: D401 - minimal args
        steps, warmup = 1, 0
    assert bench.run_reference(A()) is None          # rank 1 returns without work
