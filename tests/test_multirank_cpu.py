"""The multi-process path of bench.py on CPU ranks (gloo, world size 2).

The Gauss sum does not exchange data between GPUs: `bench.py --gpus N`
runs N replicas, one per rank, and reports the whole-job rate from the
slowest rank.  These tests run that host logic on two gloo ranks."""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, step_ms, queue):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    slowest = bench.reduce_max(step_ms[rank], "cpu")
    value = bench.replica_value(world, 1000, slowest)
    dist.barrier()
    dist.destroy_process_group()
    queue.put((rank, slowest, value))


def test_two_gloo_ranks_take_the_slowest_step():
    pytest.importorskip("torch")
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    port = _free_port()
    step_ms = [2.0, 5.0]
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, step_ms, queue)) for r in range(2)]
    for p in procs:
        p.start()
    results = sorted(queue.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # Both ranks see the slowest rank's time; the rate counts both replicas.
    assert [r[1] for r in results] == [5.0, 5.0]
    assert results[0][2] == pytest.approx(2 * 1000 / 5e-3)


def test_single_process_needs_no_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(3.25, "cpu") == 3.25
    assert bench.replica_value(1, 4096, 2.0) == pytest.approx(4096 / 2e-3)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    assert bench.main(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "0"]) == 0
    assert capsys.readouterr().out == ""
