"""The replica (N > 1) path of bench.py on CPU: world-size-2 gloo ranks.

The hot path has no exchange step, so N GPUs run N independent replicas; the
only cross-rank logic is the max-over-ranks timing and the whole-job
throughput, checked here without a GPU."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    local = [3.5, 7.25][rank]
    slowest = bench.max_over_ranks(local)
    q.put((rank, slowest, bench.job_throughput(100.0, world, slowest)))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_throughput_gloo():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank, slowest, thr in out:
        assert slowest == 7.25                      # every rank sees the slowest rank's time
        assert thr == pytest.approx(2 * 100.0 / 7.25)  # replicas: units of all ranks / max time


def test_single_process_passthrough():
    import bench
    assert bench.max_over_ranks(1.25) == 1.25
    assert bench.job_throughput(10.0, 1, 2.0) == 5.0


def test_reference_arm_other_ranks_exit_without_work(monkeypatch):
    import bench

    class A:
        workload = "tiny-f32"
        steps = 1
        warmup = 3
        batch = 0
    assert bench.run_reference(A(), rank=1, world=2) == 0   # returns at once: no data, no pool
