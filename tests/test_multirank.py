"""The N > 1 path of bench.py on CPU: two gloo ranks (127.0.0.1), as torchrun
would start them.  The path has no exchange between GPUs (replicas only), so
what is checked is the host-side job logic: the slowest rank's time decides,
the job's value counts every rank's samples, and the reference arm runs on
rank 0 alone."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = [3.0, 5.0][rank]
    slow = bench.slowest_rank(ms)
    value = bench.job_throughput(1000, world, slow / 1e3)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, slow, value))


def test_two_gloo_ranks_take_the_slowest_time():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = free_port()
    procs = [ctx.Process(target=worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, slow, value in res:
        assert slow == 5.0
        assert value == pytest.approx(2 * 1000 / 5e-3)


def test_single_process_has_no_reduction():
    import bench
    assert bench.slowest_rank(7.5) == 7.5
    assert bench.job_throughput(1024, 1, 0.5) == 2048


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    bench.run_reference(bench.parse(["--impl", "reference", "--gpus", "2"]))
    assert capsys.readouterr().out == ""
