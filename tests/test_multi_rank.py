"""The N > 1 host path of bench.py on CPU: two gloo ranks.

bench.py runs one replica per GPU (the path shards by sequence with no
exchange step): each rank times its own batch (seed + rank), the job's step
time is the slowest rank's (an all-reduce MAX), and the job's throughput
counts every rank's tokens. The reference arm runs on rank 0 only.
"""
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


def _worker(rank, ws, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=ws, init_method=f"tcp://127.0.0.1:{port}")
    try:
        import bench
        ms = bench.max_over_ranks(1.5 + rank, ws, "cpu")  # rank 1 is the slower replica
        q.put((rank, ms, bench.job_throughput(ws, 2176, ms)))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_step_time_is_the_slowest_rank_and_value_counts_all_ranks():
    pytest.importorskip("torch")
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
    assert [r[1] for r in res] == [2.5, 2.5]
    assert all(abs(r[2] - 2 * 2176 / 2.5e-3) < 1e-6 for r in res)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(3.0, 1, "cpu") == 3.0
    assert bench.job_throughput(1, 64, 2.0) == 64 / 2e-3


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    assert bench.main(["--impl", "reference", "--gpus", "2", "--steps", "1", "--warmup", "3"]) == 0
    assert capsys.readouterr().out == ""  # no line, no oracle run on rank 1
