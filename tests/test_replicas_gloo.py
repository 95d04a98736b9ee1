"""The multi-process path of bench.py on CPU (world_size 2, gloo): replicas
with no data-path collective, a barrier around the timed region, the job time
as the max over ranks, whole-job throughput, and the reference arm running on
rank 0 only."""
import contextlib
import io
import os
import socket

import pytest
import torch
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(world),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import bench
    import torch.distributed as dist
    r, local, w = bench.dist_setup(world, backend="gloo")
    assert (r, local, w) == (rank, rank, world)
    bench.barrier(w, cuda=False)
    ms = 10.0 + 5.0 * rank                       # rank 1 is the slowest
    m = bench.reduce_max(ms, w, device="cpu")
    out[rank] = (m, bench.job_throughput(1000, w, m))
    dist.destroy_process_group()


def test_two_ranks_max_time_and_job_throughput():
    world, port = 2, _free_port()
    out = mp.get_context("spawn").Manager().dict()  # no fork of a threaded process
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for rank in range(world):
        m, v = out[rank]
        assert m == 15.0                          # max over ranks, seen by every rank
        assert v == pytest.approx(2 * 1000 / 0.015)


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        bench.run_reference(type("A", (), {"warmup": 3, "steps": 1})())
    assert buf.getvalue() == ""


def test_world_mismatch_is_rejected(monkeypatch):
    import bench
    monkeypatch.setenv("WORLD_SIZE", "1")
    with pytest.raises(SystemExit):
        bench.dist_setup(2, backend="gloo")
