"""The N > 1 replica path of bench.py on CPU (gloo, world size 2): timing is
the maximum over ranks, the barrier passes, the whole-job value counts every
replica's steps, and the reference arm runs on rank 0 only."""

import io
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        t_ms = 10.0 + 5.0 * rank                       # rank 1 is the slower replica
        mx = bench.max_over_ranks(t_ms, world)
        q.put((rank, mx, bench.job_value(mx, world)))
        bench.barrier(world)
    finally:
        dist.destroy_process_group()


def test_two_ranks_max_and_job_value():
    torch = pytest.importorskip("torch")
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    for rank, mx, val in res:
        assert mx == 15.0                              # every rank sees the slowest rank's time
        assert val == pytest.approx(2 * 1000.0 / 15.0)  # both replicas' steps over the slowest time


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("LOCAL_RANK", "1")
    args = bench.parse_args(["--impl", "reference", "--gpus", "2", "--steps", "2", "--warmup", "3"])
    out = io.StringIO()
    with redirect_stdout(out):
        bench.run_reference(args)
    assert out.getvalue() == ""
