"""The N > 1 path of bench.py on the CPU: world-size-2 gloo ranks (one process
each) run the timing aggregation every rank of a `--gpus 2` job runs, and the
reference arm's non-zero ranks leave without work.  The path has no data
collective (replicas only); the one all-reduce is the max over ranks."""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, ms_by_rank, out):
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    ms, value = bench.job_rate(ms_by_rank[rank], 1000, 4, world, "cpu")
    dist.barrier()
    dist.destroy_process_group()
    out.put((rank, ms, value))


def test_job_rate_takes_the_slowest_rank():
    world, port = 2, _free_port()
    ms_by_rank = [120.0, 150.0]
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, ms_by_rank, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    res = sorted(out.get(timeout=10) for _ in range(world))
    for _, ms, value in res:
        assert ms == 150.0
        assert value == pytest.approx(1000 * world * 4 / 0.150)


def test_reference_arm_other_ranks_do_nothing(capsys, monkeypatch):
    sys.path.insert(0, ROOT)
    import bench

    monkeypatch.setenv("RANK", "1")

    class Args:
        steps, warmup, gpus = 1, 3, 2

    spec = bench.wl.config(bench.CONFIG_ID)
    bench.run_reference(Args, spec, bench.wl.lengths(spec))
    assert capsys.readouterr().out == ""
