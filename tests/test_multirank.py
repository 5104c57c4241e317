"""The multi-rank path of bench.py on CPU (gloo, world size 2): each rank
runs an independent replica of the layer (no data-path collective), and the
timing is the slowest rank's, so the whole-job rate is world x units x steps
over that time.  Rendezvous on 127.0.0.1."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as tmp  # noqa: E402

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier()
        # rank r took (r + 1) seconds for its 10 steps of 3 units
        slowest = bench.max_over_ranks(float(rank + 1), device="cpu")
        rate = bench.whole_job_rate(3, 10, world, slowest)
        bench.barrier()
        q.put((rank, slowest, rate))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time():
    world = 2
    ctx = tmp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [2.0, 2.0]
    assert [r[2] for r in res] == [30.0, 30.0]


def test_single_process_helpers_need_no_group():
    assert bench.max_over_ranks(1.5, device="cpu") == 1.5
    bench.barrier()
    assert bench.whole_job_rate(4, 5, 1, 2.0) == 10.0
