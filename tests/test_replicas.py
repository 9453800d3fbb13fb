"""The multi-rank host logic of bench.py, as world size 2 on CPU (gloo).

Layers are independent problems, so the N-GPU run is N replicas with no data-path
collective: every rank quantizes its own layer (seed + rank), the step time is the
slowest rank's, and the job's throughput is the units of all ranks over that time.
"""
import os
import socket

import torch
import torch.multiprocessing as mp

import bench
from paper_2309_01885_gb300 import inputs


def _free_port() -> int:
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ms = bench.max_over_ranks(10.0 + 5.0 * rank, "cpu")          # rank 1 is the slow one
        value = bench.job_throughput(1000.0, world, ms)
        W = inputs.layer_weights(8, 16, dtype=torch.float32, seed=5 + rank, device="cpu")
        got = [torch.empty_like(W) for _ in range(world)]
        dist.all_gather(got, W)
        out.put((rank, ms, value, bool(torch.equal(got[0], got[1]))))
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_slowest_time_and_count_every_rank():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for pr in procs:
        pr.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for pr in procs:
        pr.join(timeout=60)
        assert pr.exitcode == 0
    for rank, ms, value, same in res:
        assert ms == 15.0                          # both ranks report the slowest rank's time
        assert value == 2 * 1000.0 / 0.015         # units of both ranks over that time
        assert not same                            # each rank owns a different layer


def test_one_rank_is_unchanged():
    assert bench.max_over_ranks(12.5, "cpu") == 12.5
    assert bench.job_throughput(3.0, 1, 1000.0) == 3.0
