"""The multi-process path of bench.py on CPU: two gloo ranks (no GPU).

Under torchrun every rank runs its own replica of the workload (weak
scaling, no collective on the data path); the only collectives are the
barriers around the timed region and the max over ranks of the measured
time.  These tests run that host logic with the gloo backend: the job value
is world x the bytes of one replica over the slowest rank's time, every rank
agrees on it, and the reference arm runs on rank 0 alone.
"""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, results):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        bench.barrier(world)
        value, ms = bench.whole_job_value(10 ** 9, 10, 100.0 + 50.0 * rank, world)

        class Args:
            steps, warmup, gpus = 1, 0, world
        # the reference arm: ranks other than 0 return at once, doing nothing
        ran = None if rank == 0 else bench.run_reference(Args, world, rank)
        bench.barrier(world)
        results.put((rank, value, ms, ran))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_job_value():
    world = 2
    ctx = mp.get_context("spawn")
    results = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, results)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = sorted(results.get(timeout=10) for _ in range(world))
    # slowest rank: 150 ms; the job moved 2 x 10 x 1 GB in that time
    for rank, value, ms, ran in got:
        assert ms == pytest.approx(150.0)
        assert value == pytest.approx(2 * 10 * 1e9 / 0.150 / 1e9)
        assert ran is None
