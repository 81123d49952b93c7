"""The multi-rank timing path of bench.py on CPU: two gloo ranks take the max
of their step times over ranks and report whole-job values, as the benchmark
does under torchrun with one replica per GPU (the cohort step does not shard:
one global decision per step)."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w, r, l = bench.dist_env()
        assert (w, r, l) == (world, rank, rank)
        step_ms = 2.0 + rank  # the slower rank sets the job's time
        mx = bench.max_over_ranks(step_ms)
        out[rank] = (mx, bench.whole_job_us_per_invocation(mx, world, 1000))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_max_and_report_whole_job_values():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
    assert out[0] == out[1]
    mx, us = out[0]
    assert mx == 3.0
    # 2 ranks x 1,000 invocations in 3 ms: 1.5 us per invocation for the job
    assert us == pytest.approx(1.5)


def test_single_process_needs_no_group():
    import bench
    assert bench.max_over_ranks(4.25) == 4.25
    assert bench.whole_job_us_per_invocation(2.0, 1, 1000) == pytest.approx(2.0)
