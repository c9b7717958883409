"""The N > 1 path of bench.py on CPU: two gloo ranks, launched the way torchrun launches
bench.py (one process per GPU, rendezvous on 127.0.0.1).

Decode attention shards by sequence with no exchange step, so N GPUs run N independent
replicas (weak scaling): each rank draws its own seeded batch, the job's time is the
MAX over ranks of the timed region and the job's work the SUM of the ranks' units, and
the reference arm runs on rank 0 alone."""
import os
import socket
import sys

import numpy as np
import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        ms = [3.0, 5.0, 4.0, 1.0][rank]
        nbytes = [100.0, 250.0, 7.0, 1.0][rank]
        keys = [10.0, 20.0, 30.0, 40.0][rank]
        got = bench.across_ranks(dist, "cpu", ms, nbytes, keys)
        only_time = bench.across_ranks(dist, "cpu", ms)
        os.environ["RANK"], os.environ["WORLD_SIZE"] = str(rank), str(world)
        ref = None if rank == 0 else bench.run_reference(_Args())
        q.put((rank, got, only_time, ref))
        dist.barrier()
    finally:
        dist.destroy_process_group()


class _Args:
    workload, batch, steps, warmup = "tiny", 0, 1, 3


@pytest.mark.parametrize("world", [2])
def test_two_gloo_ranks_max_time_sum_work(world):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = {}
    for _ in range(world):
        rank, got, only_time, ref = q.get(timeout=300)
        res[rank] = (got, only_time, ref)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank in range(world):
        got, only_time, ref = res[rank]
        assert got == (5.0, 350.0, 30.0)          # max of 3 and 5 ms; 100 + 250 B; 10 + 20 keys
        assert only_time == (5.0,)
        if rank:
            assert ref is None                     # the reference arm: rank 0 alone


def test_single_process_needs_no_process_group():
    import bench
    assert bench.across_ranks(None, "cpu", 2.5, 7, 9) == (2.5, 7.0, 9.0)


def test_ranks_draw_distinct_batches_of_the_same_shape():
    import bench
    from paper_2607_06601_gb300 import workloads as wl
    spec = wl.SPECS["160m"]
    s0, s1 = bench.rank_spec(spec, 0), bench.rank_spec(spec, 1)
    assert s0 == spec                              # rank 0 runs the workload as defined
    b0, m0 = wl.policy(s0, 0, 0, 2048)
    b1, m1 = wl.policy(s1, 0, 0, 2048)
    assert b0.shape == b1.shape and m0.shape == m1.shape
    assert not np.array_equal(b0, b1) and not np.array_equal(m0, m1)
    # same mixes: the per-rank maps are draws from one distribution
    for b in (2, 4, 8, 16):
        assert abs(np.mean(b0 == b) - np.mean(b1 == b)) < 0.06
    assert (wl.contexts(s0) == wl.contexts(s1)).all()
