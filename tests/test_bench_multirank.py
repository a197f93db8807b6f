"""The N > 1 path of the benchmark on CPU: two gloo ranks get distinct sweep
batches and agree on the whole-job timing (slowest rank's time, all ranks'
units), with no collective on the data path."""
import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2605_30574_gb300.synth import workloads as WL


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    wl = WL.get("qwen3-8b-ladder")
    b = bench.rank_batch(wl.num_batches(), 0, rank)
    lo, hi = wl.batch_range(b)
    ms = 10.0 + 5.0 * rank                      # pretend rank 1 is slower
    units = (hi - lo) * 3
    q.put((rank, b, bench.reduce_timing(ms, units, dist, "cpu")))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_weak_scaling():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, b0, t0), (r1, b1, t1) = got
    assert (b0, b1) == (0, 1)
    assert t0 == t1 == (15.0, 512 * 3 * 2)


def test_rank_batch_wraps():
    assert [bench.rank_batch(7, 0, r) for r in range(9)] == [0, 1, 2, 3, 4, 5, 6, 0, 1]
    assert bench.rank_batch(7, 6, 1) == 0
    assert bench.reduce_timing(3.0, 5) == (3.0, 5)
