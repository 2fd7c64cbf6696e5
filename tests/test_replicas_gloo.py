"""The multi-GPU form of the benchmark is replicas only: each rank runs the
whole stack on its own GPU and the ranks meet only to time.  This checks its
host side with two gloo ranks on the CPU: the rendezvous from the torchrun
environment, the barrier, the max over ranks of the timed region, the
whole-job rate built from it, and that only rank 0 runs the reference arm."""
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


def _rank_main(rank, world, port, out):
    os.environ.update(RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE=str(world), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    import bench

    class Args:
        pass

    ws, r, local = bench.dist_setup(Args())
    assert (ws, r, local) == (world, rank, rank)
    assert dist.get_backend() == "gloo"
    bench.barrier(ws)
    ms = 10.0 + 5.0 * rank  # a rank's timed region
    t = bench.max_over_ranks(ms, ws)
    m, steps = 3, 7
    value = ws * m * steps / (t / 1e3)  # tokens/s of the whole job, as run_gpu reports it
    # the reference arm: rank 0 alone runs; the others return at once
    args = Args()
    args.steps, args.warmup, args.config, args.m, args.layers = 1, 0, "small_d256_i768", 1, 1
    ran = None
    if rank != 0:
        bench.run_reference(args)  # returns before any work
        ran = False
    out.put((rank, t, value, ran))
    bench.barrier(ws)
    dist.destroy_process_group()


def test_two_gloo_replicas():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    res = sorted(q.get(timeout=10) for _ in range(world))
    for rank, t, value, ran in res:
        assert t == pytest.approx(15.0)  # the slowest rank sets the time
        assert value == pytest.approx(world * 3 * 7 / 0.015)
        assert ran in (None, False) and (ran is False) == (rank != 0)
