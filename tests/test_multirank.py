"""Multi-rank plumbing of bench.py on CPU with gloo (world_size 2): the job
time is the slowest rank's, throughput counts every rank's shard, ranks draw
disjoint shards, and a rank that fails is seen by the others as an error."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from paper_2310_07177_gb300 import workloads as W
    local = [12.5, 30.0][rank]
    t = bench.job_time_ms(local)
    spec = W.VerifySpec(4, 2, 64, torch.float32, 2.0, 1.0, 1.0, 1.0)
    inp = W.verify_inputs(spec, seed=bench.shard_seed(W.seed_for(2), rank))
    gathered = [torch.zeros_like(inp["draft"]) for _ in range(world)]
    dist.all_gather(gathered, inp["draft"])
    out[rank] = (t, bench.job_throughput(100, world, t), bool(torch.equal(gathered[0], gathered[1])))
    dist.barrier()
    dist.destroy_process_group()


def test_job_time_is_max_over_ranks_and_shards_differ():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        t, thr, same = res[rank]
        assert t == 30.0                    # slowest rank
        assert thr == pytest.approx(2 * 100 / 0.030)
        assert not same                     # disjoint shards


def _failing_worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    from datetime import timedelta
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=timedelta(seconds=5))
    if rank == 1:
        dist.destroy_process_group()
        raise SystemExit(3)  # leaves between steps, before the timing reduction
    import bench
    try:
        bench.job_time_ms(1.0)
        out[rank] = "no error"
    except Exception as e:  # the surviving rank learns of it through the collective
        out[rank] = type(e).__name__


def test_a_rank_that_leaves_is_reported_to_the_others():
    world = 2
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        procs = [ctx.Process(target=_failing_worker, args=(r, world, port, out)) for r in range(world)]
        for p in procs:
            p.start()
        for p in procs:
            p.join(timeout=120)
            if p.is_alive():
                p.kill()
        assert procs[1].exitcode == 3
        assert out.get(0) not in (None, "no error")
