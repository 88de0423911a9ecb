"""The N > 1 path of bench.py on CPU: independent replicas, gloo, world size 2.

Each rank owns its own pool (here: its own oracle run on a rank-specific seed);
ranks exchange nothing but their timings, and the whole-job value is all ranks'
bytes over the slowest rank's time."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    from oracle import OracleManager
    from workloads import make_workload
    wl = make_workload("thinker", 10 + rank, n_turns=3)
    om = OracleManager(wl, with_bytes=False, rank_on="none")
    om.run()
    moved = om.pool.bytes_out + om.pool.bytes_in
    seconds = 1.0 + rank                      # a stand-in per-rank duration
    t = torch.tensor([seconds, float(moved)], dtype=torch.float64)
    gathered = [torch.zeros_like(t) for _ in range(world)]
    dist.barrier()
    dist.all_gather(gathered, t)
    g = torch.stack(gathered).numpy()
    val = bench.aggregate(g[:, 1], g[:, 0])
    out[rank] = (val, moved, float(g[:, 1].sum()))
    dist.destroy_process_group()


def test_two_replicas_aggregate_over_gloo():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    (v0, m0, tot0), (v1, m1, tot1) = out[0], out[1]
    assert v0 == v1 == pytest.approx((m0 + m1) / 2.0)   # slowest rank took 2 s
    assert tot0 == tot1 == m0 + m1 and m0 != m1          # different seeds, different work


def test_aggregate_single_rank():
    import bench
    assert bench.aggregate([10.0], [2.0]) == 5.0
    assert bench.aggregate([10.0, 30.0], [2.0, 4.0]) == 10.0
