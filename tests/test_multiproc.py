"""The N > 1 path of bench.py on CPU with gloo, world size 2 (no GPU): every rank gets its own
seeded instance of the workload, the data path has no collective, and only the timing is
reduced (max of the time, sum of the work over ranks)."""
import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
import workloads as W


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        w = W.tiny(seed=bench.rank_seed(1, rank), nloc=9, nreal=5 + rank, sel=12)
        total, evals = bench.reduce_over_ranks(1.5 + rank, float(w.evals), world, torch.device("cpu"))
        sums = [None] * world
        dist.all_gather_object(sums, float(np.abs(w.Rt).sum()))

        class A:
            workload, pad, seed, dtype, steps, warmup = "tiny", 0.3, 1, "f64", 2, 3

        ref = bench.run_reference(A, rank, world) if rank == 1 else "skipped"

        class S:
            workload, seed, scaling = "tiny", 1, "strong"

        part = bench.rank_workload(S, rank, world)
        _, strong_evals = bench.reduce_over_ranks(0.0, float(part.evals), world, torch.device("cpu"))
        q.put((rank, total, evals, float(w.evals), sums, ref, strong_evals, part.nloc))
    finally:
        dist.destroy_process_group()


def test_two_ranks_gloo():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = {}
    for _ in range(world):
        r = q.get(timeout=120)
        out[r[0]] = r
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    ev = [out[r][3] for r in range(world)]
    for r in range(world):
        _, total, evals, _, sums = out[r][:5]
        assert total == 2.5  # max over ranks
        assert evals == sum(ev)  # work of all ranks
        assert sums[0] != sums[1]  # independent seeded instances
    assert out[1][5] is None  # the reference arm runs on rank 0 only
    full = W.tiny(seed=1)
    assert out[0][6] == out[1][6] == float(full.evals)  # strong scaling: the shards cover the instance
    assert out[0][7] + out[1][7] == full.nloc
