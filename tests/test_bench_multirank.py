"""bench.py's multi-rank host logic on CPU with gloo, world size 2: each rank
draws its own batch (weak scaling, no data exchange), the step time is the max
over ranks and the byte count the sum over ranks."""
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


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    from paper_2609_36899_gb300.workloads import MIXED, draw_lengths
    import numpy as np

    w, r, _ = bench.dist_setup(None)
    assert (w, r) == (world, rank)
    t = bench.max_over_ranks(1.0 + rank, w)
    s = bench.sum_over_ranks(10.0 * (rank + 1), w)
    rng = np.random.Generator(np.random.PCG64(MIXED.seed + r))
    lens = draw_lengths(MIXED.lengths, MIXED.length_args, 8, rng)
    bench.barrier(w)
    q.put((rank, t, s, lens.tolist()))
    dist.destroy_process_group()


def test_two_rank_weak_scaling_logic():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    assert [x[1] for x in res] == [2.0, 2.0]          # max over ranks
    assert [x[2] for x in res] == [30.0, 30.0]        # sum over ranks
    assert res[0][3] != res[1][3]                     # each rank its own batch
