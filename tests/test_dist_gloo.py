"""Multi-rank host logic of bench.py on CPU (gloo, world_size 2).

With N GPUs every rank trains an independent replica (model seed + rank) with
no collective on the data path; the only collectives are the timing reductions
(max of the elapsed time, sum of the samples) and barriers."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import numpy as np
    import torch.distributed as dist

    import bench
    import oracle as O

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    r, w, lr = bench.dist_env()
    elapsed = 1.5 + rank                      # rank 1 is the slow one
    mx = bench.max_over_ranks(elapsed)
    total = bench.sum_over_ranks(1000.0 * (rank + 1))
    bench.barrier()
    seed = bench.replica_seed(5, rank)
    m = O.OracleModel([16, 8], 2, seed=seed, bs=4)
    H = m.H(1)
    m.close()
    out.put((rank, r, w, lr, mx, total, seed, H.tobytes()))
    dist.destroy_process_group()


def test_two_rank_reductions_and_independent_replicas():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, rr0, w0, l0, mx0, tot0, s0, H0), (r1, rr1, w1, l1, mx1, tot1, s1, H1) = res
    assert (rr0, rr1, w0, w1, l0, l1) == (0, 1, 2, 2, 0, 1)
    assert mx0 == mx1 == 2.5                      # time = max over ranks
    assert tot0 == tot1 == 3000.0                 # samples = sum over ranks
    assert s0 != s1 and H0 != H1                  # independent replicas


def test_single_process_helpers_are_identity():
    import bench
    assert bench.max_over_ranks(3.0) == 3.0
    assert bench.sum_over_ranks(7.0) == 7.0
    bench.barrier()
    assert bench.dist_env()[1] >= 1


def test_bench_arithmetic():
    import bench
    w = (8192, 8192, 8192, 8192, 8192)
    assert bench.bitpairs_per_sample(w, 10) == 4 * 8192 * (8192 + 10)
    # int16 H read + write (8192 x 8192 x 2 x 2 bytes) + packed W (8192 x 128 x 8) per layer
    assert bench.update_bytes_per_launch(w) == 4 * (8192 * 8192 * 4 + 8192 * 128 * 8)
    assert bench.update_bytes_per_launch((784, 256)) == 256 * (13 * 64 * 4 + 13 * 8)
