"""The multi-GPU path of bench.py on the CPU: two gloo ranks.

The batch shards with no data-path exchange (each rank transforms its own
transforms); the only collective is the max of the timings.  These tests run
bench's own helpers in two processes over gloo at 127.0.0.1.
"""
import os
import socket

import numpy as np
import pytest


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import inputs
    wl = dict(inputs.WORKLOADS["n4096_b64"])
    wl["batch"] = 2
    seed = bench.rank_seed(wl, rank)
    x = inputs.make(wl["kind"], wl["n"], wl["batch"], seed)
    # per-rank "time": rank 1 is slower
    local_ms = 10.0 + 5.0 * rank
    job_ms = bench.max_over_ranks(local_ms, dist, "cpu")
    rate = bench.job_rate(bench.dft_flops(wl["n"], wl["batch"]), world, 3, job_ms)
    dist.barrier()
    dist.destroy_process_group()
    q.put((rank, seed, float(np.abs(x).sum()), job_ms, rate))


def test_two_rank_weak_scaling_helpers():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in range(2))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, s0, a0, t0, v0), (r1, s1, a1, t1, v1) = res
    assert (r0, r1) == (0, 1)
    assert s0 != s1 and a0 != a1          # each rank its own inputs
    assert t0 == t1 == 15.0               # the slowest rank sets the time
    assert v0 == v1
    import bench
    assert v0 == pytest.approx(bench.dft_flops(4096, 2) * 2 * 3 / 15e-3 / 1e9)


def test_single_process_is_identity():
    import bench
    assert bench.max_over_ranks(3.5, None, "cpu") == 3.5
