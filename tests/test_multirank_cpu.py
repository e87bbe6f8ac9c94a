"""The N > 1 host path of bench.py on CPU: two gloo ranks (no GPU).

Each rank decodes its own sequences (no data-path collective); the only
cross-rank operation is the max over ranks of the timed interval."""
import os
import socket

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


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    import gen

    ms = [12.5, 20.0][rank]
    mx = bench.max_over_ranks(ms, dist, "cpu")
    w = gen.config(0).with_(seed=bench.rank_seed(gen.config(0).seed, rank))
    u = w.u_table()
    k, _ = w.kv_block(0, 0, 0, 8, u)
    q.put((rank, mx, bench.job_throughput(100, world, mx), w.seed, float(k.sum())))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_max_time_and_distinct_sequences():
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
    (r0, mx0, v0, s0, k0), (r1, mx1, v1, s1, k1) = res
    assert mx0 == mx1 == 20.0                       # job time = slowest rank
    assert v0 == v1 == pytest.approx(2 * 100 / 0.020)
    assert s0 != s1 and k0 != k1                     # ranks decode different sequences


def test_single_rank_passthrough():
    import bench

    assert bench.max_over_ranks(3.0, None) == 3.0
    assert bench.job_throughput(10, 1, 1000.0) == 10.0
