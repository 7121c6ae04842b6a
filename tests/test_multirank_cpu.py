"""The N > 1 benchmark path on CPU: two gloo ranks split the matrices of a
model (flop-balanced, disjoint, complete) and reduce their step times with a
max, as bench.py does over NCCL on GPUs."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _rank_main(rank, world, port, q):
    import torch
    import torch.distributed as dist

    import bench
    from paper_2609_35701_gb300 import workloads as W

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    wl = W.get_workload("llama350m")
    shapes = [(r, c) for _, r, c in wl.shapes]
    parts = bench.partition(shapes, world)
    mine = parts[rank]
    # every rank derives the same split
    got = [None] * world
    dist.all_gather_object(got, mine)
    # the reported time is the max over ranks
    t = torch.tensor([float(10 + rank)])
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    q.put((rank, got, [sum(bench.ns_flops(min(shapes[i]), max(shapes[i]), 5)[0] for i in p) for p in parts],
           float(t.item())))
    dist.destroy_process_group()


def test_two_rank_partition_and_max_time():
    world = 2
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    from paper_2609_35701_gb300 import workloads as W

    n = len(W.get_workload("llama350m").shapes)
    for rank, got, loads, tmax in res:
        assert tmax == 11.0
        assert got[0] == res[0][1][0] and got[1] == res[0][1][1]
        allidx = sorted(got[0] + got[1])
        assert allidx == list(range(n)) and not set(got[0]) & set(got[1])
        assert max(loads) / min(loads) < 1.02   # flop-balanced
