"""Host logic of the multi-GPU bench path (replicas: every rank owns its own sequences and no
data crosses ranks), run as two gloo ranks on the CPU."""
import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)

    def rsum(x):
        t = torch.tensor([float(x)], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.SUM)
        return float(t.item())

    def rmax(x):
        t = torch.tensor([float(x)], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    seqs = bench.shard_sequences(rank, world, 128, 1024)
    tokens = 100.0 * (rank + 1)
    secs = 2.0 + rank
    value, tok, el = bench.aggregate(tokens, secs, rsum, rmax)
    q.put((rank, seqs[0], seqs[-1], value, tok, el))
    dist.destroy_process_group()


def test_two_rank_sharding_and_aggregation():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, a0, b0, v0, t0, e0), (r1, a1, b1, v1, t1, e1) = res
    assert (a0, b0) == (0, 127) and (a1, b1) == (128, 255)   # disjoint sequence groups
    assert t0 == t1 == 300.0 and e0 == e1 == 3.0             # all tokens over the slowest rank
    assert abs(v0 - 100.0) < 1e-12 and v0 == v1


def test_sharding_wraps_the_stream():
    assert bench.shard_sequences(7, 8, 128, 1024)[-1] == 1023
    assert bench.shard_sequences(8, 9, 128, 1024)[0] == 0
