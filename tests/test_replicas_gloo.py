"""Multi-process host logic of bench.py's replica mode, on CPU with gloo (world size 2):
the job time is the slowest rank's, the barrier releases every rank, and each
replica decodes its own token batch.  The data path has no collective."""
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


def _worker(rank, world, port, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    t = bench.max_over_ranks(1.5 + rank, world)
    bench.barrier(world)
    toks = bench.replica_tokens(4096, rank)
    out.put((rank, t, toks.shape, int(toks[:, :8].sum())))
    dist.destroy_process_group()


def test_two_replicas_timing_and_token_streams():
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
    (r0, t0, s0, h0), (r1, t1, s1, h1) = res
    assert t0 == t1 == 2.5            # max over ranks, seen by both
    assert s0 == s1 == (16, 1537)     # batch 16, prompt 512 + 1024 steps + 1 target
    assert h0 != h1                   # distinct token streams per replica
