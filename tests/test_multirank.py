"""The multi-GPU path of bench.py on CPU: two gloo ranks, each with its own
query shard and the same assets, aggregated as all queries over the slowest
rank's step time (no collective on the data path, only the timing reduction)."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    w = bench.workload(True, rank)
    ms_local = 2.0 + rank  # rank 1 is the slower one
    value, ms = bench.aggregate(len(w.queries), ms_local, dist)
    digest = int(np.frombuffer(w.queries.tobytes(), dtype=np.uint64).sum() % (1 << 62))
    adigest = int(np.frombuffer(w.assets.latents.tobytes(), dtype=np.uint64).sum() % (1 << 62))
    out[rank] = (value, ms, digest, adigest, len(w.queries))
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_queries_and_take_the_slowest_step():
    world, port = 2, _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
    (v0, ms0, q0, a0, n0), (v1, ms1, q1, a1, n1) = out[0], out[1]
    assert ms0 == ms1 == 3.0                    # max over ranks
    assert v0 == v1 == pytest.approx((n0 + n1) / 3.0e-3)
    assert q0 != q1                             # different query shards
    assert a0 == a1                             # replicated assets
