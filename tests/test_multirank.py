"""The multi-GPU path of bench.py on CPU: two gloo ranks run the benchmark's
per-rank path -- each builds the headline workload's assets and its own query
stream of the same recipe, decodes its shard (here with the oracle, the one
decoder a CPU rank has), times the step, and takes the whole-job rate as all
queries over the slowest rank's step time (no collective on the data path, only
the timing reduction)."""
import os
import socket
import time

import numpy as np
import pytest
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
    import oracle
    w = bench.workload(bench.HEADLINE, True, rank)
    dist.barrier()
    t0 = time.perf_counter()
    dec, bad = oracle.decode(w.assets, w.queries, nthreads=1)
    ms_local = 1e3 * (time.perf_counter() - t0)
    value, ms = bench.aggregate(len(w.queries), ms_local, dist)
    digest = int(np.frombuffer(w.queries.tobytes(), dtype=np.uint64).sum() % (1 << 62))
    adigest = int(np.frombuffer(w.assets.latents.tobytes(), dtype=np.uint64).sum() % (1 << 62))
    out[rank] = (value, ms, ms_local, digest, adigest, len(w.queries), bad, float(dec.min()), float(dec.max()),
                 dec[:64].copy())
    dist.barrier()
    dist.destroy_process_group()


def test_two_gloo_ranks_decode_their_own_shards_and_take_the_slowest_step():
    world, port = 2, _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_rank, args=(world, port, out), nprocs=world, join=True)
    (v0, ms0, l0, q0, a0, n0, b0, lo0, hi0, d0), (v1, ms1, l1, q1, a1, n1, b1, lo1, hi1, d1) = out[0], out[1]
    assert ms0 == ms1 == pytest.approx(max(l0, l1))  # max over ranks
    assert v0 == v1 == pytest.approx((n0 + n1) / (ms0 / 1e3))
    assert q0 != q1                                   # different query streams
    assert a0 == a1                                   # replicated assets
    assert n0 == n1 and b0 == b1 == 0
    assert 0.0 <= min(lo0, lo1) and max(hi0, hi1) <= 1.0  # sigmoid outputs
    assert not np.array_equal(d0, d1)                 # each rank decoded its own queries
