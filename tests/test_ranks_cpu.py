"""The benchmark's multi-rank bookkeeping on CPU with the gloo backend
(world size 2): replicas take one independent event per rank (different
seeds, the same shape), and the job's time is the slowest rank's while its
work is the sum of the ranks' hits."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
torch = pytest.importorskip("torch")


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    from paper_2009_04509_gb300 import synth
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        planes = synth.apa(seed=rank, hits=(120, 100, 80))
        nhits = sum(p.nhits for p in planes)
        ms, units = bench.reduce_over_ranks(10.0 + 5.0 * rank, nhits * 3, dist, "cpu")
        first_adc = float(planes[0].adc[0, :64].sum())
        out.put((rank, ms, units, nhits, first_adc))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=10) for _ in range(2))
    (_, ms0, u0, n0, a0), (_, ms1, u1, n1, a1) = res
    assert ms0 == ms1 == 15.0                  # the slowest rank's time, on every rank
    assert u0 == u1 == 3 * (n0 + n1)           # every rank's hits counted once
    assert n0 == n1 == 300 and a0 != a1        # same shape, independent events


def test_single_process_passthrough():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_over_ranks(12.5, 7, None, "cpu") == (12.5, 7)
