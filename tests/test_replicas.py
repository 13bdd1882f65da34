"""Multi-GPU means independent replicas (requests never interact): the only
cross-rank steps are a barrier and a max over ranks of the timed region.
Checked here with two gloo ranks on the CPU."""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch.distributed as dist

    dist.init_process_group("gloo", rank=rank, world_size=world, init_method=f"tcp://127.0.0.1:{port}")
    import bench

    g = bench.ReplicaGroup(world, rank, "cpu")
    g.barrier()
    worst = g.max(1.0 + rank)
    thr = g.throughput(10, 2.0 + rank)  # each rank did 10 units; the slowest took 3 s
    g.barrier()
    q.put((rank, worst, thr))
    dist.destroy_process_group()


def test_two_replicas_barrier_and_max_over_ranks():
    pytest.importorskip("torch")
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
    assert [r[0] for r in res] == [0, 1]
    for _, worst, thr in res:
        assert worst == 2.0
        assert thr == pytest.approx(2 * 10 / 3.0)


def test_single_replica_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench

    g = bench.ReplicaGroup(1, 0, "cpu")
    g.barrier()
    assert g.max(4.5) == 4.5
    assert g.throughput(8, 2.0) == 4.0
