"""Host-side logic of bench.py's N > 1 path (independent replicas) with two
gloo ranks on the CPU: each rank contributes its own timings, every rank gets
the maximum, and the job's rate counts all ranks' work over that time."""
import os
import socket
import sys

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r measured (1 + r) ms per step and 10 - r ms per e2e step
        got = bench.reduce_max_over_ranks([1.0 + rank, 10.0 - rank], world)
        dist.barrier()
        out[rank] = got + [bench.whole_job_rate(6.0, world, got[0])]
    finally:
        dist.destroy_process_group()


def test_replica_reduction_two_gloo_ranks():
    world = 2
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][:2] == [2.0, 10.0] and res[1][:2] == [2.0, 10.0]
    # 2 ranks x 6 units over the slowest rank's 2 ms
    assert res[0][2] == res[1][2] == 2 * 6.0 / 2e-3


def test_single_rank_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max_over_ranks([3.0, 4.0], 1) == [3.0, 4.0]
    assert bench.whole_job_rate(5.0, 1, 1.0) == 5000.0
