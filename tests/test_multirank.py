"""The multi-process path of bench.py on CPU (gloo, world size 2): every rank is
an independent replica, the job time is the slowest rank's, and the whole-job
throughput counts the tokens of all ranks."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    w, r, _ = bench.dist_setup(world)
    assert (w, r) == (world, rank) and dist.get_backend() == "gloo"
    bench.barrier(w)
    ms = 100.0 + 50.0 * rank            # the second replica is slower
    m = bench.max_over_ranks(ms, w)
    out[rank] = (m, bench.replica_throughput(w, 1000, 10, m))
    bench.barrier(w)
    dist.destroy_process_group()


def test_two_replicas_on_gloo():
    if torch.cuda.is_available():
        pytest.skip("exercises the CPU (gloo) branch")
    world, port = 2, _free_port()
    out = mp.Manager().dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for rank in range(world):
        m, tps = out[rank]
        assert m == 150.0
        assert tps == pytest.approx(2 * 1000 * 10 / 0.150)
