"""The multi-GPU replica path of bench.py on CPU (gloo, world size 2): every
rank times its own batch, the job time is the slowest rank's, the value is
all ranks' checks over that time.  No data-path collective exists."""
import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(('127.0.0.1', 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, out):
    import bench
    os.environ['MASTER_ADDR'] = '127.0.0.1'
    os.environ['MASTER_PORT'] = str(port)
    dist.init_process_group('gloo', rank=rank, world_size=world)
    ms, vms = bench.max_over_ranks([10.0 + 5 * rank, 3.0 - rank])
    out[rank] = (ms, vms, bench.job_value(1024, world, ms))
    dist.barrier()
    dist.destroy_process_group()


def test_replicas_take_the_slowest_rank():
    world = 2
    port = _free_port()
    mgr = mp.Manager()
    out = mgr.dict()
    mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
    for r in range(world):
        ms, vms, v = out[r]
        assert ms == 15.0 and vms == 3.0
        assert v == pytest.approx(2 * 1024 / 0.015)
