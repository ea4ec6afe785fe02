"""Host-side logic of bench.py's N-GPU path on CPU ranks (gloo, world size 2):
every rank times its own replica; the job's time is the max over ranks and the
whole-job ms per step divides it by all ranks' steps."""
import os
import socket

import pytest
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import torch.distributed as dist
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    local = [120.0, 95.5][rank]
    mx = bench.reduce_max_ms(local)
    out[rank] = (mx, bench.job_ms_per_step(mx, 8, world))
    dist.barrier()
    dist.destroy_process_group()


def test_max_over_ranks_and_whole_job_rate():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    assert out[0] == out[1] == (120.0, 120.0 / 16)


def test_single_process_path():
    import bench
    assert bench.reduce_max_ms(42.0) == 42.0
    assert bench.job_ms_per_step(80.0, 8, 1) == 10.0
