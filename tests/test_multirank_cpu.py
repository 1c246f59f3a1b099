"""The N>1 bench path on CPU ranks (gloo, world size 2): every rank runs an independent
replica, so the only collective is the timing reduction (max over ranks), and the
whole-job value counts every rank's work against the slowest rank's time."""
import multiprocessing as mp
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w, r, lr = bench.dist_setup()
    local_ms = 100.0 + 50.0 * rank
    ms_max = bench.dist_max(local_ms, w)
    bench.barrier(w)
    q.put((r, w, lr, ms_max, bench.job_value(2e12, 10, w, ms_max)))
    dist.destroy_process_group()


def test_two_rank_timing_reduction_and_job_value():
    pytest.importorskip("torch.distributed")
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [o[0] for o in out] == [0, 1]
    for r, w, lr, ms_max, val in out:
        assert w == 2 and lr == r
        assert ms_max == 150.0                       # the slower rank sets the time
        assert abs(val - 2e12 * 10 * 2 / 0.150 / 1e12) < 1e-9
