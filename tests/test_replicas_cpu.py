"""The multi-GPU path is replicas only (no exchange step): bench.py times every rank on its own
workload and reports all ranks' tokens over the slowest rank's time.  Checked here with two gloo
ranks on the CPU, each claiming a different time."""
import os
import socket

import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _rank(rank, world, port, q):
    import sys

    import torch.distributed as dist

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench

    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        value, ms_max = bench.replica_throughput(10.0 * (rank + 1), 1000, device="cpu")
        q.put((rank, value, ms_max))
    finally:
        dist.destroy_process_group()


def test_replica_throughput_two_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(q.get(timeout=10) for _ in range(2))
    for rank, value, ms_max in got:
        assert ms_max == 20.0  # the slowest rank's time
        assert abs(value - 2 * 1000 / 0.020) < 1e-6  # both ranks' tokens over that time


def test_single_process_needs_no_group():
    import sys

    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench

    value, ms = bench.replica_throughput(4.0, 500, device="cpu")
    assert ms == 4.0 and abs(value - 500 / 0.004) < 1e-6
