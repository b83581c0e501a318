"""Multi-process host logic of bench.py's N>1 path (weak-scaling replicas),
run as world_size-2 gloo ranks on the CPU: every rank times its own batch and
the job takes the slowest rank."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    ms = [10.0, 25.0][rank]  # rank 1 is the slower replica
    value, mx = bench.combine_ranks(ms, units_per_rank=1000, dist=dist)
    # every rank also seeds its own batch: rank-dependent inputs, same shape
    import workloads

    b = workloads.exact_enum(seed=rank, rows_scale=1.0, groups=((4, 64),))[0]
    q.put((rank, value, mx, float(b.logits[0])))
    dist.destroy_process_group()


def test_weak_scaling_takes_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    for rank, value, mx, _ in res:
        assert mx == 25.0
        assert value == pytest.approx(2 * 1000 / 25e-3)
    assert res[0][3] != res[1][3]  # replicas draw different inputs
