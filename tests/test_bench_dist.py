"""Host logic of the multi-rank benchmark on CPU: world_size-2 gloo ranks
combine their local times and work the way bench.py does (whole-job units
over the slowest rank's time), and only rank 0 of the reference arm runs."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)

    def rmax(v):
        t = torch.tensor([v], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        return float(t.item())

    def rsum(v):
        t = torch.tensor([v], dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.SUM)
        return float(t.item())

    local_s = [0.5, 2.0][rank]
    local_units = [10.0, 30.0][rank]
    value, tmax = bench.aggregate(local_s, local_units, world, rmax, rsum)
    assert bench.dist_setup() == (world, rank, rank)
    q.put((rank, value, tmax))
    dist.destroy_process_group()


def test_two_rank_aggregation_uses_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, value, tmax in res:
        assert tmax == 2.0
        assert value == pytest.approx(40.0 / 2.0)


def test_reference_arm_other_ranks_do_nothing(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class A:
        steps, warmup = 3, 3
    bench.run_reference(A())
    assert capsys.readouterr().out == ""
