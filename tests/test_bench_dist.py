"""Host logic of the multi-rank benchmark on CPU: world_size-2 gloo ranks
combine their local times and work the way bench.py does (whole-job units
over the slowest rank's time), only rank 0 of the reference arm runs, and
`bench.py --gpus 2` started without torchrun launches two ranks itself; and
the key of the recorded ncu traffic follows the kernel's code only."""
import json
import os
import socket
import subprocess
import sys

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


ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_gpus_flag_launches_that_many_ranks():
    """--gpus 2 without a torchrun environment: bench.py starts two ranks through
    torch.distributed.run (gloo in the dry run) and rank 0 prints one line for
    the whole job."""
    env = {k: v for k, v in os.environ.items()
           if k not in ("WORLD_SIZE", "RANK", "LOCAL_RANK", "MASTER_ADDR", "MASTER_PORT")}
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--gpus", "2",
                        "--dry-run", "--steps", "5"], capture_output=True, text=True,
                       timeout=300, env=env, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    out = json.loads(lines[0])
    assert out["n_gpus"] == 2 and out["dry_run"]
    # rank r does (r + 1) * 1e6 units per step: 3e6 per step in total
    assert out["units"] == pytest.approx(3.0e6 * 5)
    assert out["value"] == pytest.approx(out["units"] / out["seconds_max"])


def test_gpus_flag_must_match_the_launch(monkeypatch):
    env = dict(os.environ, WORLD_SIZE="1", RANK="0", LOCAL_RANK="0")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--gpus", "2",
                        "--dry-run"], capture_output=True, text=True, timeout=120, env=env,
                       cwd=ROOT)
    assert r.returncode != 0
    assert "WORLD_SIZE" in r.stderr


def test_kernel_source_hash_ignores_comments_only(tmp_path):
    """The recorded ncu traffic is keyed on the product kernel's code: a
    comment or whitespace edit keeps the key, a code edit changes it."""
    import shutil

    sys.path.insert(0, ROOT)
    import bench

    src = os.path.join(ROOT, "paper_2111_11581_gb300", "csrc")
    for f in ("bp_mma.cu", "bp_common.cuh", "bp_internal.h"):
        shutil.copy(os.path.join(src, f), tmp_path / f)
    base = bench.kernel_source_sha(str(tmp_path))
    assert base == bench.kernel_source_sha()
    p = tmp_path / "bp_internal.h"
    text = p.read_text()
    p.write_text("// a note\n/* a block\n   comment */\n" + text.replace("\n", "\n\n", 3))
    assert bench.kernel_source_sha(str(tmp_path)) == base
    p.write_text(text + "\nconstexpr int kUnused = 1;\n")
    assert bench.kernel_source_sha(str(tmp_path)) != base
