"""The multi-GPU path's host logic on CPU: two ranks over gloo (127.0.0.1).

Every rank runs its own batch (distinct seeds, same shapes), the timing is
reduced with MAX over ranks, the job throughput counts every rank's work over
the slowest rank's time, and only rank 0 reports -- in the GPU arm and in the
reference arm, whose other ranks exit without work."""
import io
import json
import os
import socket
import sys
import contextlib

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    from paper_1807_11091_gb300 import ranks
    import workloads as wl
    ws, r, local = ranks.dist_env()
    # each rank's batch: same shape, distinct images
    L = wl.single2d()[0]
    x = wl.gen_tensors(L.shape, seed=ranks.shard_seed(L.seed, r))["x"]
    xs = [torch.zeros_like(x) for _ in range(world)]
    dist.all_gather(xs, x)
    distinct = not torch.equal(xs[0], xs[1])
    # slowest rank's time
    mine = 10.0 + 5.0 * r
    worst = ranks.max_over_ranks(mine)
    value = ranks.job_throughput(1e9, ws, 4, worst)
    out[r] = {"ws": ws, "rank": r, "local": local, "distinct": distinct, "worst": worst, "value": value,
              "reports": ranks.reports(r)}
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_over_gloo():
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.start_processes(_worker, args=(2, port, out), nprocs=2, join=True, start_method="spawn")
        res = dict(out)
    assert sorted(res) == [0, 1]
    for r in (0, 1):
        assert res[r]["ws"] == 2 and res[r]["rank"] == r and res[r]["local"] == r
        assert res[r]["distinct"]
        assert res[r]["worst"] == 15.0  # the slower rank's total
        assert res[r]["value"] == pytest.approx(1e9 * 2 * 4 / 15e-3)
    assert res[0]["reports"] and not res[1]["reports"]


def test_reference_arm_other_ranks_exit_without_work(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = type("A", (), {"workload": "single2d", "steps": 1, "warmup": 1, "gpus": 2})()
    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        assert bench.run_reference(args) == 0
    assert buf.getvalue() == ""


def test_single_process_needs_no_process_group():
    sys.path.insert(0, ROOT)
    from paper_1807_11091_gb300 import ranks
    assert ranks.max_over_ranks(3.5) == 3.5
    assert ranks.job_throughput(2.0, 1, 3, 1.5) == pytest.approx(2.0 * 3 / 1.5e-3)
