"""The benchmark's multi-rank path on the host (world size 2, gloo, no GPU).

`bench.py --gpus N` runs one replica of the workload per rank with no collective on the data path:
a barrier before each timed region, the max of the ranks' timings, rank 0 printing.  These tests
run that host logic in two processes: the barrier, the max over ranks, the whole-job rate of the
replicas (weak scaling), and the reference arm leaving ranks other than 0 without work.
"""
import io
import json
import os
import socket
import sys
from contextlib import redirect_stdout

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, outdir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import torch
    import bench

    ctx = bench.DistCtx(backend="gloo")
    ctx.init(torch)
    try:
        ctx.barrier()
        ms_local = 10.0 * (rank + 1)                  # rank 1 is the slow one
        ms = ctx.max(ms_local)
        units = 1000
        rec = {"rank": ctx.rank, "world": ctx.world, "ms_max": ms, "value": bench.job_rate(ctx.world, units, ms)}
        with open(os.path.join(outdir, f"rank{rank}.json"), "w") as f:
            json.dump(rec, f)
        ctx.barrier()
    finally:
        ctx.pg.destroy_process_group()


def test_two_rank_barrier_max_and_job_rate(tmp_path):
    mp = pytest.importorskip("torch.multiprocessing")
    world = 2
    mp.spawn(_rank, args=(world, _free_port(), str(tmp_path)), nprocs=world, join=True)
    recs = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(world)]
    assert [r["rank"] for r in recs] == [0, 1]
    for r in recs:
        assert r["world"] == world
        assert r["ms_max"] == 20.0                     # the slowest rank's time, seen by every rank
        # weak scaling: 2 replicas x 1000 units in 20 ms
        assert r["value"] == pytest.approx(2 * 1000 / 0.020)


def test_job_rate_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.job_rate(1, 500, 250.0) == pytest.approx(2000.0)
    assert bench.job_rate(4, 500, 250.0) == pytest.approx(8000.0)


def test_reference_arm_other_ranks_exit_without_work(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("LOCAL_RANK", "1")

    class Args:
        gpus, steps, warmup = 2, 1, 3

    buf = io.StringIO()
    with redirect_stdout(buf):
        assert bench.run_reference(Args()) == 0
    assert buf.getvalue() == ""


def test_refresh_flops_and_tensor_peak():
    sys.path.insert(0, ROOT)
    import bench
    import workloads as W
    cfg = W.config("cfg2_resnet")
    # (2 q + 1) passes of 2 m' n' k flops over the stack's 6,266,880 matrix elements, q = 4, k = 16
    assert bench.refresh_flops(cfg, 16) == 9 * 2 * 6_266_880 * 16
    peak, kind = bench.tensor_peak_tflops()
    assert peak > 100 and kind in ("measured", "fallback")
