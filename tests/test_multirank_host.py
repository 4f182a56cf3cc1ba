"""Host logic of a multi-GPU bench run, on CPU with two gloo ranks.

Batch rows are independent problems, so N GPUs scan N batches of the same
shape (weak scaling) with no collective on the data path; the only exchange is
the reduction that reports the slowest rank's time. These tests run that logic
in two processes over gloo, without a GPU.
"""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import bench
    from paper_2406_12580_gb300 import inputs as I
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local = 10.0 + 5.0 * rank                      # this rank's step time
        slowest = bench.max_over_ranks(local, world, device="cpu")
        cfg = bench.rank_workload(I.CONFIGS[1], rank)
        out[rank] = (slowest, cfg.seed, (cfg.B, cfg.L, cfg.D, cfg.io))
    finally:
        dist.destroy_process_group()


def test_two_ranks_report_the_slowest_time_and_scan_distinct_batches():
    world, port = 2, _free_port()
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][0] == res[1][0] == 15.0           # every rank sees the max
    assert res[0][1] != res[1][1]                   # each rank its own batch
    assert res[0][2] == res[1][2]                   # of the same shape


def test_reference_arm_runs_on_rank_zero_only(monkeypatch):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    # a non-zero rank returns at once, before reading its arguments or
    # building anything
    assert bench.run_reference(None) == 0
