"""The N > 1 host path of bench.py on CPU: two gloo ranks (world size 2)
combine their timed totals the way the GPU run does (max over ranks, whole-job
rate over all ranks' tokens), draw different inputs, and the reference arm runs
on rank 0 only. No GPU, no NCCL."""
import os
import socket
import sys

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        local_ms = 10.0 * (rank + 1)           # rank 1 is the slow one
        t, v = bench.whole_job(local_ms, 1000, world, "cpu")
        seeds = [None] * world
        dist.all_gather_object(seeds, bench.rank_seed(4, rank))
        out[rank] = (t, v, tuple(seeds))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_the_slowest_rank_and_all_tokens():
    world = 2
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True)
        res = dict(out)
    for rank in range(world):
        t, v, seeds = res[rank]
        assert t == 20.0                              # max over ranks
        assert abs(v - 2 * 1000 / 20e-3 / 1e6) < 1e-12  # all ranks' tokens over the slowest time
        assert len(set(seeds)) == world               # every rank draws its own batch


def test_single_rank_needs_no_collective():
    sys.path.insert(0, ROOT)
    import bench
    t, v = bench.whole_job(5.0, 500, 1, "cpu")
    assert t == 5.0 and abs(v - 0.1) < 1e-12


def test_reference_arm_runs_on_rank_0_only(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    monkeypatch.setenv("RANK", "1")

    class A:
        steps = warmup = None
        workload = "single"
    assert bench.run_reference(A()) == 0  # returns at once, prints nothing
