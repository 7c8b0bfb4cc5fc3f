"""The multi-rank path of bench.py on CPU: two gloo ranks, each a replica,
exchange only their timings (MAX) and report the whole-job throughput."""
import os
import socket

import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        mine = [1.0 + rank, 5.0 - rank, 0.25 * (rank + 1)]
        got = bench.reduce_max(mine, dist, "cpu")
        q.put((rank, got, bench.job_value(320, world, got[0])))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_take_max_and_weak_scale():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    out = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, got, value in out:
        assert got == [2.0, 5.0, 0.5]
        assert abs(value - 2 * 320 / 2e-3) < 1e-6


def test_single_rank_is_identity():
    assert bench.reduce_max([1.5, 2.5]) == [1.5, 2.5]
    assert bench.job_value(100, 1, 1.0) == 1e5


def test_reference_arm_runs_on_rank_zero_only(monkeypatch, capsys):
    """Under torchrun the reference arm (the oracle on the host) runs and
    prints on rank 0 alone; every other rank exits 0 without work."""
    import argparse
    import workloads as wl
    monkeypatch.setenv("RANK", "1")
    args = argparse.Namespace(steps=1, warmup=3, gpus=2)
    assert bench.reference_arm(args, wl.CONFIGS["tiny"]) == 0
    assert capsys.readouterr().out == ""
