"""bench.py's multi-rank logic on CPU: two gloo ranks on this host.

With N GPUs, bench.py runs N independent replicas; the job time is the
slowest rank's (max over ranks, after a barrier), and only rank 0 runs the
CPU reference arm. These tests check that host-side logic without a GPU.
"""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        bench.barrier(world)
        # each rank reports a different time; every rank must see the largest
        t = bench.max_over_ranks(1.5 + rank, world)
        # the reference arm: only rank 0 does work (the others return at once)
        class A:
            steps, warmup, gpus = 1, 0, world
        did = bench.run_reference(A(), world, rank) if rank != 0 else None
        out.put((rank, t, did))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_rank0_only_reference():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = sorted(q.get(timeout=5) for _ in range(world))
    assert [r for r, _, _ in got] == [0, 1]
    assert all(t == 1.5 + (world - 1) for _, t, _ in got)
    assert got[1][2] is None   # rank 1's reference arm returned without work


def test_single_rank_max_is_identity():
    import bench
    assert bench.max_over_ranks(3.25, 1) == 3.25
    bench.barrier(1)   # no process group needed


def test_reference_arm_prints_one_line(capsys):
    # the reference arm (the oracle on the host cores) on the headline
    # workload's config, at one step: one JSON line with the contract's keys
    import json

    import bench

    class A:
        steps, warmup, gpus = 1, 0, 1
    bench.run_reference(A(), 1, 0)
    lines = [ln for ln in capsys.readouterr().out.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "GFLOP/s" and d["value"] > 0
    assert d["higher_is_better"] is True and d["cpu_baseline"]["cores"] >= 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["config"]["workload"] == bench.WORKLOAD
