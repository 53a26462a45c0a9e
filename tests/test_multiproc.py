"""Host logic of the multi-replica benchmark with two gloo ranks on the CPU:
every rank verifies its own seeded replica (no data exchange); the timings
are reduced to the slowest rank and the job value counts all ranks' nodes."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        from paper_2609_02897_gb300 import synth
        # timings: the job is as slow as its slowest rank, element by element
        got = bench.slowest_rank([1.0 + rank, 10.0 - rank], world, "cpu")
        # replicas: distinct seeded workloads, same shapes
        wl = synth.make_workload(2, rep=rank, small=True)
        sig = [float(np.sum(wl.q)), int(wl.T)]
        sigs = [None] * world
        dist.all_gather_object(sigs, sig)
        value = bench.job_value(wl.T, world, got[0])
        q.put((rank, got, sigs, value))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
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
    for rank, got, sigs, value in res:
        assert got == [2.0, 10.0]
        assert sigs[0][0] != sigs[1][0]          # different replicas
        assert value == pytest.approx(2 * sigs[rank][1] / 2.0)


def test_reference_arm_other_ranks_do_nothing(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")

    class A:
        steps, warmup, gpus = 1, 0, 2
    bench.run_reference(A())
    assert capsys.readouterr().out == ""
