"""The benchmark's multi-GPU host logic on CPU with two gloo ranks (no GPU): one
batch per rank with the same shape and different data (weak scaling, no collective on
the data path), the slowest rank's time as the job's time, the whole-job value, and
the reference arm's other ranks leaving without work."""
import os
import socket

import numpy as np
import pytest


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    import torch.distributed as dist
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ms = [3.0, 5.0][rank]  # rank 1 is the slower one
    slowest = bench.max_over_ranks(ms)
    b = bench.make_workload("tiny", rank)
    shape = (len(b["group_rollout_off"]), len(b["step_len"]), b["emb"].shape)
    T = bench.batch_tokens(b)
    total = bench.sum_over_ranks(T)
    dist.barrier()
    q.put((rank, slowest, bench.whole_job_value(total, slowest), shape, float(np.asarray(b["emb"]).sum()),
           bench.dist_env(), T, total))
    dist.destroy_process_group()


def test_two_gloo_ranks():
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=240) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    (r0, s0, v0, sh0, e0, env0, T0, tot0), (r1, s1, v1, sh1, e1, env1, T1, tot1) = res
    assert s0 == s1 == 5.0  # every rank sees the slowest rank's time
    assert tot0 == tot1 == T0 + T1  # the job's tokens: all ranks'
    assert v0 == v1 == pytest.approx((T0 + T1) / 5e-3)
    assert sh0 == sh1  # the same shape on every rank ...
    assert e0 != e1  # ... with its own data (seed offset by rank)
    assert env0 == (2, 0, 0) and env1 == (2, 1, 1)


def test_whole_job_value_and_single_rank(monkeypatch):
    import bench
    assert bench.whole_job_value(4000, 2.0) == pytest.approx(4000 / 2e-3)
    assert bench.max_over_ranks(7.5) == 7.5  # no process group: the rank's own value
    assert bench.sum_over_ranks(7.5) == 7.5


def test_reference_arm_other_ranks_exit_without_work(monkeypatch, capsys):
    import argparse

    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = argparse.Namespace(config="math", steps=1, warmup=0, gpus=2)
    assert bench.run_reference(args) == 0
    assert capsys.readouterr().out == ""
