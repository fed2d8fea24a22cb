"""Host logic of the multi-rank bench (one rank per GPU) on CPU ranks.

bench.py --gpus N shards one global batch of N x B sequences over the ranks
(the read is independent per (b, h), so no exchange): the step time is the
maximum over ranks and the reported value is the whole job's throughput.
These tests run that plumbing with world_size 2 on the gloo backend, without a
GPU, and check that the shards read separately equal the read of the whole
batch.
"""
import os
import socket
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, queue):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    w_, r_, l_ = bench.dist_env()
    dist = bench.init_dist(w_, backend="gloo")
    bench.barrier(dist)
    ms = 2.0 + rank  # rank 1 is the slow one
    slowest = bench.max_over_ranks(dist, ms)
    value = bench.job_throughput(1.0e12, w_, slowest)
    bench.barrier(dist)
    dist.destroy_process_group()
    queue.put((rank, w_, r_, l_, slowest, value))


def test_two_ranks_take_the_slowest_step_and_sum_the_work():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, queue)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = sorted(queue.get(timeout=10) for _ in range(world))
    for rank, (r, w_, r_, l_, slowest, value) in enumerate(got):
        assert (r, w_, r_, l_) == (rank, 2, rank, rank)
        assert slowest == 3.0
        assert value == pytest.approx(2.0e12 / 3.0e-3 / 1e12)


def _reference_worker(rank, world, port, queue):
    os.environ.update(WORLD_SIZE=str(world), RANK=str(rank), LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import bench
    import io
    import contextlib

    class Args:
        workload, steps, warmup, gpus = "tiny_f32_causal", 1, 0, world

    buf = io.StringIO()
    with contextlib.redirect_stdout(buf):
        bench.run_reference(Args())
    queue.put((rank, buf.getvalue()))


def test_reference_arm_prints_on_rank_zero_only():
    pytest.importorskip("numpy")
    world = 2
    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    procs = [ctx.Process(target=_reference_worker, args=(r, world, 0, queue)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
        assert p.exitcode == 0
    out = dict(queue.get(timeout=10) for _ in range(world))
    assert out[1] == ""
    import json
    line = json.loads(out[0].strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0 and line["n_gpus"] == 2
    assert line["cpu_baseline"]["kind"] == "oracle"


def test_job_throughput_is_weak_scaling():
    sys.path.insert(0, ROOT)
    import bench
    one = bench.job_throughput(1.0995e12, 1, 1.0)
    assert one == pytest.approx(1099.5)
    assert bench.job_throughput(1.0995e12, 4, 1.0) == pytest.approx(4 * one)


def _shard_worker(rank, world, port, queue):
    """One rank: draw this rank's shard of the global batch, read it with the oracle
    (no exchange), then gather the outputs -- in the test only -- for rank 0 to check."""
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE=str(world), RANK=str(rank),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import numpy as np
    import torch
    import torch.distributed as dist

    import oracle
    from paper_2602_07160_gb300 import workloads as W
    w = W.WORKLOADS["tiny_f32_causal"]
    dist.init_process_group("gloo", rank=rank, world_size=world)
    q, k, v, beta = W.make_batch_shard(w, rank, world)
    o, lse = oracle.fem_read(q, k, v, beta, w.causal, nthreads=1)
    got = [torch.empty(o.shape, dtype=torch.float64) for _ in range(world)]
    dist.all_gather(got, torch.from_numpy(np.ascontiguousarray(o)))
    dist.destroy_process_group()
    queue.put((rank, torch.cat(got).numpy() if rank == 0 else None))


def test_batch_shards_read_without_exchange_equal_the_global_read():
    """bench.py's N > 1 layout: the ranks' shards of one global batch, each read on its
    own, give exactly the read of the whole batch (the read is independent per (b, h))."""
    pytest.importorskip("numpy")
    import dataclasses

    import numpy as np
    import torch
    sys.path.insert(0, ROOT)
    import oracle
    from paper_2602_07160_gb300 import workloads as W
    world, port = 2, _free_port()
    w = W.WORKLOADS["tiny_f32_causal"]
    wg = dataclasses.replace(w, B=world * w.B)
    qg, kg, vg, bg = W.make_batch_shard(wg, 0, 1)
    shards = [W.make_batch_shard(w, r, world) for r in range(world)]
    for i in range(3):
        assert torch.equal(torch.cat([s[i] for s in shards]), (qg, kg, vg)[i])
    assert all(torch.equal(s[3], bg) for s in shards)
    assert not torch.equal(shards[0][0], shards[1][0])  # distinct sequences, not copies
    ref, _ = oracle.fem_read(qg, kg, vg, bg, w.causal, nthreads=1)

    ctx = mp.get_context("spawn")
    queue = ctx.Queue()
    procs = [ctx.Process(target=_shard_worker, args=(r, world, port, queue)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    got = dict(queue.get(timeout=10) for _ in range(world))
    np.testing.assert_array_equal(got[0], ref)
