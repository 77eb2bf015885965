"""The N > 1 path of bench.py on the CPU: two gloo ranks (world size 2).

Attention has no exchange step, so the multi-GPU path is replicas: every rank
runs its own seeded copy of the workload, the ranks meet at barriers around the
timed region, and the slowest rank's time sets the whole-job throughput.
"""
import os
import socket
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist
    import bench
    from paper_2405_13226_gb300 import workloads as wl

    r, w, local = bench.dist_setup(world, backend="gloo")
    assert (r, w, local) == (rank, world, rank)
    # the slowest rank's time is the job's time
    t = bench.max_over_ranks(10.0 + 5.0 * rank, w)
    bench.barrier(w)
    # every rank draws its own replica of the inputs (seed = rank)
    q, _, _, _ = wl.attn_inputs(1, 256, 2, 64, seed=rank)
    digest = torch.tensor([int(np.bitwise_xor.reduce(q.view(np.uint16).ravel().astype(np.int64)))],
                          dtype=torch.int64)
    gathered = [torch.zeros_like(digest) for _ in range(w)]
    dist.all_gather(gathered, digest)
    # the reference arm runs on rank 0 only; other ranks return without work
    ref = None
    if rank != 0:
        ref = bench.run_reference(type("A", (), {"steps": 1, "warmup": 0})())
    np.save(os.path.join(out_dir, "rank%d.npy" % rank),
            np.array([t, float(len({int(g.item()) for g in gathered})), 0.0 if ref is None else 1.0]))
    dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    mp = pytest.importorskip("torch.multiprocessing")
    port = _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    for r in range(2):
        t, n_distinct, ref_ran = np.load(tmp_path / ("rank%d.npy" % r))
        assert t == 15.0             # MAX over ranks, seen by every rank
        assert n_distinct == 2       # the replicas' inputs differ
        assert ref_ran == 0.0        # rank 1 did no reference work


def test_replica_value_is_weak_scaling():
    sys.path.insert(0, ROOT)
    import bench
    one = bench.replica_value(1e12, 10, 1000.0, 1)
    assert one == pytest.approx(10.0)
    # twice the ranks, the same per-rank work in the same time: twice the job throughput
    assert bench.replica_value(1e12, 10, 1000.0, 2) == pytest.approx(2 * one)
