"""The N > 1 benchmark path on the CPU: two gloo ranks (one process each, as
torchrun launches them) draw disjoint requests, take the slowest rank's
time with an all-reduce, and only rank 0 reports.  No data-path collective
exists: requests are independent replicas."""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      RANK=str(rank), WORLD_SIZE=str(world))
    import bench
    from workloads import WORKLOADS, draw_request
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        ids = bench.rank_requests(rank, world, n_sets=3, batch=2)
        gathered = [None] * world
        dist.all_gather_object(gathered, ids)
        # per-rank "timings": the job time is the slowest rank's
        mx = bench.max_over_ranks([10.0 + rank, 3.0 * (world - rank)], world)
        # the first request of each rank drafts different base logits
        wl = WORKLOADS["tiny"].with_(batch=3 * 2 * world)
        L = draw_request(wl, ids[0][0])[0]
        Ls = [None] * world
        dist.all_gather_object(Ls, L[0, :8].tolist())
        q.put((rank, gathered, mx, Ls))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q))
             for r in range(world)]
    for p in procs:
        p.start()
    out = {}
    for _ in range(world):
        rank, gathered, mx, Ls = q.get(timeout=120)
        out[rank] = (gathered, mx, Ls)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    gathered, mx, Ls = out[0]
    flat = [i for ids in gathered for s in ids for i in s]
    assert sorted(flat) == list(range(world * 3 * 2))     # disjoint, complete
    assert out[1][0] == gathered
    assert mx == [11.0, 6.0] and out[1][1] == mx           # same max on all
    assert Ls[0] != Ls[1]


def test_aggregate_and_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([1.5, 2.0], 1) == [1.5, 2.0]
    # 4 ranks x 100 steps x 1 request in 250 ms (slowest rank)
    assert bench.job_rounds_per_s(250.0, 100, 4, 1) == pytest.approx(1600.0)
    ids = bench.rank_requests(0, 1, 2, 3)
    assert ids == [[0, 1, 2], [3, 4, 5]]


def test_reference_arm_other_ranks_do_nothing(capsys):
    sys.path.insert(0, ROOT)
    import bench
    from workloads import WORKLOADS

    class A:
        steps, warmup = 1, 1
    assert bench.run_reference(A(), WORKLOADS["tiny"], rank=1, world=2) is None
    assert capsys.readouterr().out == ""
