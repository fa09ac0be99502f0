"""The N > 1 path of the benchmark on CPU: two gloo ranks, each with its own
batch, the job time taken as the maximum over ranks, and the whole-job value
counting every rank's tokens (weak scaling, no data-path collective)."""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2608_13578_gb300.inputs import HEADLINE, WORKLOADS, make_inputs


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, lr, ws = bench.dist_env()
        assert (r, lr, ws) == (rank, rank, world)
        w = WORKLOADS[HEADLINE].replace(B=1, T=16, D=64, H=1)
        x = make_inputs(w, seed=bench.rank_seed(w.seed, rank))["x"]
        gathered = [torch.zeros_like(x) for _ in range(world)]
        dist.all_gather(gathered, x)
        my_ms = 10.0 + 5.0 * rank               # rank 1 is the slow one
        job_ms = bench.max_over_ranks(my_ms, world)
        value = bench.job_tokens_per_s(world, w.B * w.T, 4, job_ms)
        out.put((rank, job_ms, value, [g.sum().item() for g in gathered]))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_rank, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    res = [q.get(timeout=120) for _ in range(world)]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    res.sort()
    # both ranks agree on the slowest time and on the job value
    assert res[0][1] == res[1][1] == 15.0
    assert res[0][2] == res[1][2] == pytest.approx(2 * 16 * 4 / 0.015)
    # the ranks drew different batches
    sums = res[0][3]
    assert sums[0] != sums[1]
