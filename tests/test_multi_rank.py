"""The path shards by images with no data-path collective (CPU, gloo, world size 2).

* bench.py's cross-rank reduction: the job time is the slowest rank's, the work the sum.
* Every rank draws its own shard (seeded by rank) and runs the whole schedule on it alone.
* Sharding is exact: the stages run on each shard separately equal the same stages run on the
  two shards concatenated into one batch, split back per image (the oracle, on the CPU).
"""
import os
import socket
import sys

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import oracle  # noqa: E402
from workloads import Batch, StageSpec, make_workload  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    dist.init_process_group("gloo", rank=rank, world_size=world, init_method=f"tcp://127.0.0.1:{port}")
    try:
        sys.path.insert(0, ROOT)
        import bench
        t, u = bench.reduce_over_ranks(10.0 + 3.0 * rank, 100 * (rank + 1), world, torch.device("cpu"))
        w = make_workload("deit_s_chain12_bf16_b256", batch=6, seed_offset=rank)
        res = oracle.chain(w, stages=4)
        digest = (float(np.asarray(w.batch.x, np.float64).sum()), [int(r["n_out"]) for r in res])
        got = [None] * world
        dist.all_gather_object(got, (rank, t, u, digest))
        if rank == 0:
            out.put(got)
    finally:
        dist.destroy_process_group()


def test_two_ranks_reduce_and_shard():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = q.get(timeout=300)
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    for rank, t, u, _ in got:
        assert t == 13.0 and u == 300.0, (rank, t, u)
    assert got[0][3][0] != got[1][3][0]            # each rank drew its own shard


def _concat(b0: Batch, b1: Batch) -> Batch:
    offs = np.concatenate([b0.offsets, b0.offsets[-1] + b1.offsets[1:]]).astype(np.int32)
    cat = lambda a, c: None if a is None else np.concatenate([a, c])  # noqa: E731
    return Batch(b0.dtype, offs, cat(b0.x, b1.x), cat(b0.keys, b1.keys), cat(b0.sizes, b1.sizes),
                 cat(b0.scores, b1.scores))


@pytest.mark.parametrize("stage", [0, 3])
def test_sharded_stages_equal_the_whole_batch(stage):
    w0 = make_workload("deit_s_chain12_bf16_b256", batch=5, seed_offset=0)
    w1 = make_workload("deit_s_chain12_bf16_b256", batch=7, seed_offset=1)
    s0, s1 = w0.stages[stage], w1.stages[stage]
    head = s0.head
    cat = lambda a, c: None if a is None else np.concatenate([a, c])  # noqa: E731
    whole = oracle.stage(_concat(w0.batch, w1.batch),
                         StageSpec(s0.merge, s0.exit, s0.prune, r=cat(s0.r[:5], s1.r[:7]),
                                   rho=cat(s0.rho[:5], s1.rho[:7]) if s0.rho is not None else None, head=head))
    parts = [oracle.stage(w0.batch, StageSpec(s0.merge, s0.exit, s0.prune, r=s0.r[:5],
                                               rho=None if s0.rho is None else s0.rho[:5], head=head)),
             oracle.stage(w1.batch, StageSpec(s1.merge, s1.exit, s1.prune, r=s1.r[:7],
                                               rho=None if s1.rho is None else s1.rho[:7], head=head))]
    assert whole["n_out"] == parts[0]["n_out"] + parts[1]["n_out"]
    np.testing.assert_array_equal(whole["ids"], np.concatenate([parts[0]["ids"], 5 + parts[1]["ids"]]))
    n0 = int(parts[0]["offsets"][-1])
    np.testing.assert_array_equal(whole["x"][:n0], parts[0]["x"])
    np.testing.assert_array_equal(whole["x"][n0:], parts[1]["x"])
    np.testing.assert_array_equal(whole["sizes"], np.concatenate([parts[0]["sizes"], parts[1]["sizes"]]))
    if s0.exit:
        np.testing.assert_array_equal(whole["exit_mask"], np.concatenate([parts[0]["exit_mask"], parts[1]["exit_mask"]]))
