"""The N > 1 path on CPU: two gloo ranks (world size 2, 127.0.0.1).

Chains are independent, so bench.py runs one batch per rank with no data-path
collective (weak scaling); its only collectives are the barrier and the
max-over-ranks of the timed region.  These tests run that host logic on two
processes, and check on the oracle that chains verified on different ranks give
exactly what one process gives for the whole batch.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

import bench
import workloads as W
from oracle import verify as OV


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, fn, out):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out[rank] = fn(rank, world, dist)
    finally:
        dist.barrier()
        dist.destroy_process_group()


def _run(fn, world=2):
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        mp.start_processes(_rank_main, args=(world, _free_port(), fn, out), nprocs=world,
                           start_method="spawn", join=True)
        return dict(out)


def _both(rank, world, dist):
    ms = [3.0, 5.0][rank]                      # the ranks' own timed regions
    slowest = bench.max_over_ranks(ms, dist, "cpu")
    rate = bench.whole_job_rate(world, 256 * 8, slowest * 1e-3)
    inp = W.make_verify_inputs("tiny", B=12, L=6, d=40)
    chains = np.arange(rank, 12, world)
    o = OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], 99,
                  OV.MODE_BLOCK, chains=chains)
    return slowest, rate, chains.tolist(), o["accepted_len"].tolist(), o["y"].tolist()


@pytest.fixture(scope="module")
def two_ranks():
    return _run(_both)


def test_max_over_ranks_and_whole_job_rate(two_ranks):
    assert two_ranks[0][:2] == two_ranks[1][:2]
    slowest, rate = two_ranks[0][:2]
    assert slowest == 5.0
    assert rate == pytest.approx(2 * 256 * 8 / 5e-3)
    assert bench.max_over_ranks(7.0, None, "cpu") == 7.0


def test_chain_shards_equal_one_process_run(two_ranks):
    inp = W.make_verify_inputs("tiny", B=12, L=6, d=40)
    full = OV.verify(inp["x_draft"], inp["mu_target"], inp["mu_draft"], inp["sigma"], 99, OV.MODE_BLOCK)
    for rank in (0, 1):
        chains, acc, y = two_ranks[rank][2:]
        np.testing.assert_array_equal(np.asarray(acc), full["accepted_len"][chains])
        np.testing.assert_array_equal(np.asarray(y), full["y"][chains])


def test_ranks_verify_distinct_inputs():
    base = W.VERIFY_CONFIGS["tiny"]["seed"]
    seeds = {(i, r): bench.input_seed(base, i, r) for i in range(8) for r in range(8)}
    assert len(set(seeds.values())) == len(seeds)
    a = W.make_verify_inputs("tiny", seed=bench.input_seed(base, 0, 0))
    b = W.make_verify_inputs("tiny", seed=bench.input_seed(base, 0, 1))
    assert not np.array_equal(a["x_draft"], b["x_draft"])
