"""Host logic of the multi-rank bench (one replica per rank, no data-path
collective): world-size-2 gloo ranks on CPU check that every rank gets the
slowest rank's time, that the whole-job rate counts every rank's tokens, that
ranks draw distinct batches, and that only rank 0 of the reference arm works."""
import os
import socket
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    try:
        torch.distributed.barrier()
        mine = [10.0 + 5.0 * rank, 30.0 - 7.0 * rank]  # rank 1 slower, rank 0 slower in e2e
        got = bench.max_over_ranks(mine, world, "cpu")
        out[rank] = got
    finally:
        torch.distributed.destroy_process_group()


def test_max_over_ranks_gloo_world2():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, join=True,
                           start_method="spawn")
        res = dict(out)
    assert res[0] == res[1] == [15.0, 30.0]


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks([1.5, 2.5], 1) == [1.5, 2.5]


def test_whole_job_rate_counts_every_rank():
    # 64 tokens per rank-step, 100 steps, 4 ranks, slowest rank 20 ms
    assert bench.whole_job_rate(64, 100, 4, 20.0) == pytest.approx(64 * 100 * 4 / 0.02)
    assert bench.whole_job_rate(64, 100, 1, 20.0) * 4 == pytest.approx(
        bench.whole_job_rate(64, 100, 4, 20.0))


def test_ranks_draw_distinct_batches():
    seeds = {bench.batch_seed(r, b) for r in range(8) for b in range(8)}
    assert len(seeds) == 64


def test_reference_arm_only_rank0_works():
    class A:
        workload, ref_tokens, warmup, steps = "decode64", 2, 3, 1
    assert bench.run_reference(A(), rank=1, world=2) is None
