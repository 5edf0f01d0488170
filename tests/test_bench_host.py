"""Host logic of the multi-rank bench (one replica per rank, no data-path
collective): world-size-2 gloo ranks on CPU check that every rank gets the
slowest rank's time, that the whole-job rate counts every rank's tokens, that
ranks draw distinct batches, and that only rank 0 of the reference arm works."""
import os
import socket
import sys

import numpy as np
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


def _routed_stats(src, T, seed):
    import oracle
    import synth
    x = synth.tokens(src, T, seed=seed)
    ids, _, _ = oracle.route(src, x)
    b = oracle.buckets(src, ids)
    return bench.routing_stats(src, b["node_off"], T, src.top_k), b


def test_tensor_core_flop_table_sums_to_the_cost_model():
    """The six tensor-core GEMMs' FLOPs (bench.kernel_flops) add up to the
    amortised forward's expert FLOPs (cost.step_counts) on the realised
    routing: each (token, node) pair counted once, anchors 2*3IH, rank-r
    corrections 2*3r(I+H)."""
    import synth
    from paper_2608_07814_gb300 import cost
    for src in (synth.tree_layer(256, 192, 2, 4, 3, 128, 64, 8, "bf16", seed=15,
                                 skew=synth.TREE_SKEW),
                synth.flat_layer(320, 448, [1, 3, 1, 5, 2], [64, 128, 192, 64, 64, 128, 192], 3,
                                 "bf16", seed=14)):
        st, b = _routed_stats(src, 300, seed=3)
        total = sum(bench.kernel_flops(n, st, src) for n in
                    ("tc_up_anchor", "tc_up_V", "tc_up_U", "tc_dn_anchor", "tc_dn_V", "tc_dn_U"))
        ref = cost.step_counts(src.d_model, src.d_ff, src.n_experts, src.node_parent,
                               src.node_rank, st["cnt"], 300, 2, 2)["expert_flops"]
        assert total == ref


def test_routing_stats_match_the_buckets():
    import synth
    src = synth.flat_layer(256, 128, [4] * 4, 64, 4, "bf16", seed=10, skew=synth.QWEN_SKEW)
    st, b = _routed_stats(src, 200, seed=1)
    cnt = np.diff(b["node_off"].astype(np.int64))
    anchors = np.asarray(src.node_parent) < 0
    assert st["R_anchor"] + st["R_corr"] == len(b["node_tok"])
    assert st["touched_anchor"] == int(np.sum((cnt > 0) & anchors))
    assert st["corr_r_rows"] == int(np.sum(cnt[~anchors] * np.asarray(src.node_rank)[~anchors]))


def test_streaming_weight_bytes_match_the_cost_model():
    """The weight bytes inside the four streaming ops' byte counts (the part
    that scales with the element size, less the gathered token rows) are the
    cost model's touched-weight bytes: every touched node's weights once."""
    import synth
    from paper_2608_07814_gb300 import cost
    src = synth.tree_layer(256, 192, 2, 4, 3, 128, 64, 8, "bf16", seed=15, skew=synth.TREE_SKEW)
    st, b = _routed_stats(src, 64, seed=2)
    ops = ("stream_up_anchor_V", "stream_up_U", "stream_dn_anchor_V", "stream_dn_U")
    scaled = sum(bench.kernel_bytes(n, st, src, 2) - bench.kernel_bytes(n, st, src, 0) for n in ops)
    x_rows = (st["R_anchor"] + st["R_corr"]) * src.d_model * 2
    ref = cost.step_counts(src.d_model, src.d_ff, src.n_experts, src.node_parent, src.node_rank,
                           st["cnt"], 64, 2, 2)["weight_bytes"]
    assert scaled - x_rows == ref
    assert bench.kernel_bytes("stream_up", st, src, 2) + bench.kernel_bytes("stream_dn", st, src, 2) \
        == sum(bench.kernel_bytes(n, st, src, 2) for n in ops)
