"""Screened routing against the full router, through the C ABI.

Large bf16 batches whose caller needs only the ids and gates (lx_moe_forward,
or lx_route without a logits buffer) take approximate logits from the tensor
cores and compute the canonical fp32 logits of the candidates only: every
expert whose approximate logit is within twice the error bound of the k-th
largest.  The bound makes the candidate set contain the exact top-k, so the
ids, their order and the gates must equal the full router's bit for bit (the
full router runs when a logits buffer is passed) and the oracle's ids.  The
cases cover the Qwen3-shaped router, E = 256, exact ties (duplicated router
rows, decided by the lower id), all logits equal (every expert a candidate:
the fallback to all E canonical logits) and a dense cluster of near-ties.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu

T_SCREEN = 2048  # above the large-batch router's threshold (8 tokens x 152 SMs)


def _routes(src, x_host, k):
    L = lx.Layer(src)
    x = lx.host_to_torch(x_host, "bf16").cuda()
    ids_s, w_s = L.route(x, k)                                  # screened
    ids_f, w_f, logits = L.route(x, k, want_logits=True)        # full router
    torch.cuda.synchronize()
    L.free()
    return (ids_s.cpu().numpy(), w_s.cpu().numpy(), ids_f.cpu().numpy(), w_f.cpu().numpy(),
            logits.cpu().numpy())


def _check(src, x_host, k):
    ids_s, w_s, ids_f, w_f, _ = _routes(src, x_host, k)
    assert np.array_equal(ids_s, ids_f), "screened ids differ from the full router's"
    assert np.array_equal(w_s.view(np.uint32), w_f.view(np.uint32)), "gates differ"
    o_ids, _, _ = oracle.route(src, x_host)
    assert np.array_equal(ids_s, o_ids), "ids differ from the oracle's"
    return ids_s


def test_screened_equals_full_qwen_router():
    src = synth.flat_layer(2048, 128, [4] * 32, 64, 8, "bf16", seed=41, skew=synth.QWEN_SKEW)
    _check(src, synth.tokens(src, T_SCREEN, seed=3), 8)


def test_screened_equals_full_256_experts():
    src = synth.flat_layer(512, 128, [8] * 32, 64, 8, "bf16", seed=42)
    _check(src, synth.tokens(src, T_SCREEN + 37, seed=4), 8)


def test_screened_exact_ties():
    src = synth.flat_layer(512, 128, [4] * 8, 64, 4, "bf16", seed=43)
    src.router_w[5] = src.router_w[2]   # experts 2, 5 and 7 tie on every token
    src.router_w[7] = src.router_w[2]
    ids = _check(src, synth.tokens(src, T_SCREEN, seed=5), 4)
    for row in ids:
        pos = {e: list(row).index(e) for e in (2, 5, 7) if e in row}
        assert sorted(pos, key=pos.get) == sorted(pos)


def test_screened_all_equal_logits_fall_back():
    src = synth.flat_layer(512, 128, [4] * 16, 64, 8, "bf16", seed=44)
    src.router_w[:] = src.router_w[0]
    src.router_bias = None
    ids = _check(src, synth.tokens(src, T_SCREEN, seed=6), 8)
    assert np.all(ids == np.arange(8)[None, :])   # every tie goes to the lower ids


def test_screened_near_ties():
    src = synth.flat_layer(512, 128, [4] * 16, 64, 8, "bf16", seed=45)
    rng = np.random.default_rng(7)
    base = synth.from_storage(src.router_w[0:1], "bf16")
    pert = base + rng.standard_normal((64, 512)).astype(np.float32) * np.float32(1e-3)
    src.router_w[:] = synth.to_storage(pert, "bf16")
    src.router_bias = None
    _check(src, synth.tokens(src, T_SCREEN, seed=8), 8)
