"""GPU parity of neuron alignment (lx_align_cost, lx_permute_neurons, and
lx_lap_solve on the GPU's cost) against the CPU oracle (oracle/align.py),
through the C ABI.

Bar: cost within max|C - C_ref| / max|C_ref| <= 1e-5 (fp32 accumulation
against the float64 squared-distance definition); the permutation found from
the GPU cost is optimal for the oracle's cost up to that rounding (several
permutations can be optimal) and equals a planted permutation exactly;
permuted matrices bit-exact.  Sizes: the Qwen3-30B-A3B expert shape
(H = 2048, I = 768) and ragged shapes that leave partial 64-neuron tiles and
partial 32-deep K chunks.
"""
import numpy as np
import pytest
import torch

import synth
from oracle import align
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu


def _dev(a, dtype):
    return lx.host_to_torch(a, dtype).cuda()


def _pair(H, I, dtype, seed, planted=False, noise=0.02):
    """(dominant, member) storage triples: independent N(0, 0.02) experts, or a
    member that is the dominant with its neurons permuted plus N(0, noise)."""
    rng = np.random.default_rng(seed)
    draw = lambda s, std: rng.standard_normal(s).astype(np.float32) * np.float32(std)
    dom = [draw((I, H), 0.02), draw((I, H), 0.02), draw((H, I), 0.02)]
    if planted:
        sigma = rng.permutation(I)
        mem = [dom[0][sigma] + draw((I, H), noise), dom[1][sigma] + draw((I, H), noise),
               dom[2][:, sigma] + draw((H, I), noise)]
    else:
        sigma = None
        mem = [draw((I, H), 0.02), draw((I, H), 0.02), draw((H, I), 0.02)]
    dom = tuple(synth.to_storage(w, dtype) for w in dom)
    mem = tuple(synth.to_storage(w, dtype) for w in mem)
    return dom, mem, sigma


def _f64(t, dtype):
    return tuple(synth.from_storage(w, dtype) for w in t)


# bf16 with d_model a multiple of 256 takes the tensor-core form (ragged
# 128-row tiles and column chunks below); the other bf16 shapes the 64 x 64
# tile form
CASES = [(2048, 768, "bf16", False), (2048, 768, "bf16", True), (40, 72, "f32", False),
         (40, 72, "bf16", True), (136, 200, "f32", True), (8, 8, "f32", False),
         (264, 64, "bf16", False), (128, 200, "bf16", False), (256, 200, "bf16", False),
         (256, 136, "bf16", True), (256, 24, "bf16", True), (512, 328, "bf16", False)]


@pytest.mark.parametrize("H,I,dtype,planted", CASES)
def test_cost_and_assignment(H, I, dtype, planted):
    """Every cost entry at the small sizes; at the full expert shape 24 sampled
    dominant neurons' rows (the oracle computes a row at a time)."""
    dom, mem, sigma = _pair(H, I, dtype, seed=H + I, planted=planted)
    full = I * H <= 64 * 1024
    rows = None if full else np.unique(np.concatenate(
        [[0, I - 1], np.random.default_rng(I).choice(I, 22, replace=False)]))
    C = align.cost_matrix(_f64(dom, dtype), _f64(mem, dtype), rows=rows)
    cost = lx.align_cost(tuple(_dev(w, dtype) for w in dom), tuple(_dev(w, dtype) for w in mem))
    torch.cuda.synchronize()
    cg = cost.cpu().numpy().astype(np.float64)
    assert np.max(np.abs((cg if full else cg[rows]) - C)) <= 1e-5 * np.max(np.abs(C))
    P, tot = lx.lap_solve(cost.cpu().numpy())
    assert sorted(P.tolist()) == list(range(I))
    if full:
        best = align.assignment_cost(C, align.assign(C))
        assert align.assignment_cost(C, P) - best <= 1e-5 * abs(best) + 1e-9
    if planted:
        inv = np.empty(I, np.int64)
        inv[sigma] = np.arange(I)
        assert np.array_equal(P, inv)


@pytest.mark.parametrize("H,I,dtype", [(2048, 768, "bf16"), (40, 72, "f32"), (136, 200, "bf16")])
def test_permute_bit_exact_and_residual_vanishes(H, I, dtype):
    dom, mem, sigma = _pair(H, I, dtype, seed=7 * H + I, planted=True, noise=0.0)
    P = np.empty(I, np.int32)
    P[sigma] = np.arange(I, dtype=np.int32)          # the planted alignment
    ref = align.permute_expert(*mem, P)
    outs = lx.permute_neurons(torch.from_numpy(P).cuda(), *[_dev(w, dtype) for w in mem])
    torch.cuda.synchronize()
    for o, r, d in zip(outs, ref, dom):
        got = o.cpu()
        got = got.view(torch.int16).numpy().view(np.uint16) if dtype == "bf16" else got.numpy()
        assert np.array_equal(got, r)
        assert np.array_equal(got, d)          # W_m^P - W_dom = 0 for an exact permutation


def test_rejected_calls():
    g = torch.zeros((16, 16), dtype=torch.float32, device="cuda")
    L = lx.lib()
    p = lx._ptr(g)
    assert L.lx_align_cost(7, 16, 16, p, p, p, p, p, p, p, None) == lx.LX_ERR_ARG
    assert L.lx_align_cost(lx.LX_F32, 12, 16, p, p, p, p, p, p, p, None) == lx.LX_ERR_SHAPE
    assert L.lx_align_cost(lx.LX_F32, 16, 16, None, p, p, p, p, p, p, None) == lx.LX_ERR_ARG
    odd = torch.zeros(16 * 16 + 1, dtype=torch.float32, device="cuda")[1:]
    assert L.lx_align_cost(lx.LX_F32, 16, 16, lx._ptr(odd), p, p, p, p, p, p,
                           None) == lx.LX_ERR_ARG
    perm = torch.arange(16, dtype=torch.int32, device="cuda")
    assert L.lx_permute_neurons(lx.LX_F32, 16, 16, lx._ptr(perm), p, p, p, p, p, p,
                                None) == lx.LX_ERR_ARG   # in place
