"""The compression pipeline end to end on the GPU, through the C ABI: each
member is aligned to its dominant (lx_align_cost, lx_lap_solve,
lx_permute_neurons; Sec. 3.2 Stage 3 i), its three residuals are compressed
at full rank (lx_compress_factor; Stage 3 ii), the compressed layer is
installed (lx_load_compressed_layer; Stage 3 iii) and run (lx_moe_forward).

Members are planted as the dominant with its neurons permuted plus a smaller
independent N(0, 0.005) part, so the alignment must recover the planted
permutation exactly.  At full rank the factors reproduce the aligned residual,
and the permutation preserves each expert's function, so the compressed
layer's output equals the uncompressed MoE of the original members (the
oracle's dense forward).  Bar: 1e-4 of max|y| -- the fp32 compression
(relative error ~1e-6 of the residual, measured on the emulated algorithm)
stacked on the fp32 forward (1e-5).
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu

H, I, E, K = 128, 64, 4, 2


def _draw(rng, shape, std):
    return (rng.standard_normal(shape) * std).astype(np.float32)


def planted_members(seed=0):
    rng = np.random.default_rng(seed)
    dom = (_draw(rng, (I, H), 0.02), _draw(rng, (I, H), 0.02), _draw(rng, (H, I), 0.02))
    members, sigmas = [], []
    for _ in range(E - 1):
        s = rng.permutation(I)
        mem = (dom[0][s] + _draw(rng, (I, H), 0.005), dom[1][s] + _draw(rng, (I, H), 0.005),
               dom[2][:, s] + _draw(rng, (H, I), 0.005))
        members.append(mem)
        sigmas.append(s)
    router = _draw(rng, (E, H), 0.02)
    omegas = [[rng.standard_normal((shape[1], I)).astype(np.float32)
               for shape in ((I, H), (I, H), (H, I))] for _ in range(E - 1)]
    return dom, members, sigmas, router, omegas


def dense_layer(dom, members, router):
    """Every expert its own anchor holding its full (unaligned) weights."""
    experts = [dom] + members
    return synth.CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype="f32",
        node_parent=np.full(E, -1, np.int32), node_rank=np.zeros(E, np.int32),
        expert_node=np.arange(E, dtype=np.int32), node_w=[tuple(e) for e in experts],
        router_w=router, router_bias=None, top_k=K)


def compressed_layer(dom, factors, router):
    """Expert 0 the dominant (the anchor), experts 1.. its rank-min(H, I) corrections."""
    r = min(H, I)
    return synth.CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype="f32",
        node_parent=np.asarray([-1] + [0] * (E - 1), np.int32),
        node_rank=np.asarray([0] + [r] * (E - 1), np.int32),
        expert_node=np.arange(E, dtype=np.int32), node_w=[tuple(dom)] + factors,
        router_w=router, router_bias=None, top_k=K)


def test_align_compress_install_forward():
    dom, members, sigmas, router, omegas = planted_members()
    d = lambda a: torch.from_numpy(np.ascontiguousarray(a)).cuda()
    dom_d = tuple(d(w) for w in dom)
    factors = []
    r = min(H, I)
    for m, (mem, sigma) in enumerate(zip(members, sigmas)):
        cost = lx.align_cost(dom_d, tuple(d(w) for w in mem))
        P, _ = lx.lap_solve(cost.cpu().numpy())
        inv = np.empty(I, np.int64)
        inv[sigma] = np.arange(I)
        assert np.array_equal(P, inv)                       # the planted alignment
        aligned = lx.permute_neurons(d(P), *[d(w) for w in mem])
        fac = []
        for p in range(3):
            U, V, s = lx.compress_factor(dom_d[p], aligned[p], d(omegas[m][p]), r, 2)
            fac += [U.cpu().numpy(), V.cpu().numpy()]
        torch.cuda.synchronize()
        factors.append(tuple(np.ascontiguousarray(f) for f in fac))
    comp = compressed_layer(dom, factors, router)
    L = lx.Layer(comp)
    x = synth.tokens(comp, 96, seed=5)
    y = L.moe_forward(d(x), K)
    torch.cuda.synchronize()
    ref = oracle.moe_forward(dense_layer(dom, members, router), x)
    err = float(np.max(np.abs(y.cpu().numpy().astype(np.float64) - ref)) / np.max(np.abs(ref)))
    assert L.info()["device_error"] == 0
    assert err <= 1e-4, f"rel err {err}"
