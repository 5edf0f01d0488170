"""Pins of the CPU oracle against facts that do not come from the oracle itself:
closed forms, library routines (SVD, torch dense algebra, sorting), invariants the
paper states, and hand-derived rounding cases of the canonical router order.

A mutation test at the end plants plausible mistakes in the oracle (on the CPU)
and checks that each one fails at least one pin.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from paper_2608_07814_gb300 import cost

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# ----------------------------------------------------------------------------
# helpers: an independent dense MoE in torch (all experts on all tokens, then a
# dense gate matrix) -- a different formulation from the oracle's slot loop.
# ----------------------------------------------------------------------------
def dense_moe_torch(dense, x64, ids, g):
    X = torch.from_numpy(x64)
    T = X.shape[0]
    E = len(dense)
    G = torch.zeros(T, E, dtype=torch.float64)
    G.scatter_(1, torch.from_numpy(ids.astype(np.int64)), torch.from_numpy(g))
    Y = torch.zeros_like(X)
    for e in range(E):
        Wg, Wu, Wd = (torch.from_numpy(np.asarray(w, np.float64)) for w in dense[e])
        h = torch.nn.functional.silu(X @ Wg.T) * (X @ Wu.T)
        Y += G[:, e:e + 1] * (h @ Wd.T)
    return Y.numpy()


def rel_err(y, ref):
    return float(np.max(np.abs(y - ref)) / np.max(np.abs(ref)))


def _full_rank_case(seed=0):
    layer, dense = synth.tiny_layer(seed=seed, rank=64, return_dense=True)
    x = synth.tokens(layer, 64, seed=seed)
    return layer, dense, x


# ----------------------------------------------------------------------------
# router: canonical fp32 order (hand-derived rounding cases)
# ----------------------------------------------------------------------------
def _router_case(H, wvals):
    """Layer with one expert whose router row has the given {index: value};
    x = all ones.  Returns the canonical fp32 logit."""
    layer = synth.tiny_layer(H=H, I=16, clusters=1, cluster_size=1, top_k=1)
    w = np.zeros((1, H), np.float32)
    for h, v in wvals.items():
        w[0, h] = v
    layer.router_w = w
    x = np.ones((1, H), np.float32)
    return float(oracle.router_logits(layer, x)[0, 0])


def test_router_order_within_lane_chain():
    # lane 0 holds h=0..7: 2^24 then +1 then +1, each fmaf rounds to even -> 2^24
    assert _router_case(256, {0: 2.0 ** 24, 1: 1.0, 2: 1.0}) == 2.0 ** 24


def test_router_order_tree_pairs():
    # 1.0 in lane 2 meets lane 0 at off=2 (2^24+1 -> 2^24) ...
    assert _router_case(256, {0: 2.0 ** 24, 8: 1.0, 16: 1.0}) == 2.0 ** 24
    # ... but 1.0 in lane 3 meets lane 1 first (1+1=2), then 2^24+2 is exact
    assert _router_case(256, {0: 2.0 ** 24, 8: 1.0, 24: 1.0}) == 2.0 ** 24 + 2.0


def test_router_chunk_to_lane_map():
    # H=512: chunk 32 (h=256) belongs to lane 0 after chunk 0, so 2^24+1 -> 2^24
    assert _router_case(512, {0: 2.0 ** 24, 256: 1.0}) == 2.0 ** 24
    # h=264 is chunk 33 -> lane 1; lane 1 then holds 2 -> 2^24+2 exact at the end
    assert _router_case(512, {0: 2.0 ** 24, 8: 1.0, 264: 1.0}) == 2.0 ** 24 + 2.0


@pytest.mark.parametrize("dtype,H", [("f32", 64), ("bf16", 2048), ("bf16", 2560)])
def test_router_logits_error_bound(dtype, H):
    rng = np.random.default_rng(1)
    E, T = 16, 32
    layer = synth.flat_layer(H, 32, [4, 4, 4, 4], 4, 2, dtype=dtype, seed=3)
    layer.router_bias = rng.standard_normal(E).astype(np.float32)
    x = synth.tokens(layer, T, seed=5)
    l = oracle.router_logits(layer, x).astype(np.float64)
    X = synth.from_storage(x, dtype)
    W = synth.from_storage(layer.router_w, dtype)
    exact = X @ W.T + layer.router_bias.astype(np.float64)
    # |fl(sum) - sum| <= gamma_n * sum|x w| with n = chain + tree + bias adds
    n = H // 256 * 8 + 8 + 5 + 1
    u = 2.0 ** -24
    gamma = n * u / (1 - n * u)
    bound = gamma * (np.abs(X) @ np.abs(W).T + np.abs(layer.router_bias))
    assert np.all(np.abs(l - exact) <= bound + 1e-30)


# ----------------------------------------------------------------------------
# top-k and gates
# ----------------------------------------------------------------------------
def test_topk_brute_force_with_ties():
    rng = np.random.default_rng(2)
    T, E, k = 200, 24, 5
    l = rng.integers(-3, 4, size=(T, E)).astype(np.float32)   # many ties
    l[:10] = rng.standard_normal((10, E)).astype(np.float32)
    l[10, :] = 0.0
    l[11, ::2] = -0.0                                            # -0 ties +0
    ids = oracle.topk(l, k)
    for t in range(T):
        ref = sorted(range(E), key=lambda e: (-float(l[t, e]), e))[:k]
        assert list(ids[t]) == ref


def test_gates_closed_form():
    rng = np.random.default_rng(3)
    l = rng.standard_normal((50, 12)).astype(np.float32)
    ids = oracle.topk(l, 4)
    g = oracle.gates(l, ids)
    assert np.allclose(g.sum(1), 1.0, atol=1e-15)
    sel = np.take_along_axis(l.astype(np.float64), ids.astype(np.int64), 1)
    assert np.allclose(g[:, 1] / g[:, 0], np.exp(sel[:, 1] - sel[:, 0]), rtol=1e-13)
    assert np.all(np.diff(g, axis=1) <= 1e-15)          # slot order = descending gates
    ids1 = oracle.topk(l, 1)
    assert np.all(oracle.gates(l, ids1) == 1.0)


def test_router_unchanged_by_compression():
    """Sec. 3.2 Stage 1: compression never touches the router, so routing of the
    compressed layer equals routing with any other expert weights."""
    layer = synth.flat_layer(256, 64, [4] * 8, 16, 8, "bf16", seed=7, skew=synth.QWEN_SKEW)
    x = synth.tokens(layer, 40, seed=1)
    ids, g, l = oracle.route(layer, x)
    other = synth.flat_layer(256, 64, [4] * 8, 16, 8, "bf16", seed=7, skew=synth.QWEN_SKEW,
                             zero_factors=True, zero_dominants=True)
    ids2, g2, l2 = oracle.route(other, x)
    assert np.array_equal(ids, ids2) and np.array_equal(g, g2) and np.array_equal(l, l2)


# ----------------------------------------------------------------------------
# forward
# ----------------------------------------------------------------------------
def test_full_rank_reconstruction_equals_uncompressed():
    """Eq. (svd)/(factors) at full rank reproduce W_m exactly, so the compressed
    forward equals the uncompressed MoE (fp32-stored factors: 1e-5)."""
    layer, dense, x = _full_rank_case()
    ids, g, _ = oracle.route(layer, x)
    y = oracle.moe_forward(layer, x)
    ref = dense_moe_torch(dense, synth.from_storage(x, "f32"), ids, g)
    assert rel_err(y, ref) < 1e-5


def test_error_falls_with_rank():
    """Truncating the SVD residual (Eq. svd) at a higher rank retains more of it
    (Table 2's trend), and full rank is exact."""
    errs = []
    for r in (8, 16, 32, 64):
        layer, dense = synth.tiny_layer(rank=r, return_dense=True)
        x = synth.tokens(layer, 64)
        ids, g, _ = oracle.route(layer, x)
        ref = dense_moe_torch(dense, synth.from_storage(x, "f32"), ids, g)
        errs.append(rel_err(oracle.moe_forward(layer, x), ref))
    assert all(a > b for a, b in zip(errs, errs[1:]))
    assert errs[0] > 1e-2 and errs[-1] < 1e-5


def test_dominant_carries_zero_correction():
    """Sec. 3.1: the dominant is stored exactly.  Tokens routed only to dominants
    give the dense MoE of the dominant matrices."""
    layer, dense = synth.tiny_layer(rank=8, return_dense=True)
    x = synth.tokens(layer, 16)
    T = x.shape[0]
    ids = np.tile(np.array([[0, 4]], np.int32), (T, 1))       # the two dominants
    g = np.tile(np.array([[0.7, 0.3]]), (T, 1))
    y = oracle.moe_forward(layer, x, routing=(ids, g))
    ref = dense_moe_torch(dense, synth.from_storage(x, "f32"), ids, g)
    assert rel_err(y, ref) < 1e-12


def test_brute_force_dense_moe_tiny():
    """Oracle slot-loop forward == dense torch MoE over the same reconstructed
    experts (fp64) on the tiny workload."""
    layer = synth.tiny_layer(rank=8)
    x = synth.tokens(layer, 256)
    ids, g, _ = oracle.route(layer, x)
    dense = [oracle.expert_weights(layer, e) for e in range(layer.n_experts)]
    ref = dense_moe_torch(dense, synth.from_storage(x, "f32"), ids, g)
    assert rel_err(oracle.moe_forward(layer, x), ref) < 1e-12


def test_swiglu_closed_form():
    """One expert, k=1, Wg = diag(a), Wu = Wd = I:  y = silu(a*x) * x."""
    H = I = 8
    layer = synth.tiny_layer(H=H, I=I, clusters=1, cluster_size=1, top_k=1, dtype="f64")
    a = np.linspace(-2.0, 2.0, H)
    layer.node_w[0] = (np.diag(a), np.eye(I), np.eye(H))
    x = np.linspace(-3.0, 3.0, H)[None, :]
    y = oracle.moe_forward(layer, x, routing=(np.zeros((1, 1), np.int32), np.ones((1, 1))))
    ref = [(a[i] * x[0, i]) / (1.0 + math.exp(-a[i] * x[0, i])) * x[0, i] for i in range(H)]
    assert np.allclose(y[0], ref, rtol=1e-14, atol=1e-15)


def _flat_from_tree(tree):
    """Flat layer in which every expert is its own anchor holding the sum of its
    tree path, summed here independently of the oracle."""
    f64 = lambda a: synth.from_storage(a, tree.dtype)
    node_w = []
    for e in range(tree.n_experts):
        n = int(tree.expert_node[e])
        acc = [np.zeros((tree.d_ff, tree.d_model)), np.zeros((tree.d_ff, tree.d_model)),
               np.zeros((tree.d_model, tree.d_ff))]
        while n >= 0:
            w = tree.node_w[n]
            if tree.node_parent[n] < 0:
                for p in range(3):
                    acc[p] = acc[p] + f64(w[p])
            else:
                sg = 1.0 if tree.node_sign is None else float(tree.node_sign[n])
                for p in range(3):
                    acc[p] = acc[p] + sg * np.einsum("ir,jr->ij", f64(w[2 * p]),
                                                     f64(w[2 * p + 1]))
            n = int(tree.node_parent[n])
        node_w.append(tuple(acc))
    return synth.CompressedLayer(
        d_model=tree.d_model, d_ff=tree.d_ff, n_experts=tree.n_experts, dtype="f64",
        node_parent=np.full(tree.n_experts, -1, np.int32),
        node_rank=np.zeros(tree.n_experts, np.int32),
        expert_node=np.arange(tree.n_experts, dtype=np.int32), node_w=node_w,
        router_w=tree.router_w, router_bias=tree.router_bias, top_k=tree.top_k)


def test_tree_equals_flat():
    """Sec. 5: the tree is an organisation of the same experts, not a change of
    function; App. C Table 6 (tree vs flat quality-neutral)."""
    tree = synth.tree_layer(64, 48, 2, 2, 3, 12, 4, 4, "f32", seed=11, factor_std="visible",
                            skew=synth.TREE_SKEW)
    x = synth.tokens(tree, 50, seed=2)
    ids, g, _ = oracle.route(tree, x)
    flat = _flat_from_tree(tree)
    y_tree = oracle.moe_forward(tree, x, routing=(ids, g))
    y_flat = oracle.moe_forward(flat, synth.from_storage(x, "f32"), routing=(ids, g))
    assert rel_err(y_tree, y_flat) < 1e-12
    # and the corrections matter (the test would be vacuous otherwise)
    zero = synth.tree_layer(64, 48, 2, 2, 3, 12, 4, 4, "f32", seed=11, zero_factors=True,
                            skew=synth.TREE_SKEW)
    assert rel_err(oracle.moe_forward(zero, x, routing=(ids, g)), y_tree) > 1e-2


# ----------------------------------------------------------------------------
# BTExperts variants: Fig. 2's binary tree with -1/+1 edges, and a single shared
# base (the single-shared-component layout of Sec. 5.2)
# ----------------------------------------------------------------------------
def test_signed_binary_tree_equals_flat():
    """A Fig. 2 binary tree with signed edges is the flat layer whose experts are
    the signed sums along their root paths (summed independently above)."""
    tree = synth.binary_tree_layer(64, 48, 2, 3, [12, 8, 4], 4, "f32", seed=21,
                                   factor_std="visible", signed=True, skew=synth.TREE_SKEW)
    assert tree.node_sign is not None and set(np.unique(tree.node_sign)) == {-1, 1}
    assert max(len(tree.path(e)) for e in range(tree.n_experts)) == 4
    x = synth.tokens(tree, 50, seed=3)
    ids, g, _ = oracle.route(tree, x)
    flat = _flat_from_tree(tree)
    y_tree = oracle.moe_forward(tree, x, routing=(ids, g))
    y_flat = oracle.moe_forward(flat, synth.from_storage(x, "f32"), routing=(ids, g))
    assert rel_err(y_tree, y_flat) < 1e-12
    # the signs matter: the unsigned tree is another function
    tree.node_sign = None
    assert rel_err(oracle.moe_forward(tree, x, routing=(ids, g)), y_tree) > 1e-2


def test_sibling_edges_cancel():
    """Two leaves below one root through edges -1 and +1 that carry the same
    factors average to the root and differ by twice the correction."""
    tree = synth.binary_tree_layer(32, 24, 1, 1, [6], 2, "f64", seed=22,
                                   factor_std="visible", signed=True)
    left, right = int(tree.expert_node[0]), int(tree.expert_node[1])
    tree.node_w[right] = tree.node_w[left]
    e_left, e_right = (0, 1) if tree.node_sign[left] < 0 else (1, 0)
    Wl = oracle.expert_weights(tree, e_left)
    Wr = oracle.expert_weights(tree, e_right)
    root = tree.node_w[0]
    fac = tree.node_w[left]
    for p in range(3):
        assert np.allclose(0.5 * (Wl[p] + Wr[p]), root[p], rtol=0, atol=1e-15)
        assert np.allclose(Wr[p] - Wl[p], 2.0 * np.einsum("ir,jr->ij", fac[2 * p], fac[2 * p + 1]),
                           rtol=0, atol=1e-14)


def test_single_base_full_rank_equals_uncompressed():
    """One shared base (not an expert) with every expert a full-rank correction
    (Eq. svd / factors of W_e - base) is the uncompressed MoE."""
    rng = np.random.default_rng(23)
    H, I, E = 32, 48, 6
    dense = [tuple(rng.standard_normal(s) * 0.02 for s in [(I, H), (I, H), (H, I)])
             for _ in range(E)]
    base = tuple(np.mean([d[p] for d in dense], axis=0) for p in range(3))
    node_w = [tuple(synth.to_storage(b, "f32") for b in base)]
    for e in range(E):
        fac = []
        for p in range(3):
            B, At = synth._svd_factors(dense[e][p] - synth.from_storage(node_w[0][p], "f32"),
                                       min(H, I))
            fac += [B, At]
        node_w.append(tuple(synth.to_storage(f, "f32") for f in fac))
    layer = synth.CompressedLayer(
        d_model=H, d_ff=I, n_experts=E, dtype="f32",
        node_parent=np.asarray([-1] + [0] * E, np.int32),
        node_rank=np.asarray([0] + [min(H, I)] * E, np.int32),
        expert_node=np.arange(1, E + 1, dtype=np.int32), node_w=node_w,
        router_w=synth.to_storage(rng.standard_normal((E, H)) * 0.02, "f32"),
        router_bias=None, top_k=3)
    x = synth.tokens(layer, 40, seed=4)
    ids, g, _ = oracle.route(layer, x)
    ref = dense_moe_torch(dense, synth.from_storage(x, "f32"), ids, g)
    assert rel_err(oracle.moe_forward(layer, x), ref) < 1e-5


# ----------------------------------------------------------------------------
# bucketing
# ----------------------------------------------------------------------------
def _bucket_reference_numpy(layer, ids):
    """Vectorised formulation: all (node, token) pairs -> np.unique."""
    T, k = ids.shape
    paths = [layer.path(e) for e in range(layer.n_experts)]
    D = max(len(p) for p in paths)
    pairs = []
    for t in range(T):
        for s in range(k):
            for n in paths[ids[t, s]]:
                pairs.append((n, t))
    keys = np.unique(np.array([n * T + t for n, t in pairs], np.int64))
    nodes, toks = keys // T, keys % T
    off = np.searchsorted(nodes, np.arange(layer.n_nodes + 1)).astype(np.int32)
    node_row = np.full(T * k * D, -1, np.int32)
    for t in range(T):
        for s in range(k):
            for l, n in enumerate(paths[ids[t, s]]):
                node_row[(t * k + s) * D + l] = np.searchsorted(keys, n * T + t)
    flat_ids = ids.reshape(-1)
    perm = np.lexsort((np.arange(T * k), flat_ids)).astype(np.int32)
    eoff = np.searchsorted(np.sort(flat_ids), np.arange(layer.n_experts + 1)).astype(np.int32)
    return off, toks.astype(np.int32), node_row, eoff, perm


@pytest.mark.parametrize("kind", ["flat", "tree", "singletons"])
def test_bucketing_brute_force(kind):
    if kind == "flat":
        layer = synth.flat_layer(64, 32, [4] * 8, 8, 8, "f32", seed=1, skew=synth.QWEN_SKEW)
    elif kind == "tree":
        layer = synth.tree_layer(64, 32, 2, 4, 3, 8, 4, 8, "f32", seed=1, skew=synth.TREE_SKEW)
    else:
        layer = synth.flat_layer(64, 32, [1, 3, 1, 4, 1, 2], 8, 3, "f32", seed=1)
    x = synth.tokens(layer, 97, seed=4)
    ids, _, _ = oracle.route(layer, x)
    b = oracle.buckets(layer, ids)
    off, toks, node_row, eoff, perm = _bucket_reference_numpy(layer, ids)
    assert np.array_equal(b["node_off"], off)
    assert np.array_equal(b["node_tok"], toks)
    assert np.array_equal(b["node_row"], node_row)
    assert np.array_equal(b["expert_off"], eoff)
    assert np.array_equal(b["perm"], perm)
    # invariants
    assert b["expert_off"][-1] == ids.size
    assert sorted(b["perm"].tolist()) == list(range(ids.size))
    for n in range(layer.n_nodes):
        seg = b["node_tok"][b["node_off"][n]:b["node_off"][n + 1]]
        assert np.all(np.diff(seg) > 0)


# ----------------------------------------------------------------------------
# closed forms of the cost model (Fig. 3, Sec. 3.1/3.3)
# ----------------------------------------------------------------------------
def test_fig3_closed_forms():
    gold = json.load(open(os.path.join(GOLDEN, "fig3_flops.json")))
    s = gold["shape"]
    I, H, k, r, b = s["I"], s["H"], s["k"], s["r"], s["bytes_per_elem"]
    assert cost.dense_proj_flops(I, H, 1) == gold["closed_form"]["two_IH"]
    assert 2 * r * (I + H) == gold["closed_form"]["two_r_I_plus_H"]
    assert abs(cost.proj_speedup(I, H, k, r) - gold["closed_form"]["speedup"]) < 1e-5
    p = gold["printed"]
    assert round(cost.dense_proj_flops(I, H, k) / 1e6) == p["original_flops_M"]
    assert round(cost.amortised_proj_flops(I, H, k, r) / 1e6) == p["amortised_flops_M"]
    assert round(I * H * b / 1e6) == p["per_expert_mb"]
    assert round(r * (I + H) * b / 1e6, 1) == p["correction_mb"]
    assert round((I * H + k * r * (I + H)) * b / 1e6) == p["amortised_mb"]
    assert round(cost.proj_speedup(I, H, k, r), 1) == p["speedup_approx"]


def test_storage_roughly_half():
    gold = json.load(open(os.path.join(GOLDEN, "storage_half.json")))
    s = gold["shape"]
    layer = synth.flat_layer(64, 32, [2] * (s["E"] // 2), 4, 2, "f32")   # structure only
    frac = cost.kept_fraction(s["H"], s["I"], s["E"], layer.node_parent,
                              [0 if p < 0 else s["r"] for p in layer.node_parent])
    assert abs(frac - gold["closed_form"]["kept_fraction"]) < 1e-6
    assert abs(frac - gold["printed"]["kept_fraction_approx"]) < 0.1


def test_step_counts_match_fig3_group():
    """One cluster, two co-selected members sharing a dominant, one token: the
    counter's gate/up/down totals are 3x Fig. 3's single-projection figures."""
    I, H, r = 14336, 4096, 64
    c = cost.step_counts(H, I, 3, [-1, 0, 0], [0, r, r], [1, 1, 1], 1, 2, 2)
    assert c["expert_flops"] == 3 * cost.amortised_proj_flops(I, H, 2, r)
    assert c["weight_bytes"] == 3 * (I * H + 2 * r * (I + H)) * 2


# ----------------------------------------------------------------------------
# mutation test: plausible mistakes planted in the oracle must fail a pin
# ----------------------------------------------------------------------------
def _mut_drop_correction(layer, n, p):
    return 0.0 * oracle.__dict__["_orig_correction"](layer, n, p)


def _mut_negative_correction(layer, n, p):
    return -oracle.__dict__["_orig_correction"](layer, n, p)


def _mut_swapped_pair(layer, n, p):
    q = {0: 1, 1: 0, 2: 2}[p]
    return oracle.__dict__["_orig_correction"](layer, n, q)


def _mut_sigmoid(z):
    return 1.0 / (1.0 + np.exp(-z))


def _mut_topk_high_id(logits, k):
    T, E = logits.shape
    ids = np.broadcast_to(np.arange(E), (T, E))
    order = np.lexsort((-ids, -logits.astype(np.float64)), axis=1)
    return np.ascontiguousarray(order[:, :k].astype(np.int32))


def _mut_uniform_gates(logits, ids):
    return np.full(ids.shape, 1.0 / ids.shape[1])


def _mut_unsigned(layer, n):
    return 1.0


def _pins_pass():
    try:
        test_full_rank_reconstruction_equals_uncompressed()
        test_dominant_carries_zero_correction()
        test_topk_brute_force_with_ties()
        test_gates_closed_form()
        test_swiglu_closed_form()
        test_tree_equals_flat()
        test_signed_binary_tree_equals_flat()
        test_sibling_edges_cancel()
        test_single_base_full_rank_equals_uncompressed()
    except AssertionError:
        return False
    return True


@pytest.mark.parametrize("target,mutant", [
    ("_correction", _mut_drop_correction),
    ("_correction", _mut_negative_correction),
    ("_correction", _mut_swapped_pair),
    ("silu", _mut_sigmoid),
    ("topk", _mut_topk_high_id),
    ("gates", _mut_uniform_gates),
    ("edge_sign", _mut_unsigned),
])
def test_planted_mistakes_fail_a_pin(monkeypatch, target, mutant):
    assert _pins_pass()
    oracle.__dict__["_orig_correction"] = oracle._correction
    monkeypatch.setattr(oracle, target, mutant)
    assert not _pins_pass()


def test_forward_from_reconstructed_experts_is_the_same_forward():
    """moe_forward with experts reconstructed beforehand (the CPU baseline's
    timing split) gives the identical result: the same weights, the same loop."""
    src = synth.tiny_layer(seed=4)
    x = synth.tokens(src, 40, seed=4)
    ids, _, _ = oracle.route(src, x)
    y0 = oracle.moe_forward(src, x)
    part = oracle.reconstruct(src, ids[:, 0])          # some experts only: the rest on demand
    assert np.array_equal(oracle.moe_forward(src, x, experts=part), y0)
    full = oracle.reconstruct(src, np.arange(src.n_experts))
    assert np.array_equal(oracle.moe_forward(src, x, experts=full), y0)
