"""Structure of the seeded workload generators (CPU): the node tables that the
parity tests and the bench rely on."""
import numpy as np

import synth


def test_binary_tree_layout_and_signs():
    L = synth.binary_tree_layer(64, 32, 2, 3, [16, 8, 8], 4, "f32", seed=1, signed=True)
    assert L.n_experts == 2 * 8 and L.n_nodes == 2 + 2 * (2 + 4 + 8)
    paths = [L.path(e) for e in range(L.n_experts)]
    assert all(len(p) == 4 for p in paths)                       # leaf, two levels, root
    leaves = {p[0] for p in paths}
    assert len(leaves) == L.n_experts                            # every leaf is one expert
    for p in paths:
        assert [int(L.node_rank[n]) for n in p] == [8, 8, 16, 0]
        assert L.node_parent[p[-1]] == -1
    # no internal correction is an expert; anchors are not experts
    internal = {n for p in paths for n in p[1:-1]}
    assert not internal & set(int(n) for n in L.expert_node)
    # siblings carry -1 / +1; anchors +1
    assert np.all(L.node_sign[:2] == 1)
    for parent in range(L.n_nodes):
        kids = [n for n in range(L.n_nodes) if L.node_parent[n] == parent]
        if kids:
            assert sorted(int(L.node_sign[k]) for k in kids) == [-1, 1]
    assert synth.binary_tree_layer(64, 32, 2, 3, [16, 8, 8], 4, "f32", seed=1).node_sign is None


def test_single_base_layout():
    L = synth.single_base_layer(64, 32, 12, 8, 4, "f32", seed=2, skew=synth.QWEN_SKEW)
    assert L.n_nodes == 13 and L.node_parent[0] == -1 and L.node_rank[0] == 0
    assert not np.any(L.expert_node == 0)                        # the base is no expert
    assert all(L.path(e)[-1] == 0 and len(L.path(e)) == 2 for e in range(12))
    assert sorted(int(n) for n in L.expert_node) == list(range(1, 13))


def test_full_size_workloads_shapes():
    b = synth.binary_tree_layer(2048, 768, 16, 3, [128, 64, 64], 8, "bf16", seed=6,
                                signed=True, skew=synth.TREE_SKEW)
    assert b.n_experts == 128 and b.n_nodes == 16 + 16 * 14
    assert max(len(b.path(e)) for e in range(128)) == 4          # k * depth = 32 for top-8
    s = synth.single_base_layer(2048, 768, 128, 128, 8, "bf16", seed=7, skew=synth.QWEN_SKEW)
    assert s.n_nodes == 129 and s.weight_bytes() == 3 * 2048 * 768 * 2 + 128 * 3 * 128 * (2048 + 768) * 2


def test_generators_are_seeded():
    a = synth.binary_tree_layer(64, 32, 1, 2, [8, 8], 2, "bf16", seed=3, signed=True)
    b = synth.binary_tree_layer(64, 32, 1, 2, [8, 8], 2, "bf16", seed=3, signed=True)
    assert all(np.array_equal(x, y) for wa, wb in zip(a.node_w, b.node_w) for x, y in zip(wa, wb))
    assert np.array_equal(a.router_w, b.router_w)


def test_small_skewed_layers_route_through_corrections():
    """The Zipf router's dead experts (25 of 96 members at E = 128) are capped
    at a third of the members, so that a small layer made with the same skew
    still selects members: parity on it then exercises the corrections."""
    import oracle
    for src in (synth.flat_layer(512, 384, [4] * 8, 64, 8, "bf16", seed=13,
                                 factor_std="visible", skew=synth.QWEN_SKEW),
                synth.flat_layer(256, 192, [4, 4, 1, 3], 64, 4, "bf16", seed=1,
                                 skew=synth.QWEN_SKEW)):
        ids, _, _ = oracle.route(src, synth.tokens(src, 200, seed=5))
        via = np.mean([len(src.path(int(e))) > 1 for e in ids.ravel()])
        assert via > 0.3, via
    # the full-size layers keep their calibrated dead counts (96 and 224 members)
    assert synth._n_dead(25, 96) == 25 and synth._n_dead(50, 224) == 50
    assert synth._n_dead(25, 24) == 8
