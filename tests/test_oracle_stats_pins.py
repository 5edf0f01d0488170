"""Pins of the router-statistics oracle (oracle/stats.py) against an
independent formulation (one-hot matrix products in torch), brute force over
token subsets, and the closed forms of NPMI (independence 0, exclusion -1,
complete co-occurrence +1)."""
import itertools

import numpy as np
import torch

from oracle import stats

import synth
import oracle


def _onehot_counts(ids, E):
    """coact = M^T M with M the [T, E] 0/1 selection matrix (a matmul)."""
    T = ids.shape[0]
    M = torch.zeros(T, E, dtype=torch.float64)
    for t in range(T):
        for e in ids[t]:
            if 0 <= e < E:
                M[t, int(e)] = 1.0
    C = (M.T @ M).numpy()
    return M.sum(0).numpy(), C


def test_counts_equal_onehot_gram():
    rng = np.random.default_rng(0)
    E, T, k = 24, 300, 5
    ids = np.stack([rng.choice(E, k, replace=False) for _ in range(T)]).astype(np.int32)
    fire, C = stats.coact_counts(ids, E)
    f2, C2 = _onehot_counts(ids, E)
    assert np.array_equal(fire.astype(np.float64), f2)
    assert np.array_equal(C.astype(np.float64), C2)
    assert np.array_equal(C, C.T)
    assert np.array_equal(np.diag(C), fire)
    assert int(fire.sum()) == T * k


def test_counts_brute_force_with_invalid_and_repeated_ids():
    ids = np.array([[0, 2, -1], [2, 2, 1], [3, 5, 0], [7, 1, 2]], np.int32)  # 5, 7 out of range
    E = 4
    fire, C = stats.coact_counts(ids, E)
    for i, j in itertools.product(range(E), repeat=2):
        want = sum(1 for row in ids if i in set(row) and j in set(row))
        assert int(C[i, j]) == want
    assert list(fire) == [2, 2, 3, 1]


def test_npmi_closed_forms():
    # 4 tokens: expert 0 on tokens {0,1}, expert 1 on {0,2} (independent:
    # p01 = 1/4 = p0 p1), expert 2 on {0,1} (always with 0), expert 3 on {3}
    # (never with 0), expert 4 on every token (p = 1), expert 5 never fires.
    ids = np.array([[0, 1, 2, 4], [0, 2, 4, -1], [1, 4, -1, -1], [3, 4, -1, -1]], np.int32)
    fire, C = stats.coact_counts(ids, 6)
    M = stats.npmi(C, 4)
    assert M[0, 1] == 0.0 and M[1, 0] == 0.0                      # independence
    assert abs(M[0, 2] - 1.0) < 1e-15                              # complete co-occurrence
    assert M[0, 3] == -1.0 and M[3, 0] == -1.0                     # exclusion
    assert M[4, 4] == 1.0                                          # p = 1
    assert M[5, 5] == -1.0 and M[5, 0] == -1.0                     # never fires
    for i in range(4):
        assert abs(M[i, i] - 1.0) < 1e-15
    # a textbook value: p_ij = 1/4, p_i = 1/2, p_j = 3/4 -> ln(2/3) / ln 4
    assert abs(M[0, 1] - 0.0) == 0.0
    assert abs(M[1, 4] - (np.log((2 / 4) / ((2 / 4) * 1.0)) / -np.log(2 / 4))) < 1e-15
    ids2 = np.array([[0, 1], [0, 2], [1, 2], [1, 3]], np.int32)
    _, C2 = stats.coact_counts(ids2, 4)
    assert abs(stats.npmi(C2, 4)[0, 1] - np.log((1 / 4) / ((2 / 4) * (3 / 4))) / np.log(4)) < 1e-15


def test_npmi_symmetric_and_bounded_on_routing():
    # d_model 2048 gives router logits of the paper's scale (std ~0.9)
    layer = synth.flat_layer(2048, 16, [4] * 8, 8, 4, "f32", seed=3, skew=(1.1, 0.6, 0.95, 2))
    x = synth.tokens(layer, 400, seed=1)
    ids, _, _ = oracle.route(layer, x)
    _, C = stats.coact_counts(ids, layer.n_experts)
    M = stats.npmi(C, 400)
    assert np.allclose(M, M.T, rtol=0, atol=0)
    assert np.all(M >= -1.0) and np.all(M <= 1.0 + 1e-15)
    # the skewed router co-selects cluster members: in-cluster NPMI is higher
    cl = layer.meta["clusters"]
    within = np.mean([M[i, j] for g in cl for i in g for j in g if i != j])
    across = np.mean([M[i, j] for a in range(len(cl)) for b in range(len(cl)) if a != b
                      for i in cl[a] for j in cl[b]])
    assert within > across


# planted mistakes in the statistics oracle must fail a pin
def _mut_unnormalised(coact, n_tokens):
    E = coact.shape[0]
    out = np.full((E, E), -1.0)
    for i in range(E):
        for j in range(E):
            if coact[i, j]:
                out[i, j] = np.log((coact[i, j] / n_tokens) /
                                   ((coact[i, i] / n_tokens) * (coact[j, j] / n_tokens)))
    return out


def _mut_no_dedupe(ids, E):
    fire = np.zeros(E, np.uint64)
    coact = np.zeros((E, E), np.uint64)
    for row in ids:
        sel = [int(e) for e in row if 0 <= int(e) < E]
        for i in sel:
            fire[i] += 1
            for j in sel:
                coact[i, j] += 1
    return fire, coact


def _mut_upper_only(ids, E):
    fire, C = _orig["coact_counts"](ids, E)
    return fire, np.triu(C)


_orig = {}


def _stats_pins_pass():
    try:
        test_counts_equal_onehot_gram()
        test_counts_brute_force_with_invalid_and_repeated_ids()
        test_npmi_closed_forms()
    except AssertionError:
        return False
    return True


import pytest  # noqa: E402


@pytest.mark.parametrize("target,mutant", [("npmi", _mut_unnormalised),
                                           ("coact_counts", _mut_no_dedupe),
                                           ("coact_counts", _mut_upper_only)])
def test_planted_stats_mistakes_fail_a_pin(monkeypatch, target, mutant):
    assert _stats_pins_pass()
    _orig["coact_counts"] = stats.coact_counts
    monkeypatch.setattr(stats, target, mutant)
    assert not _stats_pins_pass()
