"""Pins of the neuron-alignment oracle (oracle/align.py): the expanded form of
Eq. cost via an independent matrix product, brute-force assignment (Eq. assign)
on tiny problems, recovery of a planted permutation (after which the residual
W_m^P - W_dom vanishes, Sec. 3.2 Stage 3), and invariance of the expert's
function under the permutation.  A mutation test plants mistakes."""
import itertools

import numpy as np
import pytest
import torch

import oracle
from oracle import align


def _expert(rng, H, I, std=0.02):
    return (rng.standard_normal((I, H)) * std, rng.standard_normal((I, H)) * std,
            rng.standard_normal((H, I)) * std)


def _vectors_by_loops(g, u, d):
    I, H = g.shape
    A = np.zeros((I, 3 * H))
    for i in range(I):
        for h in range(H):
            A[i, h] = g[i, h]
            A[i, H + h] = u[i, h]
            A[i, 2 * H + h] = d[h, i]
    return A


def test_cost_equals_expanded_form():
    """||a - b||^2 = ||a||^2 + ||b||^2 - 2 a.b (Eq. cost), the right side from
    a torch matrix product of independently assembled neuron vectors."""
    rng = np.random.default_rng(0)
    H, I = 12, 20
    dom, mem = _expert(rng, H, I), _expert(rng, H, I)
    A = torch.from_numpy(_vectors_by_loops(*dom))
    B = torch.from_numpy(_vectors_by_loops(*mem))
    ref = (A * A).sum(1)[:, None] + (B * B).sum(1)[None, :] - 2.0 * (A @ B.T)
    C = align.cost_matrix(dom, mem)
    assert np.max(np.abs(C - ref.numpy())) <= 1e-12 * np.max(np.abs(ref.numpy()))


@pytest.mark.parametrize("n,seed", [(1, 0), (3, 1), (5, 2), (7, 3), (7, 4)])
def test_assignment_brute_force(n, seed):
    rng = np.random.default_rng(seed)
    C = rng.random((n, n))
    if seed == 4:
        C = np.round(C * 3)  # many ties
    best = min(sum(C[i, p[i]] for i in range(n)) for p in itertools.permutations(range(n)))
    P = align.assign(C)
    assert sorted(P.tolist()) == list(range(n))
    assert abs(align.assignment_cost(C, P) - best) <= 1e-12


def test_planted_permutation_recovered_and_residual_vanishes():
    rng = np.random.default_rng(5)
    H, I = 16, 24
    dom = _expert(rng, H, I)
    sigma = rng.permutation(I)                        # member neuron j = dominant neuron sigma[j]
    mem = (dom[0][sigma], dom[1][sigma], dom[2][:, sigma])
    noisy = tuple(w + rng.standard_normal(w.shape) * 1e-4 for w in mem)
    P = align.assign(align.cost_matrix(dom, noisy))
    inv = np.empty(I, np.int64)
    inv[sigma] = np.arange(I)
    assert np.array_equal(P, inv)                     # dominant neuron i <- member neuron sigma^-1(i)
    aligned = align.permute_expert(*mem, P)
    for p in range(3):
        assert np.array_equal(aligned[p], dom[p])     # W_m^P - W_dom = 0
    # before alignment the residual is large (full rank in general)
    assert np.linalg.matrix_rank(mem[0] - dom[0]) == min(H, I)


def test_permutation_preserves_the_expert_function():
    rng = np.random.default_rng(6)
    H, I = 16, 24
    g, u, d = _expert(rng, H, I, std=0.3)
    P = rng.permutation(I).astype(np.int32)
    gp, up_, dp = align.permute_expert(g, u, d, P)
    x = rng.standard_normal((9, H))
    y0 = oracle.expert_output(g, u, d, x)
    y1 = oracle.expert_output(gp, up_, dp, x)
    assert np.max(np.abs(y0 - y1)) <= 1e-14 * np.max(np.abs(y0))
    assert not np.array_equal(gp, g)


# ----------------------------------------------------------------------------
# planted mistakes must fail a pin
# ----------------------------------------------------------------------------
def _mut_no_down(gate, up, down):
    return np.concatenate([np.asarray(gate, np.float64), np.asarray(up, np.float64)], axis=1)


def _mut_down_rows(gate, up, down):
    g = np.asarray(gate, np.float64)
    d = np.asarray(down, np.float64).reshape(g.shape[0], -1)  # down read row-wise
    return np.concatenate([g, np.asarray(up, np.float64), d], axis=1)


def _mut_inverse_assign(C):
    P = _orig["assign"](C)
    inv = np.empty_like(P)
    inv[P] = np.arange(len(P), dtype=P.dtype)
    return inv


def _mut_permute_down_rows(gate, up, down, P):
    P = np.asarray(P, np.int64)
    d = np.asarray(down)
    return np.asarray(gate)[P], np.asarray(up)[P], d[P % d.shape[0]]


_orig = {}


def _align_pins_pass():
    try:
        test_cost_equals_expanded_form()
        test_planted_permutation_recovered_and_residual_vanishes()
        test_permutation_preserves_the_expert_function()
        for n, s in [(5, 2), (7, 4)]:
            test_assignment_brute_force(n, s)
    except (AssertionError, ValueError, IndexError):
        return False
    return True


@pytest.mark.parametrize("target,mutant", [("neuron_vectors", _mut_no_down),
                                           ("neuron_vectors", _mut_down_rows),
                                           ("assign", _mut_inverse_assign),
                                           ("permute_expert", _mut_permute_down_rows)])
def test_planted_align_mistakes_fail_a_pin(monkeypatch, target, mutant):
    assert _align_pins_pass()
    _orig["assign"] = align.assign
    monkeypatch.setattr(align, target, mutant)
    assert not _align_pins_pass()
