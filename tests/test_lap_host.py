"""The library's exact assignment solver (lx_lap_solve, host code behind the C
ABI; Eq. assign) against SciPy's exact solver and brute force.  Runs without a
GPU."""
import itertools
import os

import numpy as np
import pytest

from oracle import align
from paper_2608_07814_gb300 import build as lxbuild
from paper_2608_07814_gb300 import lx


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not os.path.exists(lx.LIB_PATH):
        lxbuild.build()
    lx.lib()


@pytest.mark.parametrize("n,seed", [(1, 0), (2, 1), (4, 2), (6, 3), (7, 4), (7, 5)])
def test_brute_force(n, seed):
    rng = np.random.default_rng(seed)
    C = rng.random((n, n)).astype(np.float32)
    if seed == 5:
        C = np.round(C * 2).astype(np.float32)   # ties
    P, tot = lx.lap_solve(C)
    assert sorted(P.tolist()) == list(range(n))
    best = min(sum(float(C[i, p[i]]) for i in range(n)) for p in itertools.permutations(range(n)))
    assert abs(tot - best) <= 1e-9
    assert abs(align.assignment_cost(C, P) - tot) <= 1e-9


@pytest.mark.parametrize("n,kind", [(50, "uniform"), (200, "int"), (300, "neurons"),
                                    (768, "neurons")])
def test_matches_scipy_optimum(n, kind):
    rng = np.random.default_rng(n)
    if kind == "uniform":
        C = rng.random((n, n)).astype(np.float32)
    elif kind == "int":
        C = rng.integers(0, 10, (n, n)).astype(np.float32)   # heavy ties
    else:
        # squared distances of neuron vectors, a planted permutation plus noise
        H = 32
        A = rng.standard_normal((n, 3 * H))
        sigma = rng.permutation(n)
        B = A[sigma] + 0.3 * rng.standard_normal((n, 3 * H))
        C = ((A * A).sum(1)[:, None] + (B * B).sum(1)[None, :] - 2.0 * A @ B.T).astype(np.float32)
    P, tot = lx.lap_solve(C)
    assert sorted(P.tolist()) == list(range(n))
    ref = align.assignment_cost(C, align.assign(C))
    assert abs(tot - ref) <= 1e-9 * max(1.0, abs(ref))
    if kind == "neurons" and n == 300:
        inv = np.empty(n, np.int64)
        inv[sigma] = np.arange(n)
        assert np.array_equal(P, inv)


def test_negative_costs_and_rejects():
    C = -np.arange(16, dtype=np.float32).reshape(4, 4)
    P, tot = lx.lap_solve(C)
    assert abs(tot - align.assignment_cost(C, align.assign(C))) <= 1e-9
    bad = C.copy()
    bad[1, 2] = np.nan
    with pytest.raises(lx.LxError):
        lx.lap_solve(bad)
    bad[1, 2] = np.inf
    with pytest.raises(lx.LxError):
        lx.lap_solve(bad)


def test_batch_matches_single_solves_on_threads():
    rng = np.random.default_rng(11)
    n, count = 120, 9
    costs = rng.random((count, n, n)).astype(np.float32)
    costs[3] = np.round(costs[3] * 3)          # ties in one problem
    P, tot = lx.lap_solve_batch(costs, threads=4)
    for b in range(count):
        Pb, tb = lx.lap_solve(costs[b])
        assert abs(tot[b] - tb) <= 1e-9 * max(1.0, abs(tb))
        assert sorted(P[b].tolist()) == list(range(n))
        ref = align.assignment_cost(costs[b], align.assign(costs[b]))
        assert abs(tot[b] - ref) <= 1e-9 * max(1.0, abs(ref))
    bad = costs.copy()
    bad[7, 1, 1] = np.nan
    with pytest.raises(lx.LxError):
        lx.lap_solve_batch(bad)
    P0, t0 = lx.lap_solve_batch(costs[:0])
    assert P0.shape == (0, n)


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_optimum_on_adversarial_families(seed):
    """Ties, constant matrices, identical rows, negative and large costs,
    rank-one and squared-distance costs: the optimum equals SciPy's."""
    rng = np.random.default_rng(100 + seed)
    for n in list(range(1, 10)) * 4 + [17, 40]:
        for kind in range(8):
            if kind == 0:
                C = rng.random((n, n))
            elif kind == 1:
                C = rng.integers(0, 3, (n, n))
            elif kind == 2:
                C = np.full((n, n), 7.0)
            elif kind == 3:
                C = np.tile(rng.random(n), (n, 1))
            elif kind == 4:
                C = -rng.random((n, n)) * 1e3
            elif kind == 5:
                C = rng.random((n, n)) * 1e6 - 5e5
            elif kind == 6:
                a, b = rng.standard_normal((n, 5)), rng.standard_normal((n, 5))
                C = (a * a).sum(1)[:, None] + (b * b).sum(1)[None, :] - 2 * a @ b.T
            else:
                C = np.outer(rng.random(n), rng.random(n))
            C = C.astype(np.float32)
            P, tot = lx.lap_solve(C)
            assert sorted(P.tolist()) == list(range(n))
            ref = align.assignment_cost(C, align.assign(C))
            assert abs(align.assignment_cost(C, P) - ref) <= 1e-9 * max(1.0, abs(ref))
