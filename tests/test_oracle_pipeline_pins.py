"""The oracle's compression pipeline composes (CPU): members planted as
permuted dominants are aligned (oracle/align.py), their residuals compressed at
full rank (oracle/compress.py, Eq. svd / factors), the compressed layer run by
the oracle's forward, and the output equals the uncompressed MoE of the
original members -- alignment preserves each expert's function and full-rank
factors reproduce the aligned residual.  The same inputs drive the GPU
pipeline test."""
import importlib.util
import os

import numpy as np

import oracle
import synth
from oracle import align, compress

_spec = importlib.util.spec_from_file_location(
    "gpu_pipeline", os.path.join(os.path.dirname(__file__), "test_gpu_pipeline.py"))
gp = importlib.util.module_from_spec(_spec)
_spec.loader.exec_module(gp)


def test_oracle_pipeline_reproduces_the_dense_moe():
    dom, members, sigmas, router, omegas = gp.planted_members()
    r = min(gp.H, gp.I)
    factors = []
    for m, (mem, sigma) in enumerate(zip(members, sigmas)):
        P = align.assign(align.cost_matrix(dom, mem))
        inv = np.empty(gp.I, np.int64)
        inv[sigma] = np.arange(gp.I)
        assert np.array_equal(P, inv)
        aligned = align.permute_expert(*mem, P)
        fac = []
        for p in range(3):
            R = compress.residual(dom[p], aligned[p])
            U, V, s = compress.randomized_factors(R, r, omegas[m][p].astype(np.float64), 2)
            assert np.max(np.abs(U @ V.T - R)) <= 1e-10 * np.max(np.abs(R))
            fac += [U.astype(np.float32), V.astype(np.float32)]
        factors.append(tuple(fac))
    comp = gp.compressed_layer(dom, factors, router)
    dense = gp.dense_layer(dom, members, router)
    x = synth.tokens(comp, 96, seed=5)
    ids_c, g_c, _ = oracle.route(comp, x)
    ids_d, g_d, _ = oracle.route(dense, x)
    assert np.array_equal(ids_c, ids_d) and np.array_equal(g_c, g_d)   # router untouched
    y = oracle.moe_forward(comp, x)
    ref = oracle.moe_forward(dense, x)
    # fp32-stored factors: the only error is their rounding
    assert np.max(np.abs(y - ref)) <= 1e-5 * np.max(np.abs(ref))
    # and alignment mattered: the aligned residual is a fraction of the naive
    # one, which a rank-8 truncation would leave mostly unexplained
    P0 = align.assign(align.cost_matrix(dom, members[0]))
    R_un = compress.residual(dom[0], members[0][0])
    R_al = compress.residual(dom[0], align.permute_expert(*members[0], P0)[0])
    assert np.linalg.norm(R_al) < 0.5 * np.linalg.norm(R_un)
    U8, V8, _ = compress.randomized_factors(R_un, 8, omegas[0][0][:, :8].astype(np.float64), 2)
    assert np.linalg.norm(U8 @ V8.T - R_un) > 0.5 * np.linalg.norm(R_un)
