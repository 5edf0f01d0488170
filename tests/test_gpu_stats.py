"""GPU parity of the router profiling statistics (lx_coact_accumulate,
lx_coact_npmi) against the CPU oracle (oracle/stats.py), through the C ABI.

Bar: firing and co-activation counts bit-exact (integers); NPMI within 1e-12
absolute (both sides evaluate the same float64 expression; only the last bits
of the natural logarithm may differ).  Ids are drawn by a seeded generator with
the method's structure (Zipf-skewed, cluster-correlated top-k sets) plus
invalid and repeated ids; both the shared-memory (E <= 256) and the
global-atomic (E > 256) kernels are covered.
"""
import numpy as np
import pytest
import torch

import oracle
import synth
from oracle import stats
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu


def _ids(T, k, E, seed, invalid=0.0, repeats=0.0):
    """Zipf(1.1)-skewed top-k sets of distinct ids, then a fraction of entries
    replaced by out-of-range ids or by a repeat of the row's first id."""
    rng = np.random.default_rng(seed)
    p = 1.0 / np.arange(1, E + 1) ** 1.1
    p /= p.sum()
    perm = rng.permutation(E)
    k_eff = min(k, E)
    ids = np.stack([perm[rng.choice(E, k_eff, replace=False, p=p)] for _ in range(T)])
    if k_eff < k:
        ids = np.concatenate([ids, np.full((T, k - k_eff), -1)], axis=1)
    m = rng.random(ids.shape)
    ids = np.where(m < invalid, rng.choice([-1, E, E + 7, 1 << 30], size=ids.shape), ids)
    rep = rng.random(T) < repeats
    if k > 1:
        ids[rep, k - 1] = ids[rep, 0]
    return np.ascontiguousarray(ids.astype(np.int32))


def _u64(t):
    return t.cpu().numpy().astype(np.uint64)


@pytest.mark.parametrize("E,k,T", [(8, 2, 1), (8, 2, 257), (128, 8, 37), (128, 8, 5000),
                                   (256, 8, 3001), (256, 32, 600), (257, 8, 999),
                                   (1024, 8, 2000), (1, 1, 10), (64, 1, 100)])
def test_counts_bit_exact(E, k, T):
    ids = _ids(T, k, E, seed=E * 31 + k + T, invalid=0.02, repeats=0.05)
    fire, coact = lx.coact_accumulate(torch.from_numpy(ids).cuda(), E)
    torch.cuda.synchronize()
    f_ref, c_ref = stats.coact_counts(ids, E)
    assert np.array_equal(_u64(fire), f_ref)
    assert np.array_equal(_u64(coact), c_ref)


@pytest.mark.parametrize("E", [128, 512])
def test_batches_accumulate(E):
    """Counts add over calls (a calibration set streamed batch by batch)."""
    batches = [_ids(T, 8, E, seed=100 + T) for T in (1, 64, 2048, 333)]
    fire = torch.zeros(E, dtype=torch.int64, device="cuda")
    coact = torch.zeros((E, E), dtype=torch.int64, device="cuda")
    for b in batches:
        lx.coact_accumulate(torch.from_numpy(b).cuda(), E, fire, coact)
    torch.cuda.synchronize()
    f_ref, c_ref = stats.coact_counts(np.concatenate(batches), E)
    assert np.array_equal(_u64(fire), f_ref)
    assert np.array_equal(_u64(coact), c_ref)


def test_fire_only_and_coact_only():
    E, ids = 96, _ids(700, 8, 96, seed=5)
    d = torch.from_numpy(ids).cuda()
    fire = torch.zeros(E, dtype=torch.int64, device="cuda")
    coact = torch.zeros((E, E), dtype=torch.int64, device="cuda")
    st = lx.lib().lx_coact_accumulate(lx._ptr(d), 700, 8, E, lx._ptr(fire), None, None)
    assert st == lx.LX_OK
    st = lx.lib().lx_coact_accumulate(lx._ptr(d), 700, 8, E, None, lx._ptr(coact), None)
    assert st == lx.LX_OK
    torch.cuda.synchronize()
    f_ref, c_ref = stats.coact_counts(ids, E)
    assert np.array_equal(_u64(fire), f_ref) and np.array_equal(_u64(coact), c_ref)


def test_routing_of_the_decode_layer():
    """Counts of the oracle's routing of the Qwen3-30B-A3B-shaped layer (the
    routing the paper profiles in Stage 1), and the NPMI matrix of them."""
    src = synth.qwen_decode_layer()
    x = synth.tokens(src, 2048, seed=21)
    ids, _, _ = oracle.route(src, x, 8)
    fire, coact = lx.coact_accumulate(torch.from_numpy(ids).cuda(), 128)
    torch.cuda.synchronize()
    f_ref, c_ref = stats.coact_counts(ids, 128)
    assert np.array_equal(_u64(fire), f_ref) and np.array_equal(_u64(coact), c_ref)
    ref = stats.npmi(c_ref, 2048)
    got = lx.coact_npmi(torch.from_numpy(c_ref.astype(np.int64)).cuda(), 2048)
    torch.cuda.synchronize()
    assert np.max(np.abs(got.cpu().numpy() - ref)) <= 1e-12


@pytest.mark.parametrize("E,T", [(6, 4), (256, 3000), (1024, 500)])
def test_npmi(E, T):
    ids = _ids(T, 8 if E > 8 else 3, E, seed=E + T)
    _, c_ref = stats.coact_counts(ids, E)
    ref = stats.npmi(c_ref, T)
    got = lx.coact_npmi(torch.from_numpy(c_ref.astype(np.int64)).cuda(), T)
    torch.cuda.synchronize()
    assert np.max(np.abs(got.cpu().numpy() - ref)) <= 1e-12


def test_empty_and_rejected_calls():
    E = 16
    fire = torch.zeros(E, dtype=torch.int64, device="cuda")
    assert lx.lib().lx_coact_accumulate(None, 0, 4, E, lx._ptr(fire), None, None) == lx.LX_OK
    assert int(fire.sum()) == 0
    L = lx.lib()
    assert L.lx_coact_accumulate(None, 4, 4, E, lx._ptr(fire), None, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(lx._ptr(fire), 4, 0, E, lx._ptr(fire), None, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(lx._ptr(fire), 4, 4, 0, lx._ptr(fire), None, None) == lx.LX_ERR_ARG
    assert L.lx_coact_accumulate(lx._ptr(fire), 4, 4, E, None, None, None) == lx.LX_ERR_ARG
    assert L.lx_coact_npmi(None, E, 4, None, None) == lx.LX_ERR_ARG
