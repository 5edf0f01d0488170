"""Pins of the compression oracle (oracle/compress.py): exact recovery of a
residual of rank <= r, the Eckart-Young optimum of the truncated SVD (Eq. svd),
the symmetric split of Eq. factors (B^T B = A A^T = diag(s)), agreement with
the exact truncated SVD when the spectrum has a gap, and the sign rule.  A
mutation test plants mistakes."""
import numpy as np
import pytest

from oracle import compress


def _omega(n, l, seed):
    return np.random.default_rng(seed).standard_normal((n, l))


def _decaying(out, inn, seed, decay=0.97):
    rng = np.random.default_rng(seed)
    U, _ = np.linalg.qr(rng.standard_normal((out, min(out, inn))))
    V, _ = np.linalg.qr(rng.standard_normal((inn, min(out, inn))))
    s = decay ** np.arange(min(out, inn))
    return (U * s) @ V.T, s


def test_low_rank_residual_recovered_exactly():
    rng = np.random.default_rng(0)
    out, inn, r = 96, 64, 12
    R = rng.standard_normal((out, 7)) @ rng.standard_normal((7, inn))   # rank 7 <= r
    U, V, s = compress.randomized_factors(R, r, _omega(inn, r + 8, 1), power_iters=1)
    assert np.max(np.abs(U @ V.T - R)) <= 1e-12 * np.max(np.abs(R))
    assert np.all(s[7:] <= 1e-12 * s[0])


def test_eckart_young_and_split():
    out, inn, r = 120, 80, 16
    R, sv = _decaying(out, inn, 2)
    U, V, s = compress.randomized_factors(R, r, _omega(inn, r + 8, 3), power_iters=2)
    err = np.linalg.norm(R - U @ V.T)
    opt = np.sqrt(np.sum(sv[r:] ** 2))                 # Eckart-Young
    assert opt * (1 - 1e-12) <= err <= 1.01 * opt
    assert np.allclose(U.T @ U, np.diag(s), atol=1e-12)   # B_m^T B_m = S_r
    assert np.allclose(V.T @ V, np.diag(s), atol=1e-12)   # A_m A_m^T = S_r
    # Ritz values of Q^T R interlace: never above the true singular values
    assert np.all(s <= sv[:r] * (1 + 1e-12)) and np.all(s >= 0.97 * sv[:r])


def test_matches_exact_truncated_svd_with_a_gap():
    out, inn, r = 64, 48, 8
    rng = np.random.default_rng(4)
    Uq, _ = np.linalg.qr(rng.standard_normal((out, inn)))
    Vq, _ = np.linalg.qr(rng.standard_normal((inn, inn)))
    sv = np.concatenate([np.linspace(10, 5, r), 1e-3 * np.linspace(1, 0.1, inn - r)])
    R = (Uq * sv) @ Vq.T
    U, V, s = compress.randomized_factors(R, r, _omega(inn, r + 6, 5), power_iters=2)
    Ue, Ve, se = np.linalg.svd(R)[0][:, :r], np.linalg.svd(R)[2][:r].T, np.linalg.svd(R)[1][:r]
    # sign rule: largest-magnitude entry of each left vector positive
    sg = np.sign(Ue[np.argmax(np.abs(Ue), axis=0), np.arange(r)])
    Ue, Ve = Ue * sg, Ve * sg
    assert np.allclose(U, Ue * np.sqrt(se), atol=1e-8)
    assert np.allclose(V, Ve * np.sqrt(se), atol=1e-8)
    assert np.all(U[np.argmax(np.abs(U), axis=0), np.arange(r)] > 0)


def test_truncated_factors_full_rank_reconstruct():
    rng = np.random.default_rng(6)
    R = rng.standard_normal((20, 12))
    U, V, s = compress.truncated_factors(R, 12)
    assert np.max(np.abs(U @ V.T - R)) <= 1e-13 * np.max(np.abs(R))


# ----------------------------------------------------------------------------
def _mut_no_sqrt_split(U, S, Vt, r):
    U, S, Vt = U[:, :r], S[:r], Vt[:r]
    return U * S, Vt.T, S


def _mut_no_power(R, r, omega, power_iters=2):
    return _orig["rf"](R, r, omega, 0)


def _mut_smallest(U, S, Vt, r):
    return _orig["split"](U[:, ::-1], S[::-1], Vt[::-1], r)


_orig = {}


def _pins_pass():
    try:
        test_low_rank_residual_recovered_exactly()
        test_eckart_young_and_split()
        test_matches_exact_truncated_svd_with_a_gap()
    except AssertionError:
        return False
    return True


@pytest.mark.parametrize("target,mutant", [("_split", _mut_no_sqrt_split),
                                           ("randomized_factors", _mut_no_power),
                                           ("_split", _mut_smallest)])
def test_planted_compress_mistakes_fail_a_pin(monkeypatch, target, mutant):
    assert _pins_pass()
    _orig["rf"] = compress.randomized_factors
    _orig["split"] = compress._split
    monkeypatch.setattr(compress, target, mutant)
    assert not _pins_pass()
