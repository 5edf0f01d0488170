"""CPU oracle for the compression of one member (Sec. 3.2 Stage 3 (ii)).

TEST INFRASTRUCTURE ONLY (like the rest of ``oracle``): imported by the tests,
``__graft_entry__.smoke()`` and the CPU-baseline legs of ``bench.py``.

For one projection of an aligned member, the residual ``R = W_m^P - W_dom``
([out, in], Eq. svd) is approximated at rank r by a randomized SVD, and the
singular values are split symmetrically between the two factors (Eq. factors):
``B_m = U_r S_r^(1/2)``, ``A_m = S_r^(1/2) V_r^T``; stored here as ``U = B_m``
([out, r]) and ``V = A_m^T`` ([in, r]).

The randomized solver is the range finder with power iterations of Halko,
Martinsson and Tropp (2011), with the Gaussian test matrix ``Omega`` [in, l]
(l = r + oversampling) passed in:

1. ``Y = R Omega``;  ``Q = orth(Y)``;
2. q times:  ``Q = orth(R (orth(R^T Q)))``  (power iterations);
3. ``Bs = Q^T R`` [l, in] and its SVD ``Bs = Ut S Vt`` (a library SVD of the
   small matrix);  ``U = Q Ut``;
4. keep the r largest singular triplets; sign of each left singular vector
   fixed so that its largest-magnitude entry is positive.

``orth`` is a library QR (numpy, float64).  Everything is float64.  Pinned by
``tests/test_oracle_compress_pins.py``.
"""
from __future__ import annotations

import numpy as np

__all__ = ["residual", "randomized_factors", "truncated_factors"]


def residual(W_dom, W_mem) -> np.ndarray:
    return np.asarray(W_mem, np.float64) - np.asarray(W_dom, np.float64)


def _orth(Y: np.ndarray) -> np.ndarray:
    Q, _ = np.linalg.qr(Y)
    return Q


def _split(U: np.ndarray, S: np.ndarray, Vt: np.ndarray, r: int):
    U, S, Vt = U[:, :r], S[:r], Vt[:r]
    sgn = np.sign(U[np.argmax(np.abs(U), axis=0), np.arange(U.shape[1])])
    sgn[sgn == 0] = 1.0
    U = U * sgn
    V = Vt.T * sgn
    sq = np.sqrt(S)
    return U * sq, V * sq, S


def randomized_factors(R: np.ndarray, r: int, omega: np.ndarray, power_iters: int = 2):
    """(U [out, r], V [in, r], s [r]) with U V^T ~ R (symmetric split)."""
    R = np.asarray(R, np.float64)
    Om = np.asarray(omega, np.float64)
    assert Om.shape[0] == R.shape[1] and Om.shape[1] >= r
    Q = _orth(R @ Om)
    for _ in range(power_iters):
        Z = _orth(R.T @ Q)
        Q = _orth(R @ Z)
    Bs = Q.T @ R
    Ut, S, Vt = np.linalg.svd(Bs, full_matrices=False)
    return _split(Q @ Ut, S, Vt, r)


def truncated_factors(R: np.ndarray, r: int):
    """The exact rank-r truncated SVD with the same split and sign rule."""
    U, S, Vt = np.linalg.svd(np.asarray(R, np.float64), full_matrices=False)
    return _split(U, S, Vt, r)
