"""The compression kernels' orthonormalisation schedule, emulated in fp32 on
the CPU, meets the GPU parity bars against the oracle.

lx_compress_factor differs from the oracle's plain definition in how it
orthonormalises: CholeskyQR (the Gram, an fp32 Cholesky with pivots floored at
1e-30 and a 1e-6 relative shift in the first pass, then X L^-T) instead of a
Householder QR, run twice for the final bases Q and Z and once for the
intermediate bases of the power iterations, whose span is all the next product
uses; and the small SVD of Bs = M Z2^T through the triangular factor
M = L1 L2 of Z.  This test runs that schedule in float32 numpy -- the products
with R in fp32 (the tensor cores reproduce them to fp32 accuracy), the Gram
summed in float64 and rounded (as the compensated device Gram is), the small
SVD of M in float64 (the one-sided Jacobi reaches it to fp32 accuracy) -- on
the residual families of the GPU test, with that test's bars.  It shares no
code with the CUDA library: it pins the schedule, not the kernels.
"""
import numpy as np
import pytest

from oracle import compress

F32 = np.float32


def _chol_floored(A):
    """fp32 right-looking Cholesky, pivots floored at 1e-30 (as the kernel)."""
    A = A.astype(F32).copy()
    n = A.shape[0]
    L = np.zeros_like(A)
    for j in range(n):
        d = np.sqrt(max(A[j, j], F32(1e-30)))
        L[j, j] = d
        col = A[j + 1:, j] / d
        L[j + 1:, j] = col
        A[j + 1:, j + 1:] -= np.outer(col, col).astype(F32)
    return L


def _pass(X, shift_rel):
    """One CholeskyQR pass: (X L^-T, L); a zero Gram gives zeros."""
    G = X.astype(np.float64).T @ X.astype(np.float64)
    md = G.diagonal().max()
    l = X.shape[1]
    if not md > 0:
        return np.zeros_like(X), np.zeros((l, l), F32)
    A = G.astype(F32) + F32(shift_rel * md) * np.eye(l, dtype=F32)
    L = _chol_floored(A)
    Linv = np.linalg.inv(L.astype(np.float64)).astype(F32)
    return (X @ Linv.T).astype(F32), L


def _orth1(X):
    return _pass(X, 1e-6)


def _orth2(X):
    X1, L1 = _pass(X, 1e-6)
    X2, L2 = _pass(X1, 0.0)
    return X2, L1, L2


def device_schedule(R, r, omega, q):
    """The kernels' schedule in fp32 numpy: (U, V, s) with the split of Eq. factors."""
    R = R.astype(F32)
    Y = (R @ omega.astype(F32)).astype(F32)
    if q == 0:
        Q, _, _ = _orth2(Y)
    else:
        Q, _ = _orth1(Y)
    for it in range(q):
        Z, _ = _orth1((R.T @ Q).astype(F32))
        Y = (R @ Z).astype(F32)
        if it + 1 == q:
            Q, _, _ = _orth2(Y)
        else:
            Q, _ = _orth1(Y)
    Z2, L1, L2 = _orth2((R.T @ Q).astype(F32))
    M = L1.astype(np.float64) @ L2.astype(np.float64)  # Bs = Q^T R = M Z2^T
    Um, S, Wt = np.linalg.svd(M)
    keep = (S > 1e-6 * S[0]) & (S > 0) if S[0] > 0 else np.zeros_like(S, bool)
    sq = np.where(keep, np.sqrt(S), 0.0)[:r]
    U = Q.astype(np.float64) @ Um[:, :r] * sq
    V = Z2.astype(np.float64) @ Wt.T[:, :r] * sq
    top = U[np.argmax(np.abs(U), axis=0), np.arange(r)]
    sgn = np.where(top < 0, -1.0, 1.0)
    return U * sgn, V * sgn, np.where(keep, S, 0.0)[:r]


def _pair(rows, cols, kind, rng):
    draw = lambda s: rng.standard_normal(s).astype(np.float32) * np.float32(0.02)
    Wd = draw((rows, cols))
    if kind == "flat":
        Wm = draw((rows, cols))
    elif kind == "decay":
        n = min(rows, cols)
        Uq, _ = np.linalg.qr(rng.standard_normal((rows, n)))
        Vq, _ = np.linalg.qr(rng.standard_normal((cols, n)))
        Wm = Wd + ((Uq * (0.9 ** np.arange(n))) @ Vq.T * 0.05).astype(np.float32)
    elif kind == "rank5":
        Wm = Wd + (rng.standard_normal((rows, 5)) @ rng.standard_normal((5, cols)) *
                   0.01).astype(np.float32)
    else:
        Wm = Wd.copy()
    return Wd, Wm


CASES = [  # rows, cols, r, l, power_iters, kind (the GPU test's families)
    (768, 2048, 128, 136, 2, "flat"),
    (2048, 768, 128, 136, 2, "flat"),
    (192, 256, 32, 40, 2, "decay"),
    (96, 64, 16, 24, 1, "rank5"),
    (64, 64, 8, 16, 1, "zero"),
    (136, 200, 20, 21, 0, "flat"),
]
# Decaying spectra with l at (or near) the full rank: the first, shifted pass
# leaves directions far below sqrt(fp32 eps), and the Gram of the second,
# unshifted pass has a condition number of 3e8 (l = 192) and 7e14 (l = 256),
# beyond fp32's 1 / eps; in this emulation's fp32
# rounding a pivot goes non-positive there and the factorization breaks down
# (the kernel's own rounding stays positive on these inputs: the GPU test
# passes them).  Kept as strict expected failures to document the margin.
_EDGE = "unshifted second CholeskyQR pass beyond fp32 (Gram condition 3e8 to 7e14)"
CASES += [
    pytest.param(256, 192, 192, 192, 1, "decay", marks=pytest.mark.xfail(strict=True, reason=_EDGE)),
    pytest.param(256, 320, 200, 256, 1, "decay", marks=pytest.mark.xfail(strict=True, reason=_EDGE)),
]


@pytest.mark.filterwarnings("ignore::RuntimeWarning")
@pytest.mark.parametrize("rows,cols,r,l,q,kind", CASES)
def test_device_schedule_meets_the_gpu_bars(rows, cols, r, l, q, kind):
    rng = np.random.default_rng(rows * 7 + cols + r)
    Wd, Wm = _pair(rows, cols, kind, rng)
    omega = rng.standard_normal((cols, l)).astype(np.float32)
    R = compress.residual(Wd, Wm)
    Uo, Vo, so = compress.randomized_factors(R, r, omega.astype(np.float64), q)
    U, V, s = device_schedule(R, r, omega, q)
    P, Po = U @ V.T, Uo @ Vo.T
    if kind == "zero":
        assert np.all(U == 0) and np.all(V == 0) and np.all(s == 0)
        return
    assert np.max(np.abs(P - Po)) <= 1e-4 * np.max(np.abs(Po))
    assert np.max(np.abs(s - so)) <= 1e-5 * so[0]
    e, eo = np.linalg.norm(R - P), np.linalg.norm(R - Po)
    assert abs(e - eo) <= 1e-5 * np.linalg.norm(R) + 1e-6 * eo
    if kind == "rank5":
        assert e <= 1e-5 * np.linalg.norm(R)
