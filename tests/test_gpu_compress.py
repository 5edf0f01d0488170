"""GPU parity of the member compression (lx_compress_factor) against the CPU
oracle (oracle/compress.py), through the C ABI, on the same residual and the
same Gaussian test matrix.

Bar, derived from the arithmetic (fp32 products, Cholesky factors and Jacobi
rotations; float64 Gram sums and Rayleigh quotients; the same subspaces as the
oracle's float64 algorithm, so only rounding separates the two):
  * the rank-r approximation U V^T within 1e-4 of max|U_ref V_ref^T|;
  * singular values within 1e-5 of the largest;
  * ||R - U V^T||_F within 1e-5 (relative) of the oracle's;
  * the split of Eq. factors: U^T U = V^T V = diag(s) within 1e-4 of s_0;
  * the sign rule: every column's largest-magnitude entry of U is positive.
Residuals: independent N(0, 0.02) experts (a flat spectrum, the Qwen3-30B-A3B
projection shapes), a decaying spectrum, an exactly rank-5 residual (recovered
exactly), a zero residual (the dominant compressed against itself gives zero
factors), and an odd l.
"""
import ctypes

import numpy as np
import pytest
import torch

import synth
from oracle import compress
from paper_2608_07814_gb300 import lx

pytestmark = pytest.mark.gpu


def _residual_pair(rows, cols, kind, dtype, rng):
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
    else:  # zero
        Wm = Wd.copy()
    return synth.to_storage(Wd, dtype), synth.to_storage(Wm, dtype)


CASES = [  # rows, cols, dtype, r, l, power_iters, kind
    (768, 2048, "bf16", 128, 136, 2, "flat"),
    (2048, 768, "bf16", 128, 136, 2, "flat"),
    (1536, 2560, "bf16", 64, 72, 2, "flat"),
    (192, 256, "f32", 32, 40, 2, "decay"),
    (96, 64, "f32", 16, 24, 1, "rank5"),
    (64, 64, "f32", 8, 16, 1, "zero"),
    (136, 200, "bf16", 20, 21, 0, "flat"),
    (256, 192, "bf16", 192, 192, 1, "decay"),
    (256, 320, "bf16", 200, 256, 1, "decay"),   # l = 256: 128 column pairs per round
]


@pytest.mark.parametrize("rows,cols,dtype,r,l,q,kind", CASES)
def test_compress_factor(rows, cols, dtype, r, l, q, kind):
    rng = np.random.default_rng(rows * 7 + cols + r)
    Wd, Wm = _residual_pair(rows, cols, kind, dtype, rng)
    omega = rng.standard_normal((cols, l)).astype(np.float32)
    R = compress.residual(synth.from_storage(Wd, dtype), synth.from_storage(Wm, dtype))
    Uo, Vo, so = compress.randomized_factors(R, r, omega.astype(np.float64), q)
    dev = lambda a: lx.host_to_torch(a, dtype).cuda()
    U, V, s = lx.compress_factor(dev(Wd), dev(Wm), torch.from_numpy(omega).cuda(), r, q)
    torch.cuda.synchronize()
    U = U.cpu().numpy().astype(np.float64)
    V = V.cpu().numpy().astype(np.float64)
    s = s.cpu().numpy().astype(np.float64)
    assert np.all(np.isfinite(U)) and np.all(np.isfinite(V)) and np.all(np.isfinite(s))
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
    nz = s > 1e-6 * s[0]
    assert np.max(np.abs((U.T @ U - np.diag(s))[np.ix_(nz, nz)])) <= 1e-4 * s[0]
    assert np.max(np.abs((V.T @ V - np.diag(s))[np.ix_(nz, nz)])) <= 1e-4 * s[0]
    top = U[np.argmax(np.abs(U), axis=0), np.arange(r)]
    assert np.all(top[nz] > 0)


def test_workspace_query_and_rejects():
    assert lx.compress_workspace_bytes(768, 2048, 136, 128) > 0
    L = lx.lib()
    b = ctypes.c_uint64()
    assert L.lx_compress_workspace(768, 2048, 257, 128, b) == lx.LX_ERR_SHAPE   # l > 256
    assert L.lx_compress_workspace(768, 2048, 100, 128, b) == lx.LX_ERR_SHAPE   # l < r
    assert L.lx_compress_workspace(770, 2048, 136, 128, b) == lx.LX_ERR_SHAPE   # rows % 8
    w = torch.zeros((64, 64), dtype=torch.float32, device="cuda")
    om = torch.zeros((64, 16), dtype=torch.float32, device="cuda")
    small = torch.zeros(256, dtype=torch.uint8, device="cuda")
    p = lx._ptr
    assert L.lx_compress_factor(lx.LX_F32, 64, 64, p(w), p(w), p(om), 16, 8, 1, p(w), p(w),
                                p(w), p(small), 256, None) == lx.LX_ERR_ARG    # workspace
    assert L.lx_compress_factor(lx.LX_F32, 64, 64, p(w), p(w), p(om), 16, 8, 99, p(w), p(w),
                                p(w), p(small), 256, None) == lx.LX_ERR_ARG    # power_iters


def test_member_projections_concurrent_same_bits():
    """lx.compress_member runs a member's gate, up and down projections on three
    streams; each projection's kernels are the same, so its factors equal, bit
    for bit, those of the projections run one after another."""
    rng = np.random.default_rng(99)
    shapes = [(384, 512), (384, 512), (512, 384)]
    r, l, q = 48, 56, 2
    doms, mems, oms = [], [], []
    for rows, cols in shapes:
        Wd, Wm = _residual_pair(rows, cols, "flat", "bf16", rng)
        doms.append(lx.host_to_torch(Wd, "bf16").cuda())
        mems.append(lx.host_to_torch(Wm, "bf16").cuda())
        oms.append(torch.from_numpy(rng.standard_normal((cols, l)).astype(np.float32)).cuda())
    seq = [lx.compress_factor(doms[j], mems[j], oms[j], r, q) for j in range(3)]
    conc = lx.compress_member(doms, mems, oms, r, q)
    torch.cuda.synchronize()
    for a, b in zip(seq, conc):
        for x, y in zip(a, b):
            assert torch.equal(x, y)
