"""The chunk's UT inverse M = (I + A)^{-1} (section 3.2, Eq. "prepare WY_M") as prep computes it,
emulated on the host.

Prep forms M in three levels: the four 16 x 16 diagonal blocks by fp32 forward substitution,
then in both 32 x 32 halves M10 = -M11 (A10 M00), then M21 = -M22 (A21 M11) for the 64 x 64
matrix, the two off-diagonal levels as tile products whose operands are rounded to tf32
(round to nearest, ties away from zero, 10 mantissa bits: the PTX conversion cvt.rna.tf32.f32)
with fp32 accumulation.  These tests check

* the block algebra: run in fp64, the three levels give exactly the inverse;
* the precision: in fp32 with tf32 operands, on chunks shaped like the benchmark workloads
  (unit-norm keys at d = 128, sigmoid input gates, decays exp(-0.1 softplus(x))), M's error is
  at most half the error of rounding the exact M to bf16, which every product that uses M
  takes; at feedback strength up to 2 (Comba-iplr's 2 alpha b beta) as well.
"""
import numpy as np
import pytest

C = 64


def _tf32(x):
    u = np.asarray(x, np.float32).view(np.uint32)
    return ((u + np.uint32(0x1000)) & np.uint32(0xFFFFE000)).view(np.float32)


def _bf16(x):
    u = np.asarray(x, np.float32).view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000          # round to nearest even at bit 16
    return u.astype(np.uint32).view(np.float32)


def _blocked_inverse(A, fp32=True, sign=-1.0):
    """The three-level inverse of I + A for a strictly lower 64 x 64 A."""
    dt = np.float32 if fp32 else np.float64
    A = A.astype(dt)
    M = np.zeros((C, C), dt)
    for o in range(0, C, 16):                  # level 0: column j of each diagonal block's inverse
        for j in range(16):
            s = np.zeros(16, dt)
            for r in range(16):
                x = dt(1) if r == j else (dt(0) if r < j else -s[r])
                M[o + r, o + j] = x
                s = (s + A[o:o + 16, o + r] * x).astype(dt)

    def mm(X, Y):
        if fp32:
            X, Y = _tf32(X), _tf32(Y)
        return (X.astype(np.float64) @ Y.astype(np.float64)).astype(dt)

    for o in (0, 32):                          # level 1: both 32 x 32 halves
        T = mm(A[o + 16:o + 32, o:o + 16], M[o:o + 16, o:o + 16])
        M[o + 16:o + 32, o:o + 16] = sign * mm(M[o + 16:o + 32, o + 16:o + 32], T)
    T = mm(A[32:64, 0:32], M[0:32, 0:32])      # level 2
    M[32:64, 0:32] = sign * mm(M[32:64, 32:64], T)
    return M


def _chunk_A(rng, strength=1.0, dk=128):
    k = rng.standard_normal((C, dk))
    k /= np.linalg.norm(k, axis=1, keepdims=True)
    alpha = np.exp(-0.1 * np.log1p(np.exp(rng.standard_normal(C))))
    beta = 1.0 / (1.0 + np.exp(-rng.standard_normal(C)))
    g = np.cumsum(np.log(alpha))
    gm1 = np.concatenate([[0.0], g[:-1]])
    ii, jj = np.indices((C, C))
    D = np.where(ii > jj, np.exp(np.where(ii > jj, gm1[:, None] - g[None, :], 0.0)), 0.0)
    return np.tril(strength * beta[:, None] * D * (k @ k.T), -1)


def test_block_algebra_is_the_inverse():
    rng = np.random.default_rng(5)
    for _ in range(4):
        A = _chunk_A(rng, strength=rng.uniform(0.5, 2.0))
        M = _blocked_inverse(A, fp32=False)
        assert np.allclose(M @ (np.eye(C) + A), np.eye(C), rtol=0, atol=1e-13)
        assert np.allclose(M, np.linalg.inv(np.eye(C) + A), rtol=0, atol=1e-13)


def test_off_diagonal_sign_slip_is_caught():
    A = _chunk_A(np.random.default_rng(6))
    assert not np.allclose(_blocked_inverse(A, fp32=False, sign=1.0), np.linalg.inv(np.eye(C) + A), atol=1e-6)


@pytest.mark.parametrize("strength", [1.0, 2.0])
def test_tf32_levels_stay_below_the_bf16_rounding_of_m(strength):
    rng = np.random.default_rng(7 + int(strength))
    worst = {"max": [0.0, 0.0], "fro": [0.0, 0.0]}
    for _ in range(24):
        A = _chunk_A(rng, strength)
        exact = np.linalg.inv(np.eye(C) + A)
        for i, M in enumerate((_blocked_inverse(A).astype(np.float64),
                               _bf16(exact.astype(np.float32)).astype(np.float64))):
            worst["max"][i] = max(worst["max"][i], np.abs(M - exact).max() / np.abs(exact).max())
            worst["fro"][i] = max(worst["fro"][i], np.linalg.norm(M - exact) / np.linalg.norm(exact))
    for metric, (emulated, bf16) in worst.items():
        assert emulated <= 0.5 * bf16, (metric, emulated, bf16)
