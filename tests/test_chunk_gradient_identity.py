"""The chunk backward's dA identity, checked in fp64 on the host (no GPU, no library code).

Within a chunk (section 3.2, Eq. "prepare WY_M"), with M = (I + A)^{-1},
U = M Diag(beta) V, W = M Diag(s) F (s_r = btilde_r gamma_{r-1}; F = K, or Comba-pk's
P) and E = U - W H for the chunk's starting state H, a loss that depends on the chunk
through E has

    dL/dA = -M^T dM M^T,   dM = dE (Diag(beta) V)^T + dW (Diag(s) F)^T,   dW = -dE H^T,

and M^T dM M^T = (M^T dE) U^T + (M^T dW) W^T = (M^T dE) (U - W H)^T = (M^T dE) E^T.
Both local-gradient kernels form dA from that last product.  The tests check the
identity and check dL/dA against central finite differences of L = <dE, E(A)>.
"""
import numpy as np


def _chunk(seed, C=16, dk=8, dv=6):
    rng = np.random.default_rng(seed)
    F = rng.standard_normal((C, dk)) / np.sqrt(dk)
    V = rng.standard_normal((C, dv))
    H = rng.standard_normal((dk, dv)) * 0.5
    beta = rng.uniform(0.1, 0.9, C)
    s = rng.uniform(0.2, 1.0, C)
    A = np.tril(rng.standard_normal((C, C)) * 0.3, -1)   # strictly lower, like the chunk's A
    dE = rng.standard_normal((C, dv))
    return F, V, H, beta, s, A, dE


def _E(A, F, V, H, beta, s):
    M = np.linalg.inv(np.eye(A.shape[0]) + A)
    U = M @ np.diag(beta) @ V
    W = M @ np.diag(s) @ F
    return M, U, W, U - W @ H


def test_mt_dm_mt_equals_mt_de_e_transposed():
    for seed in range(5):
        F, V, H, beta, s, A, dE = _chunk(seed)
        M, U, W, E = _E(A, F, V, H, beta, s)
        dW = -dE @ H.T
        dM = dE @ (np.diag(beta) @ V).T + dW @ (np.diag(s) @ F).T
        lhs = M.T @ dM @ M.T
        assert np.allclose(lhs, (M.T @ dE) @ U.T + (M.T @ dW) @ W.T, rtol=0, atol=1e-12)
        assert np.allclose(lhs, (M.T @ dE) @ E.T, rtol=0, atol=1e-12)


def test_da_matches_finite_differences():
    """dL/dA_ij for L = <dE, E(A)> on the strict lower triangle equals -((M^T dE) E^T)_ij."""
    F, V, H, beta, s, A, dE = _chunk(11)
    M, U, W, E = _E(A, F, V, H, beta, s)
    dA = -((M.T @ dE) @ E.T)
    h = 1e-6
    C = A.shape[0]
    worst = 0.0
    for i in range(1, C):
        for j in range(i):
            Ap, Am = A.copy(), A.copy()
            Ap[i, j] += h
            Am[i, j] -= h
            fd = (np.sum(dE * _E(Ap, F, V, H, beta, s)[3]) - np.sum(dE * _E(Am, F, V, H, beta, s)[3])) / (2 * h)
            worst = max(worst, abs(fd - dA[i, j]) / max(1.0, abs(fd)))
    assert worst < 1e-7, worst


def test_identity_needs_the_state_term():
    """Dropping the W term of dM (a plausible mistake) breaks the identity."""
    F, V, H, beta, s, A, dE = _chunk(3)
    M, U, W, E = _E(A, F, V, H, beta, s)
    dM_wrong = dE @ (np.diag(beta) @ V).T
    assert not np.allclose(M.T @ dM_wrong @ M.T, (M.T @ dE) @ E.T, atol=1e-6)
