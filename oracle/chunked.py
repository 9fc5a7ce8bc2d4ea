"""The paper's chunk-wise Comba algorithm in plain fp64 NumPy (test infrastructure only).

Section 3.2 ("Comba with Chunk-wise Parallel") states the chunk form; this
module follows it step by step, in the paper's orientation S (dv x dk), so
that tests can check that the paper's chunk equations, under this package's
reading of their notation, reproduce the token recurrence of ``comba_oracle.c``.

Readings of the notation (the paper's subscripts are garbled in places):
  * positions inside a chunk are r = 1..L (L <= C; the last chunk of a
    sequence may be short); gamma_r = prod_{j=1..r} alpha_j, gamma_0 = 1
    (the paper's alpha^{1:r});
  * the decay matrix with entries alpha^{1:i}/alpha^{1:j} is gamma_i/gamma_j,
    and the one written with (i-1)/j is gamma_{i-1}/gamma_j;
  * "lower" in the inverse (Eq. "prepare WY_M") is strictly lower, while
    "Tril" in the output equation keeps the diagonal;
  * alpha^{0 -> C-1} is (gamma_0, ..., gamma_{C-1}) and alpha^{i -> C} is
    gamma_C / gamma_i;
  * btilde = b * beta (section 3.1), Q~ = Q - d K;
  * Comba-pk (appendix B.3): with feedback vectors P the Gram inside the
    inverse is P K^T, W = M Diag(btilde * alpha^{0->C-1}) P and Q~ = Q - d P;
    U, the state update and the output keep K.

The unit-lower-triangular inverse is taken with ``numpy.linalg.solve`` (a
library primitive standing in for the paper's forward substitution).
"""
from __future__ import annotations

import numpy as np


def chunk_forward_unit(q, k, v, alpha, beta, b, d, C, S0=None, p=None):
    """One (sequence, head): q,k [T,dk], v [T,dv], alpha,beta [T], scalars b,d; optional
    Comba-pk feedback vectors p [T,dk] (default k).

    Returns ``(O [T,dv], S_T [dv,dk])`` computed chunk by chunk with chunk size C.
    """
    q, k, v, alpha, beta = (np.asarray(x, np.float64) for x in (q, k, v, alpha, beta))
    p = k if p is None else np.asarray(p, np.float64)
    T, dk = k.shape
    dv = v.shape[1]
    S = np.zeros((dv, dk)) if S0 is None else np.array(S0, np.float64)
    O = np.zeros((T, dv))
    for c0 in range(0, T, C):
        c1 = min(c0 + C, T)
        L = c1 - c0
        K, V, Q, P = k[c0:c1], v[c0:c1], q[c0:c1], p[c0:c1]
        a, be = alpha[c0:c1], beta[c0:c1]
        bt = b * be                                   # btilde (section 3.1)
        gam = np.cumprod(a)                           # gamma_1..gamma_L
        gam0 = np.concatenate([[1.0], gam[:-1]])      # gamma_0..gamma_{L-1}
        Qt = Q - d * P                                # Q~ = Q - Diag(d) P  (P = K unless pk)
        # Eq. "prepare WY_M": M = (I + lower(Diag(btilde)(A^{(i-1)/j} * P K^T)))^{-1}
        Aim1_j = gam0[:, None] / gam[None, :]         # gamma_{i-1} / gamma_j
        low = np.tril(np.diag(bt) @ (Aim1_j * (P @ K.T)), -1)
        M = np.linalg.solve(np.eye(L) + low, np.eye(L))
        W = M @ np.diag(bt * gam0) @ P                # W = M Diag(btilde * alpha^{0->C-1}) P
        U = M @ np.diag(be) @ V                       # U = M Diag(beta) V
        Vn = U - W @ S.T                              # "pseudo"-value term U - W S^T
        Ai_j = gam[:, None] / gam[None, :]            # gamma_i / gamma_j
        O[c0:c1] = np.diag(gam) @ Qt @ S.T + np.tril(Qt @ K.T * Ai_j) @ Vn
        S = gam[-1] * S + Vn.T @ np.diag(gam[-1] / gam) @ K
    return O, S


def chunk_forward(q, k, v, alpha, beta, b, d, C, h0=None, cu_seqlens=None, p=None):
    """Packed/dense driver with the same layouts as ``oracle.fwd``; returns ``(o, hT)``.

    ``hT`` is returned in the ABI orientation H = S^T, [N, H, dk, dv].
    """
    q, k, v, alpha, beta = (np.asarray(x, np.float64) for x in (q, k, v, alpha, beta))
    p = k if p is None else np.asarray(p, np.float64)
    batched = q.ndim == 4
    if batched:
        B, T, H, _ = q.shape
        cu = np.arange(B + 1) * T
        q, k, v, p = (x.reshape(B * T, H, x.shape[-1]) for x in (q, k, v, p))
        alpha, beta = alpha.reshape(B * T, H), beta.reshape(B * T, H)
    else:
        H = q.shape[1]
        cu = np.array([0, q.shape[0]]) if cu_seqlens is None else np.asarray(cu_seqlens)
    N = len(cu) - 1
    dk, dv = k.shape[-1], v.shape[-1]
    o = np.zeros((q.shape[0], H, dv))
    hT = np.zeros((N, H, dk, dv))
    for n in range(N):
        t0, t1 = int(cu[n]), int(cu[n + 1])
        for h in range(H):
            S0 = None if h0 is None else np.asarray(h0, np.float64)[n, h].T
            bh = 1.0 if b is None else float(b[h])
            O, S = chunk_forward_unit(q[t0:t1, h], k[t0:t1, h], v[t0:t1, h], alpha[t0:t1, h], beta[t0:t1, h],
                                      bh, float(d[h]), C, S0, p=p[t0:t1, h])
            o[t0:t1, h] = O
            hT[n, h] = S.T
    if batched:
        o = o.reshape(B, T, H, dv)
    return o, hT
