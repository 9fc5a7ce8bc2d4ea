"""Gate and normalisation prologue around the recurrence, fp64 (test infrastructure only).

Section 3.1's gates and the neural-architecture section's normalisation, as the
steps on either side of the chunk recurrence:

    q_hat = q / sqrt(|q|^2 + eps),  k_hat = k / sqrt(|k|^2 + eps)     (L2 norm per token and head)
    alpha = exp(-a softplus(g_alpha + c))                            (forget gate, "close to 1")
    beta  = sigmoid(g_beta)                                          (input gate)
    b     = sigmoid(b_raw)                                           (feedback strength btilde = b beta)

with per-head trainable scalars a, c, b_raw (and d, unchanged); g_alpha and
g_beta are the gate pre-activations (the projections W x are outside).  The
forward then runs the oracle recurrence on (q_hat, k_hat, v, alpha, beta, b,
d); the backward maps its gradients back through these definitions by the
chain rule.  Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU legs of
``bench.py`` use this module.
"""
from __future__ import annotations

import numpy as np

from . import bwd as _bwd
from . import fwd as _fwd

EPS = 1e-6


def softplus(x):
    return np.logaddexp(0.0, x)


def sigmoid(x):
    """1 / (1 + e^-x), evaluated on the side where the exponential does not overflow."""
    x = np.asarray(x, np.float64)
    e = np.exp(-np.abs(x))
    return np.where(x >= 0, 1.0 / (1.0 + e), e / (1.0 + e))


def prologue(q, k, g_alpha, g_beta, a, c, b_raw, eps=EPS):
    """(q_hat, k_hat, alpha, beta, b) from the raw inputs (fp64)."""
    q, k, g_alpha, g_beta = (np.asarray(x, np.float64) for x in (q, k, g_alpha, g_beta))
    a, c, b_raw = (np.asarray(x, np.float64) for x in (a, c, b_raw))
    nq = np.sqrt(np.sum(q * q, axis=-1, keepdims=True) + eps)
    nk = np.sqrt(np.sum(k * k, axis=-1, keepdims=True) + eps)
    alpha = np.exp(-a * softplus(g_alpha + c))
    beta = sigmoid(g_beta)
    return q / nq, k / nk, alpha, beta, sigmoid(b_raw)


def fwd(q, k, v, g_alpha, g_beta, a, c, b_raw, d, h0=None, cu_seqlens=None, variant="splr", eps=EPS):
    qh, kh, alpha, beta, b = prologue(q, k, g_alpha, g_beta, a, c, b_raw, eps)
    return _fwd(qh, kh, v, alpha, beta, b, d, h0=h0, cu_seqlens=cu_seqlens, variant=variant)


def bwd(q, k, v, g_alpha, g_beta, a, c, b_raw, d, dO, h0=None, dhT=None, cu_seqlens=None, variant="splr",
        eps=EPS):
    """Gradients w.r.t. every raw input: dq, dk, dv, dg_alpha, dg_beta, da, dc, db_raw, dd, dh0."""
    q, k = (np.asarray(x, np.float64) for x in (q, k))
    qh, kh, alpha, beta, b = prologue(q, k, g_alpha, g_beta, a, c, b_raw, eps)
    g = _bwd(qh, kh, v, alpha, beta, b, d, dO, h0=h0, dhT=dhT, cu_seqlens=cu_seqlens, variant=variant)
    nq = np.sqrt(np.sum(q * q, axis=-1, keepdims=True) + eps)
    nk = np.sqrt(np.sum(k * k, axis=-1, keepdims=True) + eps)
    # x_hat = x / n(x), n = sqrt(|x|^2 + eps):  dx = (dx_hat - x_hat (x_hat . dx_hat)) / n
    dq = (g["dq"] - qh * np.sum(qh * g["dq"], axis=-1, keepdims=True)) / nq
    dk = (g["dk"] - kh * np.sum(kh * g["dk"], axis=-1, keepdims=True)) / nk
    z = np.asarray(g_alpha, np.float64) + np.asarray(c, np.float64)
    a64 = np.asarray(a, np.float64)
    # alpha = exp(-a softplus(z)):  d alpha / d z = -a alpha sigmoid(z),  d alpha / d a = -alpha softplus(z)
    dg_alpha = g["dalpha"] * (-a64 * alpha * sigmoid(z))
    lead = tuple(range(dg_alpha.ndim - 1))
    da = np.sum(g["dalpha"] * (-alpha * softplus(z)), axis=lead)
    dc = np.sum(dg_alpha, axis=lead)
    dg_beta = g["dbeta"] * beta * (1.0 - beta)
    db_raw = g["db"] * b * (1.0 - b)
    return {"dq": dq, "dk": dk, "dv": g["dv"], "dg_alpha": dg_alpha, "dg_beta": dg_beta, "da": da, "dc": dc,
            "db_raw": db_raw, "dd": g["dd"], "dh0": g["dh0"]}
