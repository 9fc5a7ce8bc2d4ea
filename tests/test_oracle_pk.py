"""Pins of the oracle's Comba-pk form (appendix B.3): a per-token feedback vector p_t replaces
k_t where the state is read back (x_t = H_{t-1}^T p_t) and in the output correction
(q_t - d p_t); k_t still writes the state.  Transition on S: alpha_t I - btilde_t p_t k_t^T."""
import numpy as np
import pytest

import oracle
from oracle import chunked


def _problem(seed, T=70, H=2, dk=5, dv=4, B=1):
    rng = np.random.default_rng(seed)

    def unit(shape):
        x = rng.standard_normal(shape)
        return x / np.linalg.norm(x, axis=-1, keepdims=True)

    return dict(q=rng.standard_normal((B, T, H, dk)), k=unit((B, T, H, dk)), v=rng.standard_normal((B, T, H, dv)),
                alpha=rng.uniform(0.6, 1.0, (B, T, H)), beta=rng.uniform(0.1, 1.0, (B, T, H)),
                b=rng.uniform(0.2, 0.9, H), d=rng.uniform(-1, 1, H), h0=0.3 * rng.standard_normal((B, H, dk, dv)),
                p=unit((B, T, H, dk)))


@pytest.mark.parametrize("variant", ["splr", "iplr"])
def test_p_equal_to_k_is_the_plain_form(variant):
    """p = k: every output equals the form without p; dk + dp there is dk here."""
    pr = _problem(1)
    pr["p"] = pr["k"].copy()
    rng = np.random.default_rng(2)
    dO, dhT = rng.standard_normal(pr["v"].shape), rng.standard_normal(pr["h0"].shape)
    base = {k_: v_ for k_, v_ in pr.items() if k_ != "p"}
    o1, h1 = oracle.fwd(**pr, variant=variant)
    o0, h0 = oracle.fwd(**base, variant=variant)
    np.testing.assert_allclose(o1, o0, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(h1, h0, rtol=1e-12, atol=1e-13)
    g1 = oracle.bwd(**pr, dO=dO, dhT=dhT, variant=variant)
    g0 = oracle.bwd(**base, dO=dO, dhT=dhT, variant=variant)
    for key in ("dq", "dv", "dalpha", "dbeta", "db", "dd", "dh0"):
        np.testing.assert_allclose(g1[key], g0[key], rtol=1e-11, atol=1e-12, err_msg=key)
    np.testing.assert_allclose(g1["dk"] + g1["dp"], g0["dk"], rtol=1e-11, atol=1e-12)


def test_p_proportional_to_k_rescales_b_and_d():
    """p = c k is the plain form with b' = c b and d' = c d (the paper's p = b k reading)."""
    pr = _problem(3)
    c = 0.7
    pr["p"] = c * pr["k"]
    rng = np.random.default_rng(4)
    dO, dhT = rng.standard_normal(pr["v"].shape), rng.standard_normal(pr["h0"].shape)
    base = {k_: v_ for k_, v_ in pr.items() if k_ != "p"}
    base["b"], base["d"] = c * pr["b"], c * pr["d"]
    o1, h1 = oracle.fwd(**pr)
    o0, h0 = oracle.fwd(**base)
    np.testing.assert_allclose(o1, o0, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(h1, h0, rtol=1e-12, atol=1e-13)
    g1 = oracle.bwd(**pr, dO=dO, dhT=dhT)
    g0 = oracle.bwd(**base, dO=dO, dhT=dhT)
    for key in ("dq", "dv", "dalpha", "dbeta", "dh0"):
        np.testing.assert_allclose(g1[key], g0[key], rtol=1e-11, atol=1e-12, err_msg=key)
    np.testing.assert_allclose(g1["dk"] + c * g1["dp"], g0["dk"], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(g1["db"], c * g0["db"], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(g1["dd"], c * g0["dd"], rtol=1e-11, atol=1e-12)


def test_transition_products():
    """The state after T tokens is the explicit product of alpha I - btilde p k^T plus the writes."""
    pr = _problem(5, T=15, H=1)
    o, hT = oracle.fwd(**pr)
    S = pr["h0"][0, 0].T
    for t in range(15):
        k, f = pr["k"][0, t, 0], pr["p"][0, t, 0]
        Phi = pr["alpha"][0, t, 0] * np.eye(5) - pr["b"][0] * pr["beta"][0, t, 0] * np.outer(f, k)
        S = S @ Phi + pr["beta"][0, t, 0] * np.outer(pr["v"][0, t, 0], k)
        np.testing.assert_allclose(o[0, t, 0], S @ (pr["q"][0, t, 0] - pr["d"][0] * f), rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(hT[0, 0], S.T, rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("C", [1, 4, 16, 64])
def test_chunk_equations_reproduce_the_recurrence(C):
    """The appendix's pk chunk form (Gram P K^T, W from P, Q~ = Q - d P) equals the recurrence,
    with ragged chunks and packed sequences."""
    pr = _problem(6, T=150, H=2)
    o, hT = oracle.fwd(**pr)
    oc, hTc = chunked.chunk_forward(C=C, **pr)
    np.testing.assert_allclose(oc, o, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(hTc, hT, rtol=1e-9, atol=1e-10)
    cu = np.array([0, 37, 37, 150], np.int64)
    flat = {k_: (v_.reshape((150,) + v_.shape[2:]) if k_ in ("q", "k", "v", "p", "alpha", "beta") else v_)
            for k_, v_ in pr.items() if k_ != "h0"}
    o2, hT2 = oracle.fwd(**flat, cu_seqlens=cu)
    oc2, hTc2 = chunked.chunk_forward(C=C, cu_seqlens=cu, **flat)
    np.testing.assert_allclose(oc2, o2, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(hTc2, hT2, rtol=1e-9, atol=1e-10)


@pytest.mark.parametrize("variant", ["splr", "iplr"])
def test_gradients_match_finite_differences(variant):
    pr = _problem(7, T=70)
    rng = np.random.default_rng(8)
    dO, dhT = rng.standard_normal(pr["v"].shape), rng.standard_normal(pr["h0"].shape)
    g = oracle.bwd(**pr, dO=dO, dhT=dhT, variant=variant, threads=1)

    def loss():
        o, hT = oracle.fwd(**pr, variant=variant, threads=1)
        return float(np.sum(o * dO) + np.sum(hT * dhT))

    names = {"q": "dq", "k": "dk", "v": "dv", "p": "dp", "alpha": "dalpha", "beta": "dbeta", "b": "db", "d": "dd",
             "h0": "dh0"}
    for name, gname in names.items():
        flat = pr[name].reshape(-1)
        for i in rng.choice(flat.size, size=min(flat.size, 8), replace=False):
            old = flat[i]
            flat[i] = old + 1e-6
            lp = loss()
            flat[i] = old - 1e-6
            lm = loss()
            flat[i] = old
            fd = (lp - lm) / 2e-6
            an = g[gname].reshape(-1)[i]
            assert abs(fd - an) <= 3e-6 * max(1.0, abs(an)), (variant, name, fd, an)


def test_decode_steps_equal_the_forward():
    pr = _problem(9, T=9, H=3)
    o, hT = oracle.fwd(**pr)
    st = pr["h0"]
    for t in range(9):
        sl = lambda x: x[:, t]
        ot, st = oracle.step(sl(pr["q"]), sl(pr["k"]), sl(pr["v"]), sl(pr["alpha"]), sl(pr["beta"]), pr["b"], pr["d"],
                             st, p=sl(pr["p"]))
        np.testing.assert_allclose(ot, o[:, t], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(st, hT, rtol=1e-11, atol=1e-12)
