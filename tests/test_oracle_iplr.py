"""Pins of the oracle's Comba-iplr variant (table of state transitions for the
Comba variants): the transition alpha_t (I - 2 btilde_t k_t k_t^T) with
btilde_t = b beta_t, eigenvalues in (-1, 1) for unit keys."""
import numpy as np

import oracle


def _problem(seed, T=12, dk=4, dv=3, alpha_lo=0.6):
    rng = np.random.default_rng(seed)
    k = rng.standard_normal((T, 1, dk))
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    return dict(q=rng.standard_normal((T, 1, dk)), k=k, v=rng.standard_normal((T, 1, dv)),
                alpha=rng.uniform(alpha_lo, 1.0, (T, 1)), beta=rng.uniform(0.1, 1.0, (T, 1)),
                b=rng.uniform(0.2, 0.9, 1), d=rng.uniform(-1, 1, 1), h0=0.3 * rng.standard_normal((1, 1, dk, dv)))


def test_iplr_equals_explicit_transition_products():
    p = _problem(1)
    o, hT = oracle.fwd(variant="iplr", **p)
    dk = p["k"].shape[-1]
    S = p["h0"][0, 0].T
    for t in range(p["k"].shape[0]):
        kt, a = p["k"][t, 0], p["alpha"][t, 0]
        bt = p["b"][0] * p["beta"][t, 0]
        Phi = a * (np.eye(dk) - 2.0 * bt * np.outer(kt, kt))
        S = S @ Phi + p["beta"][t, 0] * np.outer(p["v"][t, 0], kt)
        np.testing.assert_allclose(o[t, 0], S @ (p["q"][t, 0] - p["d"][0] * kt), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(hT[0, 0], S.T, rtol=1e-10, atol=1e-12)


def test_iplr_at_half_decay_is_splr():
    """alpha = 1/2: alpha (I - 2 btilde k k^T) = alpha I - btilde k k^T, the SPLR transition."""
    p = _problem(2, T=70)
    p["alpha"] = np.full_like(p["alpha"], 0.5)
    rng = np.random.default_rng(3)
    dO = rng.standard_normal(p["v"].shape)
    dhT = rng.standard_normal(p["h0"].shape)
    oi, hi = oracle.fwd(variant="iplr", **p)
    os_, hs = oracle.fwd(**p)
    np.testing.assert_allclose(oi, os_, rtol=1e-13, atol=1e-14)
    np.testing.assert_allclose(hi, hs, rtol=1e-13, atol=1e-14)
    gi = oracle.bwd(dO=dO, dhT=dhT, variant="iplr", **p)
    gs = oracle.bwd(dO=dO, dhT=dhT, **p)
    # every gradient but dalpha agrees (iplr's btilde' = 2 alpha b beta also depends on alpha)
    for key in ("dq", "dk", "dv", "dbeta", "db", "dd", "dh0"):
        np.testing.assert_allclose(gi[key], gs[key], rtol=1e-11, atol=1e-12, err_msg=key)


def test_iplr_gradients_match_finite_differences():
    p = _problem(4, T=70)
    rng = np.random.default_rng(5)
    dO = rng.standard_normal(p["v"].shape)
    dhT = rng.standard_normal(p["h0"].shape)
    g = oracle.bwd(dO=dO, dhT=dhT, threads=1, variant="iplr", **p)

    def loss():
        o, hT = oracle.fwd(threads=1, variant="iplr", **p)
        return float(np.sum(o * dO) + np.sum(hT * dhT))

    names = {"q": "dq", "k": "dk", "v": "dv", "alpha": "dalpha", "beta": "dbeta", "b": "db", "d": "dd", "h0": "dh0"}
    for name, gname in names.items():
        flat = p[name].reshape(-1)
        for i in rng.choice(flat.size, size=min(flat.size, 8), replace=False):
            old = flat[i]
            flat[i] = old + 1e-6
            lp = loss()
            flat[i] = old - 1e-6
            lm = loss()
            flat[i] = old
            fd = (lp - lm) / 2e-6
            an = g[gname].reshape(-1)[i]
            assert abs(fd - an) <= 2e-6 * max(1.0, abs(an)), (name, fd, an)


def test_iplr_transition_spectrum_in_open_unit_interval():
    rng = np.random.default_rng(6)
    for _ in range(200):
        dk = int(rng.integers(2, 9))
        k = rng.standard_normal(dk)
        k /= np.linalg.norm(k)
        a, bt = rng.uniform(0.01, 0.999), rng.uniform(0.0, 0.999)
        lam = np.linalg.eigvalsh(a * (np.eye(dk) - 2 * bt * np.outer(k, k)))
        assert np.all(lam > -1.0) and np.all(lam < 1.0)
        np.testing.assert_allclose(sorted(lam), sorted([a * (1 - 2 * bt)] + [a] * (dk - 1)), atol=1e-12)


def test_iplr_decode_steps_equal_forward():
    p = _problem(7, T=6)
    o, hT = oracle.fwd(variant="iplr", **p)
    st = p["h0"]
    for t in range(6):
        ot, st = oracle.step(p["q"][t:t + 1], p["k"][t:t + 1], p["v"][t:t + 1], p["alpha"][t:t + 1],
                             p["beta"][t:t + 1], p["b"], p["d"], st, variant="iplr")
        np.testing.assert_allclose(ot[0], o[t], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(st, hT, rtol=1e-11, atol=1e-12)


def test_iplr_differs_from_splr():
    p = _problem(8)
    oi, _ = oracle.fwd(variant="iplr", **p)
    os_, _ = oracle.fwd(**p)
    assert np.abs(oi - os_).max() > 1e-3


def test_dropping_the_iplr_decay_gradient_term_is_caught(tmp_path):
    """A planted mistake (dalpha without the term from btilde' = 2 alpha b beta) fails the FD pin."""
    src = oracle.source_text()
    line = "if (J->variant == 1) J->dalpha[(size_t)t * Hh + h] -= 2.0 * bh * be * xde;"
    assert line in src
    lib = oracle.load_variant(oracle.build_variant(src.replace(line, ""), str(tmp_path)))
    p = _problem(9, T=40)
    rng = np.random.default_rng(10)
    dO = rng.standard_normal(p["v"].shape)
    g = oracle.bwd(dO=dO, threads=1, lib=lib, variant="iplr", **p)
    i = 7
    flat = p["alpha"].reshape(-1)
    old = flat[i]
    flat[i] = old + 1e-6
    lp = float(np.sum(oracle.fwd(threads=1, lib=lib, variant="iplr", **p)[0] * dO))
    flat[i] = old - 1e-6
    lm = float(np.sum(oracle.fwd(threads=1, lib=lib, variant="iplr", **p)[0] * dO))
    flat[i] = old
    fd = (lp - lm) / 2e-6
    assert abs(fd - g["dalpha"].reshape(-1)[i]) > 1e-4 * max(1.0, abs(fd))
