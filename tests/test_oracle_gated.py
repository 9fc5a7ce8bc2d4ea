"""Pins of the oracle's gate and normalisation prologue (section 3.1 gates, L2-normalised q and k)."""
import types

import numpy as np
import pytest

from oracle import gated


def _problem(seed, T=60, H=2, dk=5, dv=4):
    rng = np.random.default_rng(seed)
    return dict(q=rng.standard_normal((1, T, H, dk)), k=rng.standard_normal((1, T, H, dk)),
                v=rng.standard_normal((1, T, H, dv)), g_alpha=rng.standard_normal((1, T, H)),
                g_beta=rng.standard_normal((1, T, H)), a=rng.uniform(0.05, 0.3, H), c=rng.uniform(-1, 1, H),
                b_raw=rng.uniform(-1, 1, H), d=rng.uniform(-1, 1, H), h0=0.2 * rng.standard_normal((1, H, dk, dv)))


def test_gate_values_match_their_definitions():
    z = np.array([-30.0, -2.0, 0.0, 1.5, 30.0])
    np.testing.assert_allclose(gated.softplus(z), np.log1p(np.exp(z)), rtol=1e-12, atol=1e-300)
    np.testing.assert_allclose(gated.sigmoid(z), 1.0 / (1.0 + np.exp(-z)), rtol=1e-12)
    p = _problem(1)
    qh, kh, alpha, beta, b = gated.prologue(p["q"], p["k"], p["g_alpha"], p["g_beta"], p["a"], p["c"], p["b_raw"])
    assert np.all((alpha > 0) & (alpha < 1)) and np.all((beta > 0) & (beta < 1)) and np.all((b > 0) & (b < 1))
    # a = 0: no forgetting; unit-norm rows come out (to eps) unit norm
    _, _, a0, _, _ = gated.prologue(p["q"], p["k"], p["g_alpha"], p["g_beta"], 0 * p["a"], p["c"], p["b_raw"])
    np.testing.assert_array_equal(a0, 1.0)
    np.testing.assert_allclose(np.linalg.norm(qh, axis=-1), 1.0, atol=1e-5)
    np.testing.assert_allclose(np.linalg.norm(kh, axis=-1), 1.0, atol=1e-5)


def test_forward_is_invariant_to_key_and_query_scale():
    """L2 normalisation makes the output independent of positive rescaling of q and k (up to eps)."""
    p = _problem(2)
    o1, h1 = gated.fwd(**p, eps=0.0)
    p2 = dict(p, q=3.7 * p["q"], k=0.21 * p["k"])
    o2, h2 = gated.fwd(**p2, eps=0.0)
    np.testing.assert_allclose(o1, o2, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(h1, h2, rtol=1e-11, atol=1e-12)


def test_gated_gradients_match_finite_differences():
    _finite_difference_pin(gated)


def _finite_difference_pin(mod):
    for variant in ("splr", "iplr"):
        p = _problem(3)
        rng = np.random.default_rng(4)
        dO = rng.standard_normal(p["v"].shape)
        dhT = rng.standard_normal(p["h0"].shape)
        g = mod.bwd(**p, dO=dO, dhT=dhT, variant=variant)

        def loss():
            o, hT = mod.fwd(**p, variant=variant)
            return float(np.sum(o * dO) + np.sum(hT * dhT))

        names = {"q": "dq", "k": "dk", "v": "dv", "g_alpha": "dg_alpha", "g_beta": "dg_beta", "a": "da", "c": "dc",
                 "b_raw": "db_raw", "d": "dd", "h0": "dh0"}
        for name, gname in names.items():
            flat = p[name].reshape(-1)
            for i in rng.choice(flat.size, size=min(flat.size, 6), replace=False):
                old = flat[i]
                flat[i] = old + 1e-6
                lp = loss()
                flat[i] = old - 1e-6
                lm = loss()
                flat[i] = old
                fd = (lp - lm) / 2e-6
                an = g[gname].reshape(-1)[i]
                assert abs(fd - an) <= 3e-6 * max(1.0, abs(an)), (variant, name, fd, an)


# Planted mistakes in the prologue's backward, each a plausible slip of the chain rule.
SLIPS = {
    "l2norm_without_projection": ('dq = (g["dq"] - qh * np.sum(qh * g["dq"], axis=-1, keepdims=True)) / nq',
                                  'dq = g["dq"] / nq'),
    "forget_gate_without_a": ('dg_alpha = g["dalpha"] * (-a64 * alpha * sigmoid(z))',
                              'dg_alpha = g["dalpha"] * (-alpha * sigmoid(z))'),
    "da_with_sigmoid": ("(-alpha * softplus(z))", "(-alpha * sigmoid(z))"),
    "input_gate_derivative_truncated": ('dg_beta = g["dbeta"] * beta * (1.0 - beta)', 'dg_beta = g["dbeta"] * beta'),
    "dc_from_dalpha": ("dc = np.sum(dg_alpha, axis=lead)", 'dc = np.sum(g["dalpha"], axis=lead)'),
    "feedback_gate_derivative_dropped": ('db_raw = g["db"] * b * (1.0 - b)', 'db_raw = g["db"]'),
}


@pytest.mark.parametrize("name", sorted(SLIPS))
def test_planted_slip_in_the_prologue_backward_is_caught(name):
    old, new = SLIPS[name]
    with open(gated.__file__) as f:
        src = f.read()
    assert src.count(old) == 1, name
    src = src.replace("from . import bwd as _bwd", "from oracle import bwd as _bwd")
    src = src.replace("from . import fwd as _fwd", "from oracle import fwd as _fwd")
    ns = {"__name__": "gated_variant"}
    exec(compile(src.replace(old, new), "gated_variant", "exec"), ns)
    with pytest.raises(AssertionError):
        _finite_difference_pin(types.SimpleNamespace(fwd=ns["fwd"], bwd=ns["bwd"]))
