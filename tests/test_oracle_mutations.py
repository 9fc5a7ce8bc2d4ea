"""Planted mistakes in the oracle must be caught by its pins.

Each case edits one line of the C oracle (on the CPU, in a temporary build),
then runs three independent pins against the mutant: the explicit product of
the paper's transition matrices (forward), central finite differences of the
mutant's own forward against its backward, and decode steps against the
forward.  Every pin runs on a problem without and with Comba-pk feedback
vectors p (transition alpha I - btilde p k^T, appendix B.3).  At least one pin
must fail for every mutation; the unmodified source must pass all three.
"""
import numpy as np
import pytest

import oracle

MUTATIONS = {
    "feedback_reads_decayed_state": ("x[j] += row[j] * fi;", "x[j] += a * row[j] * fi;"),
    "no_output_correction": ("qn[i] = qt[i] - dh * ft[i];", "qn[i] = qt[i];"),
    "feedback_sign_flipped": ("e[j] = be * vt[j] - bt * x[j];", "e[j] = be * vt[j] + bt * x[j];"),
    "btilde_ignores_b": ("const double bt = bh * be * fb_scale(J, a);", "const double bt = be * fb_scale(J, a);"),
    "bwd_drops_feedback_term": ("const double df = -bt * pde - dh * dqn[i];", "const double df = -dh * dqn[i];"),
    "bwd_dalpha_uses_new_state": ("da += G[(size_t)i * dv + j] * P[(size_t)i * dv + j];",
                                  "da += G[(size_t)i * dv + j] * Hc[(size_t)i * dv + j];"),
    "bwd_carry_without_decay": ("G[(size_t)i * dv + j] = a * G[(size_t)i * dv + j] - bt * ft[i] * de[j];",
                                "G[(size_t)i * dv + j] = G[(size_t)i * dv + j] - bt * ft[i] * de[j];"),
    "decode_step_without_output_correction": ("qn[r] = qt[r] - J->d[h] * ft[r];", "qn[r] = qt[r];"),
    # visible only with feedback vectors p != k
    "pk_state_written_with_p": ("            const double ki = kt[i];\n            double *row = Hs + (size_t)i * dv;\n"
                                "            for (int j = 0; j < dv; ++j) row[j] = a * row[j] + ki * e[j];",
                                "            const double ki = ft[i];\n            double *row = Hs + (size_t)i * dv;\n"
                                "            for (int j = 0; j < dv; ++j) row[j] = a * row[j] + ki * e[j];"),
    "pk_correction_uses_key": ("qn[i] = qt[i] - dh * ft[i];", "qn[i] = qt[i] - dh * kt[i];"),
    "pk_dk_takes_feedback_terms": ("dkt[i] = ge;", "dkt[i] = ge + df;"),
    "pk_carry_uses_key": ("- bt * ft[i] * de[j];", "- bt * kt[i] * de[j];"),
    "pk_dd_uses_key": ("fdq += ft[i] * dqn[i];", "fdq += kt[i] * dqn[i];"),
    "pk_decode_reads_key": ("x[j] += Hs[(size_t)r * dv + j] * ft[r];", "x[j] += Hs[(size_t)r * dv + j] * kt[r];"),
}


def _problem(seed=0, T=40, dk=4, dv=3, pk=False):
    rng = np.random.default_rng(seed)
    k = rng.standard_normal((T, 1, dk))
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    p = dict(q=rng.standard_normal((T, 1, dk)), k=k, v=rng.standard_normal((T, 1, dv)),
             alpha=rng.uniform(0.6, 1.0, (T, 1)), beta=rng.uniform(0.1, 1.0, (T, 1)),
             b=rng.uniform(0.2, 0.9, 1), d=rng.uniform(-1, 1, 1), h0=0.3 * rng.standard_normal((1, 1, dk, dv)))
    if pk:
        f = rng.standard_normal((T, 1, dk))
        p["p"] = f / np.linalg.norm(f, axis=-1, keepdims=True)
    return p


def pin_transition_products(lib):
    for pk in (False, True):
        p = _problem(1, T=12, pk=pk)
        o, hT = oracle.fwd(lib=lib, **p)
        dk = p["k"].shape[-1]
        S = p["h0"][0, 0].T
        for t in range(12):
            kt = p["k"][t, 0]
            ft = p["p"][t, 0] if pk else kt
            Phi = p["alpha"][t, 0] * np.eye(dk) - p["b"][0] * p["beta"][t, 0] * np.outer(ft, kt)
            S = S @ Phi + p["beta"][t, 0] * np.outer(p["v"][t, 0], kt)
            np.testing.assert_allclose(o[t, 0], S @ (p["q"][t, 0] - p["d"][0] * ft), rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(hT[0, 0], S.T, rtol=1e-10, atol=1e-12)


def pin_finite_differences(lib):
    for pk in (False, True):
        p = _problem(2, T=70, pk=pk)
        rng = np.random.default_rng(3)
        dO = rng.standard_normal(p["v"].shape)
        dhT = rng.standard_normal(p["h0"].shape)
        g = oracle.bwd(dO=dO, dhT=dhT, lib=lib, threads=1, **p)

        def loss():
            o, hT = oracle.fwd(lib=lib, threads=1, **p)
            return float(np.sum(o * dO) + np.sum(hT * dhT))

        names = {"q": "dq", "k": "dk", "v": "dv", "alpha": "dalpha", "beta": "dbeta", "b": "db", "d": "dd",
                 "h0": "dh0"}
        if pk:
            names["p"] = "dp"
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
                assert abs(fd - an) <= 2e-6 * max(1.0, abs(an)), (pk, name, fd, an)


def pin_decode_equals_forward(lib):
    for pk in (False, True):
        p = _problem(4, T=6, pk=pk)
        o, hT = oracle.fwd(lib=lib, **p)
        st = p["h0"]
        for t in range(6):
            ot, st = oracle.step(p["q"][t:t + 1], p["k"][t:t + 1], p["v"][t:t + 1], p["alpha"][t:t + 1],
                                 p["beta"][t:t + 1], p["b"], p["d"], st, lib=lib,
                                 p=p["p"][t:t + 1] if pk else None)
            np.testing.assert_allclose(ot[0], o[t], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(st, hT, rtol=1e-11, atol=1e-12)


PINS = (pin_transition_products, pin_finite_differences, pin_decode_equals_forward)


def _run(lib):
    failed = []
    for pin in PINS:
        try:
            pin(lib)
        except AssertionError:
            failed.append(pin.__name__)
    return failed


def test_unmodified_oracle_passes_every_pin(tmp_path):
    lib = oracle.load_variant(oracle.build_variant(oracle.source_text(), str(tmp_path)))
    assert _run(lib) == []


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_planted_mistake_is_caught(name, tmp_path):
    old, new = MUTATIONS[name]
    src = oracle.source_text()
    assert old in src, name
    mutated = src.replace(old, new, 1)   # the first occurrence (forward pass where a line repeats)
    lib = oracle.load_variant(oracle.build_variant(mutated, str(tmp_path)))
    assert _run(lib), f"mutation {name} passed every pin"
