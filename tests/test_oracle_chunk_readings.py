"""Planted misreadings of the paper's chunk equations (section 3.2) fail the recurrence pin.

The chunk form's subscripts are garbled in the paper, so ``oracle/chunked.py`` fixes
a reading of each (a strictly lower ``lower``, a ``Tril`` that keeps the diagonal,
gamma_{i-1}/gamma_j inside the inverse, alpha^{0->C-1} = gamma_0..gamma_{C-1},
alpha^{i->C} = gamma_C / gamma_i).  Each test here edits one of those choices, or
drops one factor, in a copy of the module's source on the CPU and checks that the
edited chunk form no longer reproduces the token recurrence of the C oracle.  So the
readings are forced by the recurrence (section 3, Eq. "comba-S"), not picked freely.
"""
import os

import numpy as np
import pytest

import oracle
from oracle import chunked

SRC = os.path.join(os.path.dirname(chunked.__file__), "chunked.py")

# name -> (text in chunked.py, its misreading); each edit is one plausible slip
MISREADINGS = {
    # "lower" inside the inverse taken with its diagonal
    "inverse_lower_keeps_diagonal": ("low = np.tril(np.diag(bt) @ (Aim1_j * (P @ K.T)), -1)",
                                     "low = np.tril(np.diag(bt) @ (Aim1_j * (P @ K.T)), 0)"),
    # "Tril" of the output equation taken strictly lower
    "output_tril_strict": ("np.tril(Qt @ K.T * Ai_j) @ Vn", "np.tril(Qt @ K.T * Ai_j, -1) @ Vn"),
    # the (i-1)/j decay inside the inverse read as i/j
    "inverse_decay_i_over_j": ("Aim1_j = gam0[:, None] / gam[None, :]", "Aim1_j = gam[:, None] / gam[None, :]"),
    # alpha^{0->C-1} read as gamma_1..gamma_C
    "w_decay_gamma_r": ("W = M @ np.diag(bt * gam0) @ P", "W = M @ np.diag(bt * gam) @ P"),
    # alpha^{i->C} read as gamma_C / gamma_{i-1}
    "state_decay_from_previous_position": ("np.diag(gam[-1] / gam) @ K", "np.diag(gam[-1] / gam0) @ K"),
    # the inter-chunk output term decayed to position r-1
    "output_state_term_gamma_r_minus_1": ("np.diag(gam) @ Qt @ S.T", "np.diag(gam0) @ Qt @ S.T"),
    # the intra-chunk output term without its decay matrix
    "output_intra_undecayed": ("np.tril(Qt @ K.T * Ai_j) @ Vn", "np.tril(Qt @ K.T) @ Vn"),
    # feedback strength without b (section 3.1)
    "btilde_without_b": ("bt = b * be ", "bt = be "),
    # U without the input gate
    "u_without_beta": ("U = M @ np.diag(be) @ V", "U = M @ V"),
    # output correction dropped
    "no_output_correction": ("Qt = Q - d * P", "Qt = Q"),
    # the state carried to the next chunk without its decay
    "state_carried_undecayed": ("S = gam[-1] * S + Vn.T", "S = S + Vn.T"),
    # pseudo-value with the state's sign flipped
    "pseudo_value_sign": ("Vn = U - W @ S.T", "Vn = U + W @ S.T"),
}

# Comba-pk (appendix B.3): misreadings of where P replaces K
PK_MISREADINGS = {
    "pk_gram_uses_keys": ("(Aim1_j * (P @ K.T))", "(Aim1_j * (K @ K.T))"),
    "pk_w_uses_keys": ("W = M @ np.diag(bt * gam0) @ P", "W = M @ np.diag(bt * gam0) @ K"),
    "pk_correction_uses_keys": ("Qt = Q - d * P", "Qt = Q - d * K"),
    "pk_state_written_with_p": ("np.diag(gam[-1] / gam) @ K", "np.diag(gam[-1] / gam) @ P"),
}


def _module(source):
    ns = {"__name__": "chunked_variant"}
    exec(compile(source, "chunked_variant", "exec"), ns)
    return ns


def _problem(pk=False):
    rng = np.random.default_rng(21)
    lengths, H, dk, dv = [150, 37, 64], 2, 6, 5
    Tt = sum(lengths)
    k = rng.standard_normal((Tt, H, dk))
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    q = rng.standard_normal((Tt, H, dk))
    q /= np.linalg.norm(q, axis=-1, keepdims=True)
    p = dict(q=q, k=k, v=rng.standard_normal((Tt, H, dv)), alpha=rng.uniform(0.6, 1.0, (Tt, H)),
             beta=rng.uniform(0.05, 1.0, (Tt, H)), b=rng.uniform(0.2, 0.9, H), d=rng.uniform(-1.0, 1.0, H),
             h0=0.3 * rng.standard_normal((len(lengths), H, dk, dv)),
             cu_seqlens=np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64))
    if pk:
        f = k + 0.5 * rng.standard_normal((Tt, H, dk))
        p["p"] = f / np.linalg.norm(f, axis=-1, keepdims=True)
    return p


def _agrees(mod, pk):
    p = _problem(pk)
    o, hT = oracle.fwd(**p)
    oc, hTc = mod["chunk_forward"](C=16, **p)
    return np.allclose(oc, o, rtol=1e-9, atol=1e-10) and np.allclose(hTc, hT, rtol=1e-9, atol=1e-10)


def _source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("pk", [False, True])
def test_unedited_copy_reproduces_the_recurrence(pk):
    assert _agrees(_module(_source()), pk)


@pytest.mark.parametrize("name", sorted(MISREADINGS))
def test_misreading_breaks_the_recurrence(name):
    old, new = MISREADINGS[name]
    src = _source()
    assert src.count(old) == 1, name
    assert not _agrees(_module(src.replace(old, new)), pk=False), name


@pytest.mark.parametrize("name", sorted(PK_MISREADINGS))
def test_pk_misreading_breaks_the_recurrence(name):
    old, new = PK_MISREADINGS[name]
    src = _source()
    assert src.count(old) == 1, name
    assert not _agrees(_module(src.replace(old, new)), pk=True), name
