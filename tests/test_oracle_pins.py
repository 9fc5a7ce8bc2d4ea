"""Pins for the fp64 oracle against facts the paper and the mathematics fix.

Each test checks the token-recurrence oracle against something other than
itself: a hand-worked example, a closed form it must reduce to, an explicit
product of the paper's transition matrices, an invariant, or central finite
differences.  A plausible slip in the oracle (a dropped feedback term, decay
on the feedback read, a wrong orientation, a sign) fails at least one.
"""
import json
import os

import numpy as np
import pytest

import oracle
from oracle import chunked

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _rand_problem(rng, lengths, H, dk, dv, unit_k=True, with_b=True, with_h0=True, alpha_lo=0.6):
    Tt = int(np.sum(lengths))
    q = rng.standard_normal((Tt, H, dk))
    k = rng.standard_normal((Tt, H, dk))
    if unit_k:
        k /= np.linalg.norm(k, axis=-1, keepdims=True)
        q /= np.linalg.norm(q, axis=-1, keepdims=True)
    v = rng.standard_normal((Tt, H, dv))
    alpha = rng.uniform(alpha_lo, 1.0, (Tt, H))
    beta = rng.uniform(0.05, 1.0, (Tt, H))
    b = rng.uniform(0.0, 1.0, H) if with_b else None
    d = rng.uniform(-1.0, 1.0, H)
    N = len(lengths)
    h0 = 0.3 * rng.standard_normal((N, H, dk, dv)) if with_h0 else None
    cu = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
    return dict(q=q, k=k, v=v, alpha=alpha, beta=beta, b=b, d=d, h0=h0, cu_seqlens=cu)


# ---------------------------------------------------------------- worked example

def test_hand_worked_scalar_example():
    g = json.load(open(os.path.join(GOLDEN, "scalar_two_tokens.json")))
    x = g["inputs"]
    q = np.array(x["q"]).reshape(2, 1, 1)
    k = np.array(x["k"]).reshape(2, 1, 1)
    v = np.array(x["v"]).reshape(2, 1, 1)
    a = np.array(x["alpha"]).reshape(2, 1)
    be = np.array(x["beta"]).reshape(2, 1)
    o, hT = oracle.fwd(q, k, v, a, be, np.array([x["b"]]), np.array([x["d"]]),
                       h0=np.array(x["h0"]).reshape(1, 1, 1, 1))
    np.testing.assert_allclose(o.ravel(), g["expected"]["o"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(hT.ravel(), [g["expected"]["hT"]], rtol=0, atol=1e-14)


def test_hand_worked_scalar_backward():
    """The same two tokens' gradients, worked by hand (the adjoint carried through the decay)."""
    g = json.load(open(os.path.join(GOLDEN, "scalar_two_tokens.json")))
    x, bw = g["inputs"], g["backward"]
    args = [np.array(x[n]).reshape(2, 1, 1) for n in ("q", "k", "v")]
    args += [np.array(x["alpha"]).reshape(2, 1), np.array(x["beta"]).reshape(2, 1)]
    out = oracle.bwd(*args, np.array([x["b"]]), np.array([x["d"]]), np.array(bw["inputs"]["dO"]).reshape(2, 1, 1),
                     h0=np.array(x["h0"]).reshape(1, 1, 1, 1), dhT=np.array(bw["inputs"]["dhT"]).reshape(1, 1, 1, 1))
    for name, want in bw["expected"].items():
        np.testing.assert_allclose(out[name].ravel(), np.ravel(want), rtol=0, atol=1e-13, err_msg=name)


@pytest.mark.parametrize("form", ["splr", "iplr", "pk"])
def test_hand_worked_two_by_two_example(form):
    """dk = dv = 2, two tokens, worked by hand: fixes the state's orientation (S = H^T), the
    order of the transition's outer product, and the iplr and pk forms."""
    g = json.load(open(os.path.join(GOLDEN, "matrix_two_tokens.json")))
    x = g["inputs"]
    q, k, v, fv = (np.array(x[n]).reshape(2, 1, 2) for n in ("q", "k", "v", "p"))
    a = np.array(x["alpha"]).reshape(2, 1)
    be = np.array(x["beta"]).reshape(2, 1)
    h0 = np.array(x["S0"]).T.reshape(1, 1, 2, 2)
    o, hT = oracle.fwd(q, k, v, a, be, np.array([x["b"]]), np.array([x["d"]]), h0=h0,
                       variant="iplr" if form == "iplr" else "splr", p=fv if form == "pk" else None)
    np.testing.assert_allclose(o.reshape(2, 2), g["expected"][form]["o"], rtol=0, atol=1e-14)
    np.testing.assert_allclose(hT.reshape(2, 2), g["expected"][form]["hT"], rtol=0, atol=1e-14)


# ------------------------------------------------------------------ reductions

def test_reduces_to_gated_linear_attention_when_no_feedback():
    """b = 0, d = 0: the scalar-gated linear attention closed form (Mamba2/GLA row of
    the paper's model table; basic chunk form of section 2)."""
    rng = np.random.default_rng(1)
    T, H, dk, dv = 23, 2, 5, 3
    p = _rand_problem(rng, [T], H, dk, dv)
    p["b"] = np.zeros(H)
    p["d"] = np.zeros(H)
    o, hT = oracle.fwd(**p)
    q, k, v, a, be, h0 = p["q"], p["k"], p["v"], p["alpha"], p["beta"], p["h0"][0]
    for h in range(H):
        gam = np.cumprod(a[:, h])
        for t in range(T):
            ref = gam[t] * (h0[h].T @ q[t, h])
            for i in range(t + 1):
                ref = ref + (gam[t] / gam[i]) * be[i, h] * v[i, h] * (k[i, h] @ q[t, h])
            np.testing.assert_allclose(o[t, h], ref, rtol=1e-12, atol=1e-12)
        refT = gam[-1] * h0[h] + sum((gam[-1] / gam[i]) * be[i, h] * np.outer(k[i, h], v[i, h]) for i in range(T))
        np.testing.assert_allclose(hT[0, h], refT, rtol=1e-12, atol=1e-12)


def test_reduces_to_delta_rule():
    """alpha = 1, b = 1, d = 0: DeltaNet's S_t = S_{t-1}(I - beta k k^T) + beta v k^T, o = S q
    (Eq. "delta rule"), written with explicit dv x dk matrices."""
    rng = np.random.default_rng(2)
    T, dk, dv = 17, 4, 6
    p = _rand_problem(rng, [T], 1, dk, dv, with_h0=False)
    p["alpha"][:] = 1.0
    p["b"] = np.ones(1)
    p["d"] = np.zeros(1)
    o, hT = oracle.fwd(**p)
    S = np.zeros((dv, dk))
    for t in range(T):
        kt, vt, bt = p["k"][t, 0], p["v"][t, 0], p["beta"][t, 0]
        S = S @ (np.eye(dk) - bt * np.outer(kt, kt)) + bt * np.outer(vt, kt)
        np.testing.assert_allclose(o[t, 0], S @ p["q"][t, 0], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(hT[0, 0], S.T, rtol=1e-12, atol=1e-12)


def test_zero_input_gate_is_pure_decay():
    """beta = 0: no write and no feedback; o_t = gamma_t H_0^T (q_t - d k_t)."""
    rng = np.random.default_rng(3)
    T, H, dk, dv = 19, 2, 4, 5
    p = _rand_problem(rng, [T], H, dk, dv)
    p["beta"][:] = 0.0
    o, hT = oracle.fwd(**p)
    for h in range(H):
        gam = np.cumprod(p["alpha"][:, h])
        for t in range(T):
            qn = p["q"][t, h] - p["d"][h] * p["k"][t, h]
            np.testing.assert_allclose(o[t, h], gam[t] * p["h0"][0, h].T @ qn, rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(hT[0, h], gam[-1] * p["h0"][0, h], rtol=1e-12, atol=1e-13)


def test_full_strength_write_memorises_value():
    """alpha = beta = b = 1 with ||k|| = 1: after the write, S_t k_t = v_t exactly."""
    rng = np.random.default_rng(4)
    T, dk, dv = 25, 8, 5
    p = _rand_problem(rng, [T], 1, dk, dv)
    p["alpha"][:] = 1.0
    p["beta"][:] = 1.0
    p["b"] = np.ones(1)
    p["d"] = np.zeros(1)
    p["q"] = p["k"].copy()
    o, _ = oracle.fwd(**p)
    np.testing.assert_allclose(o[:, 0], p["v"][:, 0], rtol=1e-12, atol=1e-12)


# ------------------------------------------------------- brute-force unrolling

def _transition(alpha, btilde, k):
    return alpha * np.eye(k.shape[0]) - btilde * np.outer(k, k)


def test_matches_unrolled_transition_products():
    """Eq. "chunk-wise comba" over a whole sequence: S_r = S_0 prod_i (alpha_i - btilde_i k_i k_i^T)
    + sum_i beta_i v_i k_i^T prod_{j>i}(...), with explicit dk x dk products; o_r = S_r (q_r - d k_r)."""
    rng = np.random.default_rng(5)
    T, dk, dv = 14, 5, 3
    p = _rand_problem(rng, [T], 1, dk, dv, unit_k=False)
    o, hT = oracle.fwd(**p)
    b, d = p["b"][0], p["d"][0]
    S0 = p["h0"][0, 0].T
    Phi = [_transition(p["alpha"][t, 0], b * p["beta"][t, 0], p["k"][t, 0]) for t in range(T)]
    for r in range(1, T + 1):
        D = np.eye(dk)
        for i in range(r):
            D = D @ Phi[i]
        Hr = np.zeros((dv, dk))
        for i in range(r):
            prod = np.eye(dk)
            for j in range(i + 1, r):
                prod = prod @ Phi[j]
            Hr += p["beta"][i, 0] * np.outer(p["v"][i, 0], p["k"][i, 0]) @ prod
        Sr = S0 @ D + Hr
        qn = p["q"][r - 1, 0] - d * p["k"][r - 1, 0]
        np.testing.assert_allclose(o[r - 1, 0], Sr @ qn, rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(hT[0, 0], Sr.T, rtol=1e-11, atol=1e-12)


def test_transition_spectrum_and_state_norm_bound():
    """Table "splr-iplr": alpha - btilde k k^T has eigenvalue alpha (multiplicity dk-1) and
    alpha - btilde ||k||^2.  With ||k|| = 1 the oracle's states therefore obey
    ||H_t||_2 <= max(|alpha|, |alpha - btilde|) ||H_{t-1}||_2 + beta ||v||."""
    rng = np.random.default_rng(6)
    dk = 6
    for _ in range(5):
        k = rng.standard_normal(dk)
        a, bt = rng.uniform(0.5, 1), rng.uniform(0, 1)
        ev = np.sort(np.linalg.eigvalsh(_transition(a, bt, k)))
        ref = np.sort(np.r_[np.full(dk - 1, a), a - bt * (k @ k)])
        np.testing.assert_allclose(ev, ref, rtol=1e-12, atol=1e-12)
    T, dv = 30, 4
    p = _rand_problem(rng, [T], 1, dk, dv)
    prev = np.linalg.norm(p["h0"][0, 0], 2)
    b = p["b"][0]
    for t in range(1, T + 1):
        sub = {key: (val[:t] if key in ("q", "k", "v", "alpha", "beta") else val) for key, val in p.items()}
        sub["cu_seqlens"] = np.array([0, t])
        _, hT = oracle.fwd(**sub)
        cur = np.linalg.norm(hT[0, 0], 2)
        a, be = p["alpha"][t - 1, 0], p["beta"][t - 1, 0]
        bound = max(abs(a), abs(a - b * be)) * prev + be * np.linalg.norm(p["v"][t - 1, 0])
        assert cur <= bound * (1 + 1e-12) + 1e-14
        prev = cur


# ------------------------------------------------------ paper's chunk algebra

@pytest.mark.parametrize("C", [1, 4, 16, 64])
def test_paper_chunk_equations_equal_recurrence(C):
    """Section 3.2: the WY/UT chunk form (single inverse M, W, U, inter-chunk state and
    output equations) under the stated readings reproduces the token recurrence,
    including short last chunks and several packed sequences."""
    rng = np.random.default_rng(7)
    p = _rand_problem(rng, [150, 37, 64], 2, 6, 5)
    o, hT = oracle.fwd(**p)
    oc, hTc = chunked.chunk_forward(C=C, **p)
    np.testing.assert_allclose(oc, o, rtol=1e-10, atol=1e-11)
    np.testing.assert_allclose(hTc, hT, rtol=1e-10, atol=1e-11)


# ----------------------------------------------------------------- gradients

def _loss(p, dO, dhT):
    o, hT = oracle.fwd(**p, threads=1)
    return float(np.sum(o * dO) + np.sum(hT * dhT))


def test_gradients_match_central_differences():
    """Every gradient of L = <o, dO> + <hT, dhT> against fp64 central differences,
    across two packed sequences that cross the oracle's 64-token checkpoint."""
    rng = np.random.default_rng(8)
    p = _rand_problem(rng, [70, 45], 2, 3, 4)
    dO = rng.standard_normal(p["v"].shape)
    dhT = rng.standard_normal(p["h0"].shape)
    g = oracle.bwd(dO=dO, dhT=dhT, threads=1, **p)
    names = {"q": "dq", "k": "dk", "v": "dv", "alpha": "dalpha", "beta": "dbeta", "b": "db", "d": "dd",
             "h0": "dh0"}
    eps = 1e-6
    for name, gname in names.items():
        arr = p[name]
        flat = arr.reshape(-1)
        idx = rng.choice(flat.size, size=min(flat.size, 24), replace=False)
        for i in idx:
            old = flat[i]
            flat[i] = old + eps
            lp = _loss(p, dO, dhT)
            flat[i] = old - eps
            lm = _loss(p, dO, dhT)
            flat[i] = old
            fd = (lp - lm) / (2 * eps)
            an = g[gname].reshape(-1)[i]
            assert abs(fd - an) <= 2e-6 * max(1.0, abs(an)), (name, i, fd, an)


def test_gradient_without_b_and_h0():
    """b = NULL means b = 1 and h0 = NULL means a zero state; dh0 is still produced."""
    rng = np.random.default_rng(9)
    p = _rand_problem(rng, [33], 1, 3, 2, with_b=False, with_h0=False)
    dO = rng.standard_normal(p["v"].shape)
    g = oracle.bwd(dO=dO, **p)
    q = dict(p)
    q["b"] = np.ones(1)
    q["h0"] = np.zeros((1, 1, 3, 2))
    g2 = oracle.bwd(dO=dO, **q)
    for key in ("dq", "dk", "dv", "dalpha", "dbeta", "dd", "dh0"):
        np.testing.assert_allclose(g[key], g2[key], rtol=1e-13, atol=1e-14)


# ------------------------------------------- varlen, state passing, decode

def test_packed_equals_separate_runs():
    rng = np.random.default_rng(10)
    lens = [31, 64, 5, 90]
    p = _rand_problem(rng, lens, 2, 4, 3)
    o, hT = oracle.fwd(**p)
    dO = rng.standard_normal(p["v"].shape)
    g = oracle.bwd(dO=dO, **p)
    cu = p["cu_seqlens"]
    for n in range(len(lens)):
        s = slice(cu[n], cu[n + 1])
        sub = {key: p[key][s] for key in ("q", "k", "v", "alpha", "beta")}
        on, hn = oracle.fwd(b=p["b"], d=p["d"], h0=p["h0"][n:n + 1], **sub)
        np.testing.assert_allclose(o[s], on, rtol=1e-13, atol=1e-14)
        np.testing.assert_allclose(hT[n:n + 1], hn, rtol=1e-13, atol=1e-14)
        gn = oracle.bwd(b=p["b"], d=p["d"], h0=p["h0"][n:n + 1], dO=dO[s], **sub)
        for key in ("dq", "dk", "dv", "dalpha", "dbeta"):
            np.testing.assert_allclose(g[key][s], gn[key], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(g["dh0"][n:n + 1], gn["dh0"], rtol=1e-12, atol=1e-13)


def test_state_passing_split_equals_full_run():
    """Run [0,T1) then [T1,T) with h0 <- hT (and dhT <- dh0 backwards) == one run."""
    rng = np.random.default_rng(11)
    T, T1 = 100, 37
    p = _rand_problem(rng, [T], 2, 4, 5)
    dO = rng.standard_normal(p["v"].shape)
    dhT = rng.standard_normal(p["h0"].shape)
    o, hT = oracle.fwd(**p)
    g = oracle.bwd(dO=dO, dhT=dhT, **p)
    tok = ("q", "k", "v", "alpha", "beta")
    A = {key: p[key][:T1] for key in tok}
    Bp = {key: p[key][T1:] for key in tok}
    oa, ha = oracle.fwd(b=p["b"], d=p["d"], h0=p["h0"], **A)
    ob, hb = oracle.fwd(b=p["b"], d=p["d"], h0=ha, **Bp)
    np.testing.assert_allclose(np.concatenate([oa, ob]), o, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(hb, hT, rtol=1e-12, atol=1e-13)
    gb = oracle.bwd(b=p["b"], d=p["d"], h0=ha, dO=dO[T1:], dhT=dhT, **Bp)
    ga = oracle.bwd(b=p["b"], d=p["d"], h0=p["h0"], dO=dO[:T1], dhT=gb["dh0"], **A)
    for key in ("dq", "dk", "dv", "dalpha", "dbeta"):
        np.testing.assert_allclose(np.concatenate([ga[key], gb[key]]), g[key], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(ga["dh0"], g["dh0"], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(ga["db"] + gb["db"], g["db"], rtol=1e-11, atol=1e-12)
    np.testing.assert_allclose(ga["dd"] + gb["dd"], g["dd"], rtol=1e-11, atol=1e-12)


def test_decode_steps_equal_forward():
    """N calls of the one-token step from S_0 == the forward over N tokens with h0 = S_0."""
    rng = np.random.default_rng(12)
    Bd, H, dk, dv, N = 3, 2, 4, 5, 9
    p = _rand_problem(rng, [N] * Bd, H, dk, dv)
    q, k, v = (p[x].reshape(Bd, N, H, -1) for x in ("q", "k", "v"))
    a, be = p["alpha"].reshape(Bd, N, H), p["beta"].reshape(Bd, N, H)
    o, hT = oracle.fwd(q, k, v, a, be, p["b"], p["d"], h0=p["h0"])
    st = p["h0"].copy()
    for t in range(N):
        ot, st = oracle.step(q[:, t], k[:, t], v[:, t], a[:, t], be[:, t], p["b"], p["d"], st)
        np.testing.assert_allclose(ot, o[:, t], rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(st, hT, rtol=1e-12, atol=1e-13)


def test_thread_count_does_not_change_bits():
    rng = np.random.default_rng(13)
    p = _rand_problem(rng, [40, 70, 3], 3, 4, 4)
    dO = rng.standard_normal(p["v"].shape)
    o1, h1 = oracle.fwd(threads=1, **p)
    o4, h4 = oracle.fwd(threads=4, **p)
    assert np.array_equal(o1, o4) and np.array_equal(h1, h4)
    g1 = oracle.bwd(dO=dO, threads=1, **p)
    g4 = oracle.bwd(dO=dO, threads=4, **p)
    for key in g1:
        assert np.array_equal(g1[key], g4[key]), key


def test_param_gradients_are_sums_of_token_contributions():
    """dd = -sum_t k_t . dq~_t (q~ = q - d k, section 3) and db = sum_t beta_t dbtilde_t with
    dbtilde_t = (dbeta_t - v_t . dv_t / beta_t) / b (btilde = b beta, section 3.1; dv = beta de):
    the per-head sums rebuilt from the oracle's per-token outputs equal its db and dd."""
    from paper_2506_02475_gb300 import inputs
    w = inputs.make("custom", B=2, T=100, H=3, dk=8, dv=8, with_b=True, with_h0=True, with_grads=True, dtype="f32")
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT)
    cdd = -np.einsum("bthd,bthd->h", w.k, r["dq"])
    cdb = ((w.beta * r["dbeta"] - np.einsum("bthd,bthd->bth", w.v, r["dv"])) / w.b).sum((0, 1))
    np.testing.assert_allclose(cdd, r["dd"], rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(cdb, r["db"], rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("variant", ["splr", "iplr"])
def test_value_columns_split_into_independent_heads(variant):
    """The state's dv columns evolve independently given (q, k, gates): a head with dv = 8 equals two
    heads with dv = 4 that share q, k, alpha, beta, b, d (the value-head-group reading): outputs
    and dv concatenate, the key-side gradients add, h0/hT/dh0 split by columns."""
    rng = np.random.default_rng(61)
    T, H, dk, dv = 70, 2, 5, 8
    k = rng.standard_normal((1, T, H, dk))
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    p = dict(q=rng.standard_normal((1, T, H, dk)), k=k, v=rng.standard_normal((1, T, H, dv)),
             alpha=rng.uniform(0.6, 1.0, (1, T, H)), beta=rng.uniform(0.1, 1.0, (1, T, H)), b=rng.uniform(0.2, 0.9, H),
             d=rng.uniform(-1, 1, H), h0=0.3 * rng.standard_normal((1, H, dk, dv)))
    dO = rng.standard_normal((1, T, H, dv))
    dhT = rng.standard_normal((1, H, dk, dv))
    o, hT = oracle.fwd(**p, variant=variant)
    g = oracle.bwd(**p, dO=dO, dhT=dhT, variant=variant)
    halves = [slice(0, 4), slice(4, 8)]
    parts = []
    for sl in halves:
        ph = dict(p, v=p["v"][..., sl], h0=p["h0"][..., sl])
        oh, hTh = oracle.fwd(**ph, variant=variant)
        gh = oracle.bwd(**ph, dO=dO[..., sl], dhT=dhT[..., sl], variant=variant)
        parts.append((oh, hTh, gh))
    np.testing.assert_allclose(np.concatenate([x[0] for x in parts], -1), o, rtol=1e-12, atol=1e-13)
    np.testing.assert_allclose(np.concatenate([x[1] for x in parts], -1), hT, rtol=1e-12, atol=1e-13)
    for key in ("dv", "dh0"):
        np.testing.assert_allclose(np.concatenate([x[2][key] for x in parts], -1), g[key], rtol=1e-11, atol=1e-12)
    for key in ("dq", "dk", "dalpha", "dbeta", "db", "dd"):
        np.testing.assert_allclose(parts[0][2][key] + parts[1][2][key], g[key], rtol=1e-10, atol=1e-11, err_msg=key)
