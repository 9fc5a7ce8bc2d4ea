"""The state-passing forms the scan kernels run, in fp64 against the oracle (host only).

The chunk equations of section 3.2 pass the state as H_{n+1} = gamma_L H_n + Kbar^T E with
E = U - W H_n.  The scans run algebraically equal forms of that step:

* affine chunk maps (dk = 128): H_{n+1} = (gamma_L I + Atilde) H_n + B with Atilde = -Kbar^T W
  and B = Kbar^T U, where the tcgen05 scan forms B^T = U_s^T K itself from
  U_s = Diag(s) U, s_r = gamma_L / gamma_r;
* its transpose for the backward: dH_n = (gamma_L I + Atilde)^T dH_{n+1} + C_n with
  C_n = Z^T dO_n, Z = Qhat - P W, the scan forming C^T = dO^T Z itself;
* two products per chunk at dk = 256 (no dk x dk map): Pt = (U^T - S^T W^T) Diag(s),
  S^T <- gamma_L S^T + Pt K forward, and Pt = -(dH'^T K^T) Diag(s),
  dH^T <- gamma_L dH'^T + C^T + Pt W in reverse (S^T = H^T here, dv x dk).

Each form is run over every chunk of packed sequences and compared with the oracle's forward
(o, hT) and with its BPTT (dh0).
"""
import numpy as np
import pytest

import oracle


def _factors(q, k, v, a, be, b, d, C, f=None):
    """Per-chunk factors of one (sequence, head), from the chunk equations of section 3.2."""
    f = k if f is None else f
    out = []
    T = k.shape[0]
    for c0 in range(0, T, C):
        sl = slice(c0, min(c0 + C, T))
        L = sl.stop - c0
        K, F, Q, V, bt = k[sl], f[sl], q[sl], v[sl], b * be[sl]
        g = np.cumsum(np.log(a[sl]))
        gm1 = np.concatenate([[0.0], g[:-1]])
        ii, jj = np.indices((L, L))
        Gam = np.where(ii >= jj, np.exp(np.where(ii >= jj, g[:, None] - g[None, :], 0.0)), 0.0)
        D = np.where(ii > jj, np.exp(np.where(ii > jj, gm1[:, None] - g[None, :], 0.0)), 0.0)
        M = np.linalg.inv(np.eye(L) + bt[:, None] * D * (F @ K.T))
        W = M @ ((bt * np.exp(gm1))[:, None] * F)
        U = M @ (be[sl][:, None] * V)
        Qt = Q - d * F
        s = np.exp(g[-1] - g)
        out.append(dict(sl=sl, gL=np.exp(g[-1]), K=K, W=W, U=U, s=s, Kbar=s[:, None] * K,
                        Qhat=np.exp(g)[:, None] * Qt, P=(Qt @ K.T) * Gam))
    return out


def _problem(pk=False):
    rng = np.random.default_rng(41)
    lengths, Hh, dk, dv = [70, 37, 33], 2, 6, 5
    Tt = sum(lengths)
    k = rng.standard_normal((Tt, Hh, dk))
    k /= np.linalg.norm(k, axis=-1, keepdims=True)
    q = rng.standard_normal((Tt, Hh, dk))
    q /= np.linalg.norm(q, axis=-1, keepdims=True)
    p = dict(q=q, k=k, v=rng.standard_normal((Tt, Hh, dv)), alpha=rng.uniform(0.6, 1.0, (Tt, Hh)),
             beta=rng.uniform(0.05, 1.0, (Tt, Hh)), b=rng.uniform(0.2, 0.9, Hh), d=rng.uniform(-1.0, 1.0, Hh),
             h0=0.3 * rng.standard_normal((len(lengths), Hh, dk, dv)),
             cu_seqlens=np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64))
    if pk:
        fv = k + 0.5 * rng.standard_normal((Tt, Hh, dk))
        p["p"] = fv / np.linalg.norm(fv, axis=-1, keepdims=True)
    return p, rng.standard_normal((Tt, Hh, dv)), rng.standard_normal((len(lengths), Hh, dk, dv))


def _units(p):
    cu = p["cu_seqlens"]
    for n in range(len(cu) - 1):
        for h in range(p["q"].shape[1]):
            yield n, h, slice(int(cu[n]), int(cu[n + 1]))


def _fwd_affine(ch, H):
    """Forward with affine chunk maps; B^T formed as U_s^T K.  Returns the chunk-start states and hT."""
    states = []
    for c in ch:
        states.append(H)
        At = -c["Kbar"].T @ c["W"]
        BT = (c["s"][:, None] * c["U"]).T @ c["K"]
        assert np.allclose(BT, (c["Kbar"].T @ c["U"]).T, rtol=1e-12, atol=1e-13)
        H = c["gL"] * H + At @ H + BT.T
    return states, H


def _fwd_wide(ch, H):
    """Forward in the two-product form on S^T = H^T (dv x dk)."""
    St = H.T
    states = []
    for c in ch:
        states.append(St.T)
        Pt = (c["U"].T - St @ c["W"].T) * c["s"][None, :]
        St = c["gL"] * St + Pt @ c["K"]
    return states, St.T


@pytest.mark.parametrize("form", ["affine", "wide"])
@pytest.mark.parametrize("pk", [False, True])
def test_forward_state_forms_reproduce_the_recurrence(form, pk):
    p, _, _ = _problem(pk)
    o_ref, hT_ref = oracle.fwd(**p)
    run = _fwd_affine if form == "affine" else _fwd_wide
    for n, h, sl in _units(p):
        ch = _factors(p["q"][sl, h], p["k"][sl, h], p["v"][sl, h], p["alpha"][sl, h], p["beta"][sl, h], p["b"][h],
                      p["d"][h], 16, f=p["p"][sl, h] if pk else None)
        states, hT = run(ch, p["h0"][n, h])
        np.testing.assert_allclose(hT, hT_ref[n, h], rtol=1e-9, atol=1e-10)
        for c, Hn in zip(ch, states):   # the output kernel's O = Qhat H_n + P (U - W H_n)
            o = c["Qhat"] @ Hn + c["P"] @ (c["U"] - c["W"] @ Hn)
            np.testing.assert_allclose(o, o_ref[sl, h][c["sl"]], rtol=1e-9, atol=1e-10)


@pytest.mark.parametrize("form", ["affine", "wide"])
@pytest.mark.parametrize("pk", [False, True])
def test_reverse_state_forms_reproduce_bptt_dh0(form, pk):
    p, dO, dhT = _problem(pk)
    g_ref = oracle.bwd(dO=dO, dhT=dhT, **p)
    for n, h, sl in _units(p):
        ch = _factors(p["q"][sl, h], p["k"][sl, h], p["v"][sl, h], p["alpha"][sl, h], p["beta"][sl, h], p["b"][h],
                      p["d"][h], 16, f=p["p"][sl, h] if pk else None)
        dH = dhT[n, h]
        for c in reversed(ch):
            dOc = dO[sl, h][c["sl"]]
            Z = c["Qhat"] - c["P"] @ c["W"]
            CT = dOc.T @ Z                                    # C^T = dO^T Z, formed in the scan
            if form == "affine":
                At = -c["Kbar"].T @ c["W"]
                dH = c["gL"] * dH + At.T @ dH + CT.T
            else:
                dHt = dH.T
                Pt = -(dHt @ c["K"].T) * c["s"][None, :]
                dH = (c["gL"] * dHt + CT + Pt @ c["W"]).T
        np.testing.assert_allclose(dH, g_ref["dh0"][n, h], rtol=1e-8, atol=1e-9)


def test_affine_map_needs_the_decay_in_kbar():
    """A plausible slip (Atilde from K instead of Kbar) breaks the forward."""
    p, _, _ = _problem()
    _, hT_ref = oracle.fwd(**p)
    n, h, sl = next(iter(_units(p)))
    ch = _factors(p["q"][sl, h], p["k"][sl, h], p["v"][sl, h], p["alpha"][sl, h], p["beta"][sl, h], p["b"][h],
                  p["d"][h], 16)
    H = p["h0"][n, h]
    for c in ch:
        H = c["gL"] * H - c["K"].T @ c["W"] @ H + c["Kbar"].T @ c["U"]
    assert not np.allclose(H, hT_ref[n, h], rtol=1e-6, atol=1e-8)
