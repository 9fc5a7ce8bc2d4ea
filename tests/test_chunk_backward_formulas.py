"""The chunk backward as the local-gradient and reverse-scan kernels decompose it, in fp64
against the oracle's exact BPTT (host only, no GPU).

The paper prints no backward (it defers to DeltaNet's), so the kernels implement gradients
derived here from the chunk form of section 3.2.  Per chunk, with the forward's
M = (I + A)^{-1}, W = M Diag(s) F, U = M Diag(beta) V, E = U - W H, P = Tril(Q~ K^T * Gamma),
Qhat = Diag(gamma) Q~, Kbar = Diag(gamma_L / gamma_r) K (F = K, or Comba-pk's P):

  reverse scan   dE = P^T dO + Kbar dH',   dH = gamma_L dH' + Qhat^T dO - W^T dE
  local          dQ~ = Diag(gamma) dO H^T + (dO E^T * Gamma) K,   dV = Diag(beta) M^T dE,
                 dW = -dE H^T,   dA = strict_lower(-(M^T dE) E^T),   dK from P, Kbar, W and A,
                 d log-decays collected per position and reverse-cumsummed inside the chunk.

This module writes those steps out in NumPy and checks every gradient against the C oracle's
token-by-token BPTT (itself pinned by finite differences), for the Comba, Comba-iplr and
Comba-pk forms, over packed sequences with ragged last chunks.
"""
import numpy as np
import pytest

import oracle


def _chunk_unit(q, k, v, a, be, b, d, h0, dO, dhT, C, f=None, iplr=False):
    """One (sequence, head): q, k, f [T, dk], v, dO [T, dv], a, be [T], h0, dhT [dk, dv] (H = S^T).
    Returns o, hT and the gradients."""
    T, dk = k.shape
    f = k if f is None else f
    btl = (2.0 * a if iplr else 1.0) * b * be           # btilde; Comba-iplr: 2 alpha b beta
    H = h0.copy()
    saved = []
    o = np.zeros_like(v)
    for c0 in range(0, T, C):
        sl = slice(c0, min(c0 + C, T))
        L = sl.stop - c0
        K, F, Q, V, bt = k[sl], f[sl], q[sl], v[sl], btl[sl]
        g = np.cumsum(np.log(a[sl]))
        gm1 = np.concatenate([[0.0], g[:-1]])
        gam, gamm1 = np.exp(g), np.exp(gm1)
        ii, jj = np.indices((L, L))
        Gam = np.where(ii >= jj, np.exp(np.where(ii >= jj, g[:, None] - g[None, :], 0.0)), 0.0)
        D = np.where(ii > jj, np.exp(np.where(ii > jj, gm1[:, None] - g[None, :], 0.0)), 0.0)
        Qt = Q - d * F
        G = F @ K.T
        A = bt[:, None] * D * G
        M = np.linalg.inv(np.eye(L) + A)
        s = bt * gamm1
        W = M @ (s[:, None] * F)
        U = M @ (be[sl][:, None] * V)
        E = U - W @ H
        P = (Qt @ K.T) * Gam
        kb = np.exp(g[-1] - g)
        o[sl] = (gam[:, None] * Qt) @ H + P @ E
        saved.append(dict(sl=sl, L=L, g=g, gam=gam, gamm1=gamm1, Gam=Gam, D=D, Qt=Qt, G=G, A=A, M=M, s=s,
                          W=W, E=E, P=P, kb=kb, H=H.copy(), bt=bt))
        H = gam[-1] * H + (kb[:, None] * K).T @ E
    hT = H

    gr = {n: np.zeros_like(x) for n, x in (("dq", q), ("dk", k), ("df", f), ("dv", v))}
    dla = np.zeros(T)          # gradient w.r.t. log alpha
    dbt = np.zeros(T)          # gradient w.r.t. btilde
    dbeta = np.zeros(T)        # direct (through U)
    dd = 0.0
    dH = dhT.copy()
    for c in reversed(saved):
        sl, L, H, gam, kb = c["sl"], c["L"], c["H"], c["gam"], c["kb"]
        K, F, V, dOc = k[sl], f[sl], v[sl], dO[sl]
        dHp = dH
        Qhat = gam[:, None] * c["Qt"]
        Kbar = kb[:, None] * K
        # reverse-scan step
        dE = c["P"].T @ dOc + Kbar @ dHp
        dH = gam[-1] * dHp + Qhat.T @ dOc - c["W"].T @ dE
        # local gradients
        dg = np.zeros(L)
        dQhat = dOc @ H.T
        dQt = gam[:, None] * dQhat
        dg += np.sum(Qhat * dQhat, 1)
        dP = dOc @ c["E"].T
        dS = dP * c["Gam"]
        dQt += dS @ K
        dK = dS.T @ c["Qt"]
        TP = dP * c["P"]
        dg += TP.sum(1) - TP.sum(0)
        dKbar = c["E"] @ dHp.T
        dK += kb[:, None] * dKbar
        tk = np.sum(Kbar * dKbar, 1)
        dg[-1] += tk.sum() + gam[-1] * np.sum(H * dHp)
        dg -= tk
        dW = -dE @ H.T
        MtdE, MtdW = c["M"].T @ dE, c["M"].T @ dW
        gr["dv"][sl] = be[sl][:, None] * MtdE
        dbeta[sl] = np.sum(V * MtdE, 1)
        dF = c["s"][:, None] * MtdW
        ds = np.sum(F * MtdW, 1)
        dA = np.tril(-(MtdE @ c["E"].T), -1)
        dbt[sl] = np.sum(dA * c["D"] * c["G"], 1) + ds * c["gamm1"]
        dG = dA * c["bt"][:, None] * c["D"]
        dF += dG @ K
        dK += dG.T @ F
        TA = dA * c["A"]
        dg[:-1] += TA.sum(1)[1:]
        dg -= TA.sum(0)
        dg[:-1] += (ds * c["s"])[1:]
        gr["dq"][sl] = dQt
        dF -= d * dQt
        dd -= np.sum(F * dQt)
        dla[sl] = np.cumsum(dg[::-1])[::-1]
        gr["dk"][sl] = dK
        gr["df"][sl] = dF
    if f is k:
        gr["dk"] = gr["dk"] + gr["df"]
    scale = (2.0 * a if iplr else 1.0)
    dalpha = dla / a + (2.0 * b * be * dbt if iplr else 0.0)
    out = dict(dq=gr["dq"], dk=gr["dk"], dv=gr["dv"], dalpha=dalpha, dbeta=dbeta + scale * b * dbt,
               db=np.sum(scale * be * dbt), dd=dd, dh0=dH)
    if f is not k:
        out["dp"] = gr["df"]
    return o, hT, out


def _problem(seed, pk):
    rng = np.random.default_rng(seed)
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
    dO = rng.standard_normal((Tt, Hh, dv))
    dhT = rng.standard_normal((len(lengths), Hh, dk, dv))
    return p, dO, dhT


@pytest.mark.parametrize("variant", ["splr", "iplr", "pk"])
def test_kernel_decomposition_of_the_chunk_backward_equals_bptt(variant):
    pk = variant == "pk"
    p, dO, dhT = _problem(31, pk)
    ovariant = "iplr" if variant == "iplr" else "splr"
    o_ref, hT_ref = oracle.fwd(variant=ovariant, **p)
    g_ref = oracle.bwd(dO=dO, dhT=dhT, variant=ovariant, **p)
    cu = p["cu_seqlens"]
    Hh = p["q"].shape[1]
    got = {n: np.zeros_like(x) for n, x in g_ref.items()}
    o = np.zeros_like(o_ref)
    hT = np.zeros_like(hT_ref)
    for n in range(len(cu) - 1):
        t0, t1 = int(cu[n]), int(cu[n + 1])
        for h in range(Hh):
            sl = slice(t0, t1)
            on, hTn, g = _chunk_unit(p["q"][sl, h], p["k"][sl, h], p["v"][sl, h], p["alpha"][sl, h],
                                     p["beta"][sl, h], p["b"][h], p["d"][h], p["h0"][n, h], dO[sl, h], dhT[n, h],
                                     C=16, f=p["p"][sl, h] if pk else None, iplr=variant == "iplr")
            o[sl, h], hT[n, h] = on, hTn
            for key in ("dq", "dk", "dv", "dp"):
                if key in g:
                    got[key][sl, h] = g[key]
            got["dalpha"][sl, h], got["dbeta"][sl, h] = g["dalpha"], g["dbeta"]
            got["db"][h] += g["db"]
            got["dd"][h] += g["dd"]
            got["dh0"][n, h] = g["dh0"]
    np.testing.assert_allclose(o, o_ref, rtol=1e-9, atol=1e-10)
    np.testing.assert_allclose(hT, hT_ref, rtol=1e-9, atol=1e-10)
    for key in g_ref:
        np.testing.assert_allclose(got[key], g_ref[key], rtol=1e-8, atol=1e-9, err_msg=key)


SLIPS = {
    "de_without_state_term": ('dE = c["P"].T @ dOc + Kbar @ dHp', 'dE = c["P"].T @ dOc'),
    "dh_feedback_sign": ('dH = gam[-1] * dHp + Qhat.T @ dOc - c["W"].T @ dE',
                         'dH = gam[-1] * dHp + Qhat.T @ dOc + c["W"].T @ dE'),
    # dM without its W path: (M^T dE) U^T in place of (M^T dE) E^T
    "da_without_w_path": ('dA = np.tril(-(MtdE @ c["E"].T), -1)', 'dA = np.tril(-(MtdE @ (c["E"] + c["W"] @ H).T), -1)'),
    "da_transposed": ('dA = np.tril(-(MtdE @ c["E"].T), -1)', 'dA = np.tril(-(c["E"] @ MtdE.T), -1)'),
    "w_decay_at_r": ('dg[:-1] += (ds * c["s"])[1:]', 'dg += ds * c["s"]'),
    "decay_cumsum_forward": ('dla[sl] = np.cumsum(dg[::-1])[::-1]', 'dla[sl] = np.cumsum(dg)'),
    "state_decay_gradient_dropped": ('dg[-1] += tk.sum() + gam[-1] * np.sum(H * dHp)', 'dg[-1] += tk.sum()'),
}


@pytest.mark.parametrize("name", sorted(SLIPS))
def test_planted_slip_in_the_decomposition_is_caught(name):
    """Each edit of one step of the decomposition makes some gradient disagree with the BPTT."""
    import inspect
    old, new = SLIPS[name]
    src = inspect.getsource(_chunk_unit)
    assert src.count(old) == 1, name
    ns = {"np": np}
    exec(compile(src.replace(old, new), "slip", "exec"), ns)
    p, dO, dhT = _problem(33, False)
    g_ref = oracle.bwd(dO=dO, dhT=dhT, **p)
    n1 = int(p["cu_seqlens"][1])
    sl = slice(0, n1)
    _, _, g = ns["_chunk_unit"](p["q"][sl, 0], p["k"][sl, 0], p["v"][sl, 0], p["alpha"][sl, 0], p["beta"][sl, 0],
                                p["b"][0], p["d"][0], p["h0"][0, 0], dO[sl, 0], dhT[0, 0], C=16)
    ref = {"dq": g_ref["dq"][sl, 0], "dk": g_ref["dk"][sl, 0], "dv": g_ref["dv"][sl, 0],
           "dalpha": g_ref["dalpha"][sl, 0], "dbeta": g_ref["dbeta"][sl, 0], "dh0": g_ref["dh0"][0, 0]}
    assert any(not np.allclose(g[key], ref[key], rtol=1e-6, atol=1e-8) for key in ref), name
