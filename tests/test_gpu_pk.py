"""GPU parity of the Comba-pk form (appendix B.3; comba_chunk_fwd_pk / _bwd_pk /
comba_recurrent_step_pk) against the oracle with feedback vectors p: x = H^T p, e = beta v -
btilde x, H <- alpha H + k e^T, o = H^T (q - d p).  dd and db take the max-norm relative
error over their heads like every other tensor."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import np64, param_grad_errors, param_grad_report, rel, tol, to_dev
from paper_2506_02475_gb300 import (comba_chunk_bwd_pk, comba_chunk_fwd_pk, comba_recurrent_step_pk,
                                    comba_workspace_size, inputs)
from paper_2506_02475_gb300 import binding

pytestmark = pytest.mark.gpu


def _with_p(w, seed):
    p = inputs.feedback_vectors(w.k, w.dtype, seed_offset=seed)
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    return p, torch.from_numpy(np.ascontiguousarray(p)).cuda().to(tdt)


def _run(w, t, tp, variant="splr"):
    """Forward saving factors + backward reusing them (the benchmark's configuration), and a
    recomputing backward, which must agree bitwise."""
    iplr = variant == "iplr"
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], t["cu_seqlens"], backward=True, flags=binding.COMBA_PK),
                     dtype=torch.uint8, device="cuda")
    args = (t["q"], t["k"], t["v"], tp, t["alpha"], t["beta"], t["d"])
    o, hT = comba_chunk_fwd_pk(*args, b=t["b"], h0=t["h0"], cu_seqlens=t["cu_seqlens"], output_final_state=True,
                               workspace=ws, save_factors=True, iplr=iplr)
    g = comba_chunk_bwd_pk(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"], cu_seqlens=t["cu_seqlens"],
                           workspace=ws, reuse_factors=True, iplr=iplr)
    g2 = comba_chunk_bwd_pk(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"], cu_seqlens=t["cu_seqlens"],
                            iplr=iplr)
    torch.cuda.synchronize()
    g = {key: np64(val) for key, val in g.items()}
    for key in ("dq", "dk", "dv", "dp", "dalpha", "dbeta", "dd", "dh0"):
        assert np.array_equal(g[key], np64(g2[key])), key
    return np64(o), np64(hT), g


def _check(w, p, o, hT, g, variant="splr", heads=None):
    """Every output against the oracle (on the heads `heads`, all when None)."""
    sl = (lambda x, ax: x) if heads is None else (lambda x, ax: np.take(x, heads, axis=ax))
    tok_ax = -2
    ref_in = dict(q=sl(w.q, tok_ax), k=sl(w.k, tok_ax), v=sl(w.v, tok_ax), p=sl(p, tok_ax), alpha=sl(w.alpha, -1),
                  beta=sl(w.beta, -1), b=None if w.b is None else sl(w.b, 0), d=sl(w.d, 0),
                  h0=None if w.h0 is None else sl(w.h0, 1))
    ro, rhT = oracle.fwd(**ref_in, cu_seqlens=w.cu_seqlens, variant=variant)
    r = oracle.bwd(**ref_in, dO=sl(w.dO, tok_ax), dhT=None if w.dhT is None else sl(w.dhT, 1),
                   cu_seqlens=w.cu_seqlens, variant=variant)
    tl = tol(w.dtype)
    errs = {"o": rel(sl(o, tok_ax), ro), "hT": rel(sl(hT, 1), rhT)}
    for key in ("dq", "dk", "dv", "dp"):
        errs[key] = rel(sl(g[key], tok_ax), r[key])
    for key in ("dalpha", "dbeta"):
        errs[key] = rel(sl(g[key], -1), r[key])
    errs["dh0"] = rel(sl(g["dh0"], 1), r["dh0"])
    gp = {"dd": sl(g["dd"], 0), "db": sl(g["db"], 0)}
    errs.update(param_grad_errors(gp, r))
    bad = {key: e for key, e in errs.items() if not e <= tl}
    # context for dd (a sum of -p . dq over tokens: its scale takes p where the plain form takes k)
    assert not bad, (bad, errs, param_grad_report(gp, r, ref_in["p"], ref_in["v"], ref_in["beta"], ref_in["b"]))
    return errs


CASES = [
    # dtype, dk, dv, B, T, lengths, variant
    ("bf16", 128, 128, 2, 300, None, "splr"),
    ("bf16", 128, 128, 1, None, [1, 63, 64, 65, 0, 200, 7], "splr"),
    ("bf16", 128, 64, 2, 130, None, "iplr"),
    ("bf16", 64, 128, 1, 127, None, "splr"),
    ("f32", 64, 64, 2, 200, None, "splr"),
    ("f32", 64, 64, 1, None, [70, 0, 5, 133], "iplr"),
    # head dim 256: one value head of width 64, then two (dp summed over them like dq and dk)
    ("bf16", 256, 64, 2, 150, None, "splr"),
    ("bf16", 256, 128, 1, None, [1, 63, 64, 65, 0, 90], "iplr"),
]


@pytest.mark.parametrize("dtype,dk,dv,B,T,lengths,variant", CASES)
def test_pk_forward_backward(dtype, dk, dv, B, T, lengths, variant):
    w = inputs.make("custom", B=B, T=T, H=3, dk=dk, dv=dv, dtype=dtype, with_b=True, with_h0=True, with_grads=True,
                    lengths=lengths, seed_offset=dk + 7 * len(lengths or [])) if lengths else \
        inputs.make("custom", B=B, T=T, H=3, dk=dk, dv=dv, dtype=dtype, with_b=True, with_h0=True, with_grads=True,
                    seed_offset=dk + dv + T)
    p, tp = _with_p(w, seed=dk + dv)
    t = to_dev(w)
    _check(w, p, *_run(w, t, tp, variant), variant=variant)


def test_pk_with_p_equal_to_k_matches_the_plain_form_on_the_gpu():
    """p = k through the pk kernels gives the plain form's outputs (dk + dp = plain dk)."""
    from paper_2506_02475_gb300 import comba_chunk_bwd, comba_chunk_fwd
    w = inputs.make("custom", B=1, T=200, H=2, dk=128, dv=128, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=91)
    t = to_dev(w)
    o, hT, g = _run(w, t, t["k"])
    o0, hT0 = comba_chunk_fwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], b=t["b"], h0=t["h0"],
                              output_final_state=True)
    g0 = comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], b=t["b"], h0=t["h0"],
                         dhT=t["dhT"])
    torch.cuda.synchronize()
    tl = tol("bf16")
    assert rel(o, np64(o0)) <= tl and rel(hT, np64(hT0)) <= tl
    assert rel(g["dk"] + g["dp"], np64(g0["dk"])) <= tl
    for key in ("dq", "dv", "dalpha", "dbeta", "dh0"):
        assert rel(g[key], np64(g0[key])) <= tl, key


def test_pk_full_size():
    """B=4 T=4096 H=16 d=128 bf16 in the benchmark's configuration; every output against the
    oracle over the whole workload, forward and backward."""
    w = inputs.make("lm1p3b")
    p, tp = _with_p(w, seed=0)
    t = to_dev(w)
    o, hT, g = _run(w, t, tp)
    del t, tp
    print("lm1p3b pk", {k_: f"{e:.2e}" for k_, e in _check(w, p, o, hT, g).items()})


@pytest.mark.parametrize("dtype,iplr,dk,dv", [("bf16", False, 128, 128), ("f32", True, 128, 128),
                                              ("bf16", True, 256, 256)])
def test_pk_decode_steps(dtype, iplr, dk, dv):
    Bd, H, steps = 5, 3, 6
    state = inputs.decode_state(Bd, H, dk, dv, seed_offset=3)
    b = np.random.default_rng(5).uniform(0, 1, H).astype(np.float32)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    tok = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda().to(tdt)
    f32 = lambda x: torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()
    st_gpu = f32(state)
    st_ref = state.astype(np.float64)
    for s in range(steps):
        q, k, v, a, be, d = inputs.decode_tokens(s, Bd, H, dk, dv, dtype)
        p = inputs.feedback_vectors(k, dtype, seed_offset=s)
        o = comba_recurrent_step_pk(tok(q), tok(k), tok(v), tok(p), f32(a), f32(be), f32(d), st_gpu, b=f32(b),
                                    iplr=iplr)
        ro, st_ref = oracle.step(q, k, v, a, be, b, d, st_ref, variant="iplr" if iplr else "splr", p=p)
        torch.cuda.synchronize()
        assert rel(np64(o), ro) <= tol(dtype)
        assert rel(np64(st_gpu), st_ref) <= tol(dtype)
