"""GPU parity of dk != dv on the tcgen05 path through value-head groups: dv = 256 or 384 with
dk = 128 (bf16) run as dv / 128 value heads of width 128 that share their key head's q, k and
gates; the key-side gradients (dq, dk, dalpha, dbeta, db, dd) are summed over each group in a
fixed order.  Compared with the oracle, which takes any dk, dv directly."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import np64, param_grad_errors, param_grad_report, rel, tol, to_dev
from paper_2506_02475_gb300 import comba_chunk_bwd, comba_chunk_fwd, comba_recurrent_step, comba_workspace_size, inputs
from test_gpu_chunk import GRADS, check_bwd, check_fwd

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dv,B,T,lengths,variant", [(256, 2, 300, None, "splr"),
                                                    (256, 1, None, [1, 63, 64, 65, 0, 200, 7], "splr"),
                                                    (384, 2, 130, None, "splr"),
                                                    (256, 2, 200, None, "iplr")])
def test_value_groups_forward_backward(dv, B, T, lengths, variant):
    kw = dict(lengths=lengths) if lengths else dict(B=B, T=T)
    w = inputs.make("custom", H=3, dk=128, dv=dv, dtype="bf16", with_b=True, with_h0=True, with_grads=True,
                    seed_offset=dv + (len(lengths) if lengths else T), **kw)
    t = to_dev(w)
    if variant == "splr":
        check_fwd(w, t)
        check_bwd(w, t)
        return
    o, hT = comba_chunk_fwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], b=t["b"], h0=t["h0"],
                            output_final_state=True, iplr=True)
    g = comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], b=t["b"], h0=t["h0"],
                        dhT=t["dhT"], iplr=True)
    torch.cuda.synchronize()
    ro, rhT = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0, variant="iplr")
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT, variant="iplr")
    g = {key: np64(val) for key, val in g.items()}
    errs = {"o": rel(np64(o), ro), "hT": rel(np64(hT), rhT)}
    errs.update({key: rel(g[key], r[key]) for key in GRADS})
    errs.update(param_grad_errors(g, r))
    bad = {key: e for key, e in errs.items() if not e <= tol("bf16")}
    assert not bad, (bad, errs)


def test_value_groups_reuse_equals_recompute():
    w = inputs.make("custom", B=2, T=200, H=2, dk=128, dv=256, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=5)
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], None, backward=True), dtype=torch.uint8, device="cuda")
    args = (t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"])
    comba_chunk_fwd(*args, b=t["b"], h0=t["h0"], output_final_state=True, workspace=ws, save_factors=True)
    g1 = comba_chunk_bwd(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"], workspace=ws, reuse_factors=True)
    g2 = comba_chunk_bwd(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"])
    torch.cuda.synchronize()
    for key in g1:
        assert np.array_equal(np64(g1[key]), np64(g2[key])), key


def test_value_groups_full_size():
    """B=4 T=4096 H=8 dk=128 dv=256 (the value-group benchmark shape) in the benchmark's
    configuration; every output against the oracle over the whole workload."""
    w = inputs.make("lm1p3b_v256")
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], None, backward=True), dtype=torch.uint8, device="cuda")
    args = (t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"])
    o, hT = comba_chunk_fwd(*args, b=t["b"], h0=t["h0"], output_final_state=True, workspace=ws, save_factors=True)
    g = comba_chunk_bwd(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"], workspace=ws, reuse_factors=True)
    torch.cuda.synchronize()
    g = {key: np64(val) for key, val in g.items()}
    o, hT = np64(o), np64(hT)
    del t, ws
    ro, rhT = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0)
    errs = {"o": rel(o, ro), "hT": rel(hT, rhT)}
    del ro, rhT
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT)
    errs.update({key: rel(g[key], r[key]) for key in GRADS})
    errs.update(param_grad_errors(g, r))
    ctx = param_grad_report(g, r, w.k, w.v, w.beta, w.b)
    print("lm1p3b_v256", {k_: f"{e:.2e}" for k_, e in errs.items()}, "context:", {k_: f"{e:.2e}" for k_, e in ctx.items()})
    bad = {key: e for key, e in errs.items() if not e <= tol("bf16")}
    assert not bad, (bad, errs, ctx)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_decode_dv256(dtype):
    Bd, H, dk, dv, steps = 5, 2, 128, 256, 5
    state = inputs.decode_state(Bd, H, dk, dv, seed_offset=9)
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    tok = lambda x: torch.from_numpy(np.ascontiguousarray(x)).cuda().to(tdt)
    f32 = lambda x: torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()
    st_gpu = f32(state)
    st_ref = state.astype(np.float64)
    for s in range(steps):
        q, k, v, a, be, d = inputs.decode_tokens(s, Bd, H, dk, dv, dtype)
        o = comba_recurrent_step(tok(q), tok(k), tok(v), f32(a), f32(be), f32(d), st_gpu)
        ro, st_ref = oracle.step(q, k, v, a, be, None, d, st_ref)
        torch.cuda.synchronize()
        assert rel(np64(o), ro) <= tol(dtype)
        assert rel(np64(st_gpu), st_ref) <= tol(dtype)


def test_value_groups_gated():
    """The gate and normalisation prologue with dv = 256: its q_hat, k_hat and gates serve both
    value heads, and their gradients are summed over them before the epilogue."""
    from test_gpu_gated import _check as gated_check, _run as gated_run
    w = inputs.make_gated(B=2, T=150, H=2, dk=128, dv=256, dtype="bf16", seed_offset=256, lengths=[100, 0, 129])
    gated_check(w, "splr", *gated_run(w, "splr"))


def test_value_groups_pk():
    """Comba-pk feedback vectors with dv = 256: dp is summed over the two value heads like dq and dk."""
    from test_gpu_pk import _check as pk_check, _run as pk_run, _with_p
    w = inputs.make("custom", B=2, T=170, H=2, dk=128, dv=256, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=77)
    p, tp = _with_p(w, seed=256)
    t = to_dev(w)
    pk_check(w, p, *pk_run(w, t, tp))
