"""GPU parity at head dim dk = 256 (bf16): value heads 64 wide (dv = 64, 128, 192 or 256 as one to
four value heads per key head), the mma.sync chunk kernels and the scan that applies E = U - W H
per chunk (no dk x dk chunk map).  Compared with the oracle, which takes any dk, dv directly."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import np64, param_grad_errors, param_grad_report, rel, tol, to_dev
from paper_2506_02475_gb300 import comba_chunk_bwd, comba_chunk_fwd, comba_recurrent_step, comba_workspace_size, inputs
from test_gpu_chunk import GRADS, check_bwd, check_fwd

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("dv,B,T,lengths", [(64, 2, 300, None), (128, 2, 200, None), (256, 1, 330, None),
                                            (192, 1, None, [1, 63, 64, 65, 0, 200, 7]),
                                            (256, 1, None, [129, 3, 64])])
def test_head_dim_256_forward_backward(dv, B, T, lengths):
    # four heads: the per-head sums db and dd are checked with the max-norm over their heads, which
    # over two heads of a few hundred tokens rests on two sums that may both nearly cancel
    kw = dict(lengths=lengths) if lengths else dict(B=B, T=T)
    w = inputs.make("custom", H=4, dk=256, dv=dv, dtype="bf16", with_b=True, with_h0=True, with_grads=True,
                    seed_offset=dv + (len(lengths) if lengths else T), **kw)
    t = to_dev(w)
    check_fwd(w, t)
    check_bwd(w, t)


def test_head_dim_256_iplr():
    w = inputs.make("custom", B=2, T=150, H=2, dk=256, dv=128, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=31)
    t = to_dev(w)
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


def test_head_dim_256_without_initial_state():
    """h0 and dhT absent (zero states in and out of the scan), b absent (b = 1)."""
    w = inputs.make("custom", B=1, T=257, H=3, dk=256, dv=64, dtype="bf16", with_h0=False, with_grads=True,
                    seed_offset=77)
    w.dhT = None
    t = to_dev(w)
    check_fwd(w, t)
    check_bwd(w, t)


def test_head_dim_256_reuse_equals_recompute():
    w = inputs.make("custom", B=2, T=200, H=2, dk=256, dv=256, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=8)
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], None, backward=True), dtype=torch.uint8, device="cuda")
    args = (t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"])
    comba_chunk_fwd(*args, b=t["b"], h0=t["h0"], output_final_state=True, workspace=ws, save_factors=True)
    g1 = comba_chunk_bwd(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"], workspace=ws, reuse_factors=True)
    g2 = comba_chunk_bwd(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"])
    torch.cuda.synchronize()
    for key in g1:
        assert np.array_equal(np64(g1[key]), np64(g2[key])), key


def test_head_dim_256_full_size():
    """B=4 T=4096 H=8 dk=dv=256 (the head-dim-256 benchmark shape) in the benchmark's
    configuration; every output against the oracle over the whole workload."""
    w = inputs.make("lm1p3b_d256")
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
    print("lm1p3b_d256", {k_: f"{e:.2e}" for k_, e in errs.items()}, "context:", {k_: f"{e:.2e}" for k_, e in ctx.items()})
    bad = {key: e for key, e in errs.items() if not e <= tol("bf16")}
    assert not bad, (bad, errs, ctx)


@pytest.mark.parametrize("dtype,dv", [("bf16", 256), ("bf16", 64), ("f32", 128)])
def test_decode_head_dim_256(dtype, dv):
    Bd, H, dk, steps = 5, 2, 256, 5
    state = inputs.decode_state(Bd, H, dk, dv, seed_offset=19)
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
