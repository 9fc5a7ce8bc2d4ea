"""GPU parity of the gate and normalisation prologue path (comba_chunk_fwd_gated / _bwd_gated)
against the oracle composition (oracle.gated): raw q, k; alpha = exp(-a softplus(g_alpha + c)),
beta = sigmoid(g_beta), b = sigmoid(b_raw)."""
import numpy as np
import pytest
import torch

from gpu_helpers import np64, rel, tol
from oracle import gated
from paper_2506_02475_gb300 import comba_chunk_bwd_gated, comba_chunk_fwd_gated, inputs

pytestmark = pytest.mark.gpu


def _dev(w):
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32

    def tok(x):
        return torch.from_numpy(np.ascontiguousarray(x)).cuda().to(tdt)

    def f32(x):
        return None if x is None else torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()

    t = dict(q=tok(w.q), k=tok(w.k), v=tok(w.v), dO=tok(w.dO))
    for key in ("g_alpha", "g_beta", "a", "c", "b_raw", "d", "h0", "dhT"):
        t[key] = f32(getattr(w, key))
    t["cu_seqlens"] = None if w.cu_seqlens is None else torch.from_numpy(w.cu_seqlens.astype(np.int32)).cuda()
    return t


def _run(w, variant):
    """Forward (saving factors) + backward (reusing them) and a recomputing backward, as bench.py runs them."""
    from paper_2506_02475_gb300 import binding
    t = _dev(w)
    iplr = variant == "iplr"
    shape = binding.make_shape(t["q"], t["v"], t["cu_seqlens"], None, binding.COMBA_GATED)
    ws = torch.empty(binding.lib().comba_workspace_size(binding.ctypes.byref(shape), 1), dtype=torch.uint8,
                     device="cuda")
    args = (t["q"], t["k"], t["v"], t["g_alpha"], t["g_beta"], t["a"], t["c"], t["b_raw"], t["d"])
    o, hT = comba_chunk_fwd_gated(*args, h0=t["h0"], cu_seqlens=t["cu_seqlens"], output_final_state=True,
                                  workspace=ws, save_factors=True, iplr=iplr)
    g = comba_chunk_bwd_gated(*args, t["dO"], h0=t["h0"], dhT=t["dhT"], cu_seqlens=t["cu_seqlens"], workspace=ws,
                              reuse_factors=True, iplr=iplr)
    del ws
    g2 = comba_chunk_bwd_gated(*args, t["dO"], h0=t["h0"], dhT=t["dhT"], cu_seqlens=t["cu_seqlens"], iplr=iplr)
    torch.cuda.synchronize()
    g = {key: np64(val) for key, val in g.items()}
    for key in ("dq", "dk", "dv", "dg_alpha", "dg_beta", "dh0"):
        assert np.array_equal(g[key], np64(g2[key])), key             # reuse == recompute, bitwise
    return np64(o), np64(hT), g


def _check(w, variant, o, hT, g):
    """Every output against the oracle composition on w (all of its heads)."""
    raw = (w.q, w.k, w.v, w.g_alpha, w.g_beta, w.a, w.c, w.b_raw, w.d)
    ro, rhT = gated.fwd(*raw, h0=w.h0, cu_seqlens=w.cu_seqlens, variant=variant)
    r = gated.bwd(*raw, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens, variant=variant)
    tl = tol(w.dtype)
    errs = {"o": rel(o, ro), "hT": rel(hT, rhT)}
    for key in ("dq", "dk", "dv", "dg_alpha", "dg_beta", "dh0"):
        errs[key] = rel(g[key], r[key])
    # the per-head parameter gradients take the max-norm error over their heads like every tensor
    for key in ("da", "dc", "dd", "db_raw"):
        errs[key] = rel(g[key], r[key])
    bad = {key: e for key, e in errs.items() if not e <= tl}
    assert not bad, (bad, errs)
    return errs


@pytest.mark.parametrize("dtype,d,dv,lens,variant", [("bf16", 128, 128, [130, 0, 257, 64], "splr"),
                                                      ("bf16", 128, 128, None, "iplr"),
                                                      ("f32", 64, 64, [70, 5, 133], "splr"),
                                                      # head dim 256: two value heads of width 64, and
                                                      # the epilogue's two passes (q, then k)
                                                      ("bf16", 256, 128, [130, 0, 77], "splr")])
def test_gated_forward_backward(dtype, d, dv, lens, variant):
    w = inputs.make_gated(B=2, T=200, H=3, dk=d, dv=dv, dtype=dtype, seed_offset=d + len(lens or []), lengths=lens)
    _check(w, variant, *_run(w, variant))


def test_gated_many_heads():
    """H = 300: the per-head gate b and the per-head sums span several blocks of heads; 70 tokens
    leave a ragged tail in every 64-row stage split and token block of the reductions."""
    w = inputs.make_gated(B=1, T=70, H=300, dk=64, dv=64, dtype="f32", seed_offset=300)
    _check(w, "splr", *_run(w, "splr"))


def test_gated_full_size():
    """B=4 T=4096 H=16 d=128 bf16 (the gated benchmark's shape and launch configuration):
    every output against the oracle over the whole workload, forward and backward."""
    w = inputs.make_gated(B=4, T=4096, H=16, dk=128, dv=128, dtype="bf16")
    o, hT, g = _run(w, "splr")
    print("gated lm1p3b", {k_: f"{e:.2e}" for k_, e in _check(w, "splr", o, hT, g).items()})
