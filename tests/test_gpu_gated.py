"""GPU parity of the gate and normalisation prologue path (comba_chunk_fwd_gated / _bwd_gated)
against the oracle composition (oracle.gated): raw q, k; alpha = exp(-a softplus(g_alpha + c)),
beta = sigmoid(g_beta), b = sigmoid(b_raw)."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import np64, rel, rel_sum, tol
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


@pytest.mark.parametrize("dtype,d,lens,variant", [("bf16", 128, [130, 0, 257, 64], "splr"),
                                                   ("bf16", 128, None, "iplr"),
                                                   ("f32", 64, [70, 5, 133], "splr")])
def test_gated_forward_backward(dtype, d, lens, variant):
    from paper_2506_02475_gb300 import binding
    w = inputs.make_gated(B=2, T=200, H=3, dk=d, dv=d, dtype=dtype, seed_offset=d + len(lens or []), lengths=lens)
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
    g2 = comba_chunk_bwd_gated(*args, t["dO"], h0=t["h0"], dhT=t["dhT"], cu_seqlens=t["cu_seqlens"], iplr=iplr)
    torch.cuda.synchronize()
    raw = (w.q, w.k, w.v, w.g_alpha, w.g_beta, w.a, w.c, w.b_raw, w.d)
    ro, rhT = gated.fwd(*raw, h0=w.h0, cu_seqlens=w.cu_seqlens, variant=variant)
    r = gated.bwd(*raw, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens, variant=variant)
    tl = tol(dtype)
    assert rel(np64(o), ro) <= tl
    assert rel(np64(hT), rhT) <= tl
    gn = {key: np64(val) for key, val in g.items()}
    for key in ("dq", "dk", "dv", "dg_alpha", "dg_beta", "dh0"):
        assert np.array_equal(gn[key], np64(g2[key])), key             # reuse == recompute, bitwise
        assert rel(gn[key], r[key]) <= tl, (key, rel(gn[key], r[key]))
    # per-head sums on the scale of their per-token contributions, all from the oracle
    qh, kh, al, be, b = gated.prologue(w.q, w.k, w.g_alpha, w.g_beta, w.a, w.c, w.b_raw)
    inner = oracle.bwd(qh, kh, w.v, al, be, b, w.d, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens,
                       variant=variant)
    z = w.g_alpha.astype(np.float64) + w.c
    H = w.g_alpha.shape[-1]
    scale = {
        "da": np.abs(inner["dalpha"] * al * gated.softplus(z)).reshape(-1, H).sum(0),
        "dc": np.abs(r["dg_alpha"]).reshape(-1, H).sum(0),
        "dd": np.abs(np.einsum("...hd,...hd->...h", kh, inner["dq"])).reshape(-1, H).sum(0),
        "db_raw": (np.abs(be * inner["dbeta"] - np.einsum("...hd,...hd->...h", w.v, inner["dv"])).reshape(-1, H)
                   .sum(0) * (1.0 - b)),
    }
    for key, sc in scale.items():
        e = rel_sum(gn[key], r[key], sc)
        assert e <= tl, (key, e)
