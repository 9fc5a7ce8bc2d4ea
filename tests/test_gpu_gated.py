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


def _head(w, h):
    """The raw workload restricted to head h (every sequence), for the oracle."""
    def tok(x):
        return None if x is None else np.ascontiguousarray(x[..., h:h + 1, :])

    def gate(x):
        return np.ascontiguousarray(x[..., h:h + 1])

    def st(x):
        return None if x is None else np.ascontiguousarray(x[:, h:h + 1])

    return inputs.GatedWorkload(dtype=w.dtype, q=tok(w.q), k=tok(w.k), v=tok(w.v), g_alpha=gate(w.g_alpha),
                                g_beta=gate(w.g_beta), a=w.a[h:h + 1], c=w.c[h:h + 1], b_raw=w.b_raw[h:h + 1],
                                d=w.d[h:h + 1], h0=st(w.h0), dO=tok(w.dO), dhT=st(w.dhT), cu_seqlens=w.cu_seqlens)


def _check(w, variant, o, hT, g):
    """Every output against the oracle composition on w (all of its heads)."""
    raw = (w.q, w.k, w.v, w.g_alpha, w.g_beta, w.a, w.c, w.b_raw, w.d)
    ro, rhT = gated.fwd(*raw, h0=w.h0, cu_seqlens=w.cu_seqlens, variant=variant)
    r = gated.bwd(*raw, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens, variant=variant)
    tl = tol(w.dtype)
    errs = {"o": rel(o, ro), "hT": rel(hT, rhT)}
    for key in ("dq", "dk", "dv", "dg_alpha", "dg_beta", "dh0"):
        errs[key] = rel(g[key], r[key])
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
        errs[key] = rel_sum(g[key], r[key], sc)
    bad = {key: e for key, e in errs.items() if not e <= tl}
    assert not bad, (bad, errs)


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


def test_gated_full_size_sampled_heads():
    """B=4 T=4096 H=16 d=128 bf16 (the gated benchmark's shape and launch configuration):
    every sequence of two sampled heads against the oracle, forward and backward."""
    w = inputs.make_gated(B=4, T=4096, H=16, dk=128, dv=128, dtype="bf16")
    o, hT, g = _run(w, "splr")
    for h in (0, 15):
        sl = lambda x: x[..., h:h + 1, :]
        gs = {key: (g[key][..., h:h + 1, :] if g[key].ndim == 4 and key != "dh0" else
                    g[key][:, h:h + 1] if key == "dh0" else
                    g[key][..., h:h + 1] if g[key].ndim == 3 else g[key][h:h + 1]) for key in g}
        _check(_head(w, h), "splr", sl(o), hT[:, h:h + 1], gs)
