"""GPU parity of the chunk-parallel forward and backward against the fp64 oracle.

Every comparison runs the CUDA library through its C ABI (ctypes binding) on
seeded synthetic inputs and the oracle on the very same values.  Small cases
span several 64-token chunks with ragged tails; the full-size workloads run
the whole problem on the GPU exactly as the benchmark does, and are compared
on every sequence and head (the oracle takes seconds on a many-core host).
"""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import np64, param_grad_errors, param_grad_report, rel, to_dev, tol
from paper_2506_02475_gb300 import comba_chunk_bwd, comba_chunk_fwd, inputs

pytestmark = pytest.mark.gpu

GRADS = ("dq", "dk", "dv", "dalpha", "dbeta", "dh0")


def gpu_fwd(t):
    o, hT = comba_chunk_fwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], b=t["b"], h0=t["h0"],
                            cu_seqlens=t["cu_seqlens"], output_final_state=True)
    torch.cuda.synchronize()
    return np64(o), np64(hT)


def gpu_bwd(t):
    g = comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], b=t["b"], h0=t["h0"],
                        dhT=t["dhT"], cu_seqlens=t["cu_seqlens"])
    torch.cuda.synchronize()
    return {key: np64(val) for key, val in g.items()}


def check_fwd(w, t=None, report=None):
    t = t or to_dev(w)
    o, hT = gpu_fwd(t)
    ro, rhT = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0, cu_seqlens=w.cu_seqlens)
    errs = {"o": rel(o, ro), "hT": rel(hT, rhT)}
    if report is not None:
        report.update(errs)
    for key, e in errs.items():
        assert e <= tol(w.dtype), (key, e)


def check_bwd(w, t=None):
    t = t or to_dev(w)
    g = gpu_bwd(t)
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens)
    errs = {key: rel(g[key], r[key]) for key in GRADS}
    errs.update(param_grad_errors(g, r))
    bad = {k_: e for k_, e in errs.items() if not e <= tol(w.dtype)}
    assert not bad, (bad, errs, param_grad_report(g, r, w.k, w.v, w.beta, w.b))
    return errs


def test_tiny_fp32_forward_workload():
    """B=1, H=2, T=256, d=64, fp32, d=0.5, zero state: forward only, 1e-4."""
    w = inputs.make("tiny_fp32")
    check_fwd(w)


SMALL = [
    # dtype, dk, dv, B, T, with_b, with_h0
    ("f32", 64, 64, 2, 200, True, True),
    ("f32", 128, 128, 1, 130, False, True),
    ("f32", 64, 128, 1, 65, True, False),
    ("f32", 128, 64, 2, 1, True, True),
    ("bf16", 128, 128, 2, 300, True, True),
    ("bf16", 64, 64, 3, 64, False, False),
    ("bf16", 128, 64, 2, 1, True, True),
    ("bf16", 64, 128, 1, 127, True, True),
]


@pytest.mark.parametrize("dtype,dk,dv,B,T,with_b,with_h0", SMALL)
def test_forward_small(dtype, dk, dv, B, T, with_b, with_h0):
    w = inputs.make("custom", B=B, T=T, H=3, dk=dk, dv=dv, dtype=dtype, with_b=with_b, with_h0=with_h0,
                    seed_offset=T + dk)
    check_fwd(w)


BWD_SMALL = [
    ("f32", 64, 64, 2, 200, True, True),
    ("f32", 64, 64, 1, 64, False, False),
    ("bf16", 128, 128, 2, 300, True, True),
    ("bf16", 64, 64, 1, 130, False, True),
    ("bf16", 128, 64, 2, 70, True, False),
    ("bf16", 64, 128, 1, 1, True, True),
]


@pytest.mark.parametrize("dtype,dk,dv,B,T,with_b,with_h0", BWD_SMALL)
def test_backward_small(dtype, dk, dv, B, T, with_b, with_h0):
    w = inputs.make("custom", B=B, T=T, H=2, dk=dk, dv=dv, dtype=dtype, with_b=with_b, with_h0=with_h0,
                    with_grads=True, seed_offset=3 * T + dv)
    check_bwd(w)


@pytest.mark.parametrize("dtype,d", [("bf16", 128), ("f32", 64)])
def test_varlen_small_with_empty_and_ragged_sequences(dtype, d):
    """Packed sequences of length 1, 63, 64, 65, 0, 200, 7: state resets at every start,
    an empty sequence passes h0 through to hT (and dhT to dh0)."""
    lens = [1, 63, 64, 65, 0, 200, 7]
    w = inputs.make("custom", H=2, dk=d, dv=d, dtype=dtype, with_b=True, with_h0=True, with_grads=True,
                    lengths=lens, seed_offset=17)
    t = to_dev(w)
    check_fwd(w, t)
    check_bwd(w, t)


@pytest.mark.parametrize("dk,dv", [(128, 128), (256, 128)])
def test_nonfinite_inputs_stay_inside_their_packed_sequence(dk, dv):
    """Packed sequences [100, 70, 129] with k and dO = +inf on every token of the middle one:
    the other sequences' outputs, final states, token gradients and dh0 stay finite and match
    the oracle.  Their short last chunks cover the next sequence's (or no) tokens, so every
    kernel that reads a chunk tile, the scans' key and dO tiles included, must mask the rows
    past the sequence end.  Head dim 128 (tcgen05 kernels) and 256 (two value heads of 64)."""
    lens = [100, 70, 129]
    w = inputs.make("custom", H=2, dk=dk, dv=dv, dtype="bf16", with_b=True, with_h0=True, with_grads=True,
                    lengths=lens, seed_offset=41)
    cu = w.cu_seqlens
    mid = slice(int(cu[1]), int(cu[2]))
    keep = np.ones(int(cu[-1]), bool)
    keep[mid] = False
    k_ref, dO_ref = w.k.copy(), w.dO.copy()
    k_ref[mid] = 0.0
    dO_ref[mid] = 0.0
    w.k[mid] = np.inf
    w.dO[mid] = np.inf
    t = to_dev(w)
    o, hT = gpu_fwd(t)
    ro, rhT = oracle.fwd(w.q, k_ref, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0, cu_seqlens=cu)
    assert np.all(np.isfinite(o[keep])) and rel(o[keep], ro[keep]) <= tol(w.dtype)
    assert np.all(np.isfinite(hT[[0, 2]])) and rel(hT[[0, 2]], rhT[[0, 2]]) <= tol(w.dtype)
    g = gpu_bwd(t)
    r = oracle.bwd(w.q, k_ref, w.v, w.alpha, w.beta, w.b, w.d, dO_ref, h0=w.h0, dhT=w.dhT, cu_seqlens=cu)
    for key in ("dq", "dk", "dv", "dalpha", "dbeta"):
        x, ref = g[key][keep], r[key][keep]
        assert np.all(np.isfinite(x)), key
        assert rel(x, ref) <= tol(w.dtype), key
    x, ref = g["dh0"][[0, 2]], r["dh0"][[0, 2]]
    assert np.all(np.isfinite(x)) and rel(x, ref) <= tol(w.dtype)


def test_backward_is_bitwise_deterministic():
    w = inputs.make("custom", B=2, T=260, H=2, dk=128, dv=128, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=5)
    t = to_dev(w)
    a = gpu_bwd(t)
    b = gpu_bwd(t)
    for key in a:
        assert np.array_equal(a[key], b[key]), key
    o1, h1 = gpu_fwd(t)
    o2, h2 = gpu_fwd(t)
    assert np.array_equal(o1, o2) and np.array_equal(h1, h2)


@pytest.mark.parametrize("name", ["lm340m", "lm1p3b", "varlen64k"])
def test_full_size_workload(name):
    """The full workload on the GPU in the benchmark's launch configuration (forward
    saving its factors, backward reusing them), every output against the oracle over
    the whole workload (every sequence and head), forward and backward.  dd and db are
    checked over all their heads like every other tensor; their per-head figures are
    printed for context."""
    from paper_2506_02475_gb300 import comba_workspace_size
    w = inputs.make(name)
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], t["cu_seqlens"], backward=True), dtype=torch.uint8,
                     device="cuda")
    o, hT = comba_chunk_fwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], b=t["b"], h0=t["h0"],
                            cu_seqlens=t["cu_seqlens"], output_final_state=True, workspace=ws, save_factors=True)
    g = comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], b=t["b"], h0=t["h0"],
                        dhT=t["dhT"], cu_seqlens=t["cu_seqlens"], workspace=ws, reuse_factors=True)
    torch.cuda.synchronize()
    g = {key: np64(val) for key, val in g.items()}
    o, hT = np64(o), np64(hT)
    del t, ws
    ro, rhT = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0, cu_seqlens=w.cu_seqlens)
    errs = {"o": rel(o, ro), "hT": rel(hT, rhT)}
    del ro, rhT
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens)
    errs.update({key: rel(g[key], r[key]) for key in GRADS})
    errs.update(param_grad_errors(g, r))
    ctx = param_grad_report(g, r, w.k, w.v, w.beta, w.b)
    print(name, {k_: f"{e:.2e}" for k_, e in errs.items()}, "context:", {k_: f"{e:.2e}" for k_, e in ctx.items()})
    bad = {k_: e for k_, e in errs.items() if not e <= tol(w.dtype)}
    assert not bad, (name, bad, errs, ctx)


@pytest.mark.parametrize("dtype,d,lens", [("bf16", 128, None), ("f32", 64, None), ("bf16", 64, [70, 0, 129, 5])])
def test_backward_reusing_saved_forward_factors(dtype, d, lens):
    """fwd(save_factors) + bwd(reuse_factors) gives bitwise the same gradients as a
    backward that recomputes the factors, and matches the oracle."""
    from paper_2506_02475_gb300 import comba_workspace_size
    w = inputs.make("custom", B=2, T=200, H=2, dk=d, dv=d, dtype=dtype, with_b=True, with_h0=True, with_grads=True,
                    lengths=lens, seed_offset=23)
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], t["cu_seqlens"], backward=True), dtype=torch.uint8,
                     device="cuda")
    o, hT = comba_chunk_fwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], b=t["b"], h0=t["h0"],
                            cu_seqlens=t["cu_seqlens"], output_final_state=True, workspace=ws, save_factors=True)
    g = comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], b=t["b"], h0=t["h0"],
                        dhT=t["dhT"], cu_seqlens=t["cu_seqlens"], workspace=ws, reuse_factors=True)
    torch.cuda.synchronize()
    g = {key: np64(val) for key, val in g.items()}
    ref = gpu_bwd(t)
    for key in ref:
        assert np.array_equal(g[key], ref[key]), key
    o2, hT2 = gpu_fwd(t)
    assert np.array_equal(np64(o), o2) and np.array_equal(np64(hT), hT2)
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens)
    for key in GRADS:
        assert rel(g[key], r[key]) <= tol(w.dtype), key
    for key, e in param_grad_errors(g, r).items():
        assert e <= tol(w.dtype), key


@pytest.mark.parametrize("dtype,d,lens", [("bf16", 128, [130, 0, 257, 64]), ("bf16", 64, None), ("f32", 64, [70, 5, 133])])
def test_iplr_variant_forward_backward(dtype, d, lens):
    """Comba-iplr (transition alpha (I - 2 btilde k k^T)) through the same kernels, forward and backward,
    including the saved-factor step, against the oracle's iplr variant."""
    from paper_2506_02475_gb300 import comba_workspace_size
    w = inputs.make("custom", B=2, T=200, H=3, dk=d, dv=d, dtype=dtype, with_b=True, with_h0=True, with_grads=True,
                    lengths=lens, seed_offset=61)
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], t["cu_seqlens"], backward=True), dtype=torch.uint8,
                     device="cuda")
    o, hT = comba_chunk_fwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], b=t["b"], h0=t["h0"],
                            cu_seqlens=t["cu_seqlens"], output_final_state=True, workspace=ws, save_factors=True,
                            iplr=True)
    g = comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], b=t["b"], h0=t["h0"],
                        dhT=t["dhT"], cu_seqlens=t["cu_seqlens"], workspace=ws, reuse_factors=True, iplr=True)
    g2 = comba_chunk_bwd(t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"], t["dO"], b=t["b"], h0=t["h0"],
                         dhT=t["dhT"], cu_seqlens=t["cu_seqlens"], iplr=True)
    torch.cuda.synchronize()
    ro, rhT = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0, cu_seqlens=w.cu_seqlens, variant="iplr")
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT, cu_seqlens=w.cu_seqlens,
                   variant="iplr")
    assert rel(np64(o), ro) <= tol(dtype)
    assert rel(np64(hT), rhT) <= tol(dtype)
    gn = {key: np64(val) for key, val in g.items()}
    for key in GRADS:
        assert np.array_equal(gn[key], np64(g2[key])), key          # reuse == recompute, bitwise
        assert rel(gn[key], r[key]) <= tol(dtype), (key, rel(gn[key], r[key]))
    for key, e in param_grad_errors(gn, r).items():
        assert e <= tol(dtype), (key, e)
    # and it is not the SPLR result
    ro_s, _ = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0, cu_seqlens=w.cu_seqlens)
    assert rel(np64(o), ro_s) > 2 * tol(dtype)


def test_single_long_sequence():
    """One sequence of 32768 tokens (512 chunks through each scan), bf16 d=128, two heads:
    forward and backward against the oracle."""
    w = inputs.make("custom", B=1, T=32768, H=2, dk=128, dv=128, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=77)
    t = to_dev(w)
    check_fwd(w, t)
    check_bwd(w, t)


def test_thousands_of_tiny_sequences():
    """1200 packed sequences of 0-5 tokens: far more sequences than chunks of work, every chunk
    ragged, many empty sequences passing h0 through."""
    lens = np.random.default_rng(11).integers(0, 6, 1200).tolist()
    w = inputs.make("custom", H=2, dk=128, dv=128, dtype="bf16", with_b=True, with_h0=True, with_grads=True,
                    lengths=lens, seed_offset=23)
    t = to_dev(w)
    check_fwd(w, t)
    check_bwd(w, t)
