"""Device-side wait limits reach the host (the boundary's COMBA_ERR_TIMEOUT).

Every wait of the tcgen05 and TMA kernels (tensor-core completion, TMA
arrival) is bounded in time; a wait that runs past the call's limit
(comba_shape_t.wait_limit_ns) makes its kernel let the copies and products in
flight land, skip the rest of its work and mark the workspace's status word,
which comba_workspace_status reads back.  No GPU fault is involved: the
diagnostic flag COMBA_DIAG_STALL points the first tensor-core completion wait
of every CTA of the prep, output and local-gradient kernels at a barrier that
nothing arrives at, so it runs out after the limit (100 us here) with the
CTA's products in flight.  The test checks that the forward and the backward
report COMBA_ERR_TIMEOUT through the C ABI, and that the next calls with the
default limit on the same workspace succeed and match the oracle.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import np64, param_grad_errors, rel, to_dev, tol
from paper_2506_02475_gb300 import binding, comba_chunk_bwd, comba_chunk_fwd, comba_workspace_size, inputs

pytestmark = pytest.mark.gpu

TIMEOUT = 5
DIAG_STALL = 32


def _p(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _status(ws):
    L = binding.lib()
    return L.comba_workspace_status(_p(ws), ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def test_wait_that_runs_out_reports_timeout_and_the_workspace_stays_usable():
    L = binding.lib()
    w = inputs.make("custom", B=2, T=1024, H=4, dk=128, dv=128, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=500)
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], None, backward=True), dtype=torch.uint8, device="cuda")
    nbytes = ws.numel()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    o = torch.empty_like(t["v"])
    hT = torch.empty_like(t["h0"])
    g = {key: torch.empty_like(t[src]) for key, src in (("dq", "q"), ("dk", "k"), ("dv", "v"), ("dalpha", "alpha"),
                                                          ("dbeta", "beta"), ("dd", "d"), ("db", "b"),
                                                          ("dh0", "h0"))}

    # forward saving factors, its first completion waits running out after 100 us
    shape = binding.make_shape(t["q"], t["v"], None, None, binding.COMBA_SAVE_FACTORS | DIAG_STALL, 100_000)
    st = L.comba_chunk_fwd(ctypes.byref(shape), _p(t["q"]), _p(t["k"]), _p(t["v"]), _p(t["alpha"]), _p(t["beta"]),
                           _p(t["b"]), _p(t["d"]), _p(t["h0"]), _p(o), _p(hT), _p(ws), nbytes, stream)
    assert st == 0                      # the launch itself is fine; the wait's fate shows in the status word
    assert _status(ws) == TIMEOUT

    # a backward recomputing the factors, the same way
    shape = binding.make_shape(t["q"], t["v"], None, None, DIAG_STALL, 100_000)
    st = L.comba_chunk_bwd(ctypes.byref(shape), _p(t["q"]), _p(t["k"]), _p(t["v"]), _p(t["alpha"]), _p(t["beta"]),
                           _p(t["b"]), _p(t["d"]), _p(t["h0"]), _p(t["dO"]), _p(t["dhT"]), _p(g["dq"]), _p(g["dk"]),
                           _p(g["dv"]), _p(g["dalpha"]), _p(g["dbeta"]), _p(g["db"]), _p(g["dd"]), _p(g["dh0"]),
                           _p(ws), nbytes, stream)
    assert st == 0
    assert _status(ws) == TIMEOUT

    # the same workspace with the default limit: the status clears and the results are the oracle's
    args = (t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"])
    o, hT = comba_chunk_fwd(*args, b=t["b"], h0=t["h0"], output_final_state=True, workspace=ws, save_factors=True)
    gg = comba_chunk_bwd(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"], workspace=ws, reuse_factors=True)
    assert _status(ws) == 0
    torch.cuda.synchronize()
    ro, rhT = oracle.fwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, h0=w.h0)
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT)
    gg = {key: np64(val) for key, val in gg.items()}
    errs = {"o": rel(np64(o), ro), "hT": rel(np64(hT), rhT)}
    errs.update({key: rel(gg[key], r[key]) for key in ("dq", "dk", "dv", "dalpha", "dbeta", "dh0")})
    errs.update(param_grad_errors(gg, r))
    bad = {key: e for key, e in errs.items() if not e <= tol(w.dtype)}
    assert not bad, (bad, errs)


def test_default_limit_leaves_the_status_clear():
    w = inputs.make("custom", B=1, T=300, H=2, dk=128, dv=128, dtype="bf16", with_b=True, with_h0=True,
                    with_grads=True, seed_offset=501)
    t = to_dev(w)
    ws = torch.empty(comba_workspace_size(t["q"], t["v"], None, backward=True), dtype=torch.uint8, device="cuda")
    args = (t["q"], t["k"], t["v"], t["alpha"], t["beta"], t["d"])
    comba_chunk_fwd(*args, b=t["b"], h0=t["h0"], output_final_state=True, workspace=ws, save_factors=True)
    comba_chunk_bwd(*args, t["dO"], b=t["b"], h0=t["h0"], dhT=t["dhT"], workspace=ws, reuse_factors=True)
    assert _status(ws) == 0
