"""GPU parity on the method's degenerate gate values, forward and backward, on the tcgen05
path (bf16, d = 128), the fp32 path (d = 64) and head dim 256 (bf16, dk = 256, dv = 128: two
value heads of width 64 on the mma.sync kernels and the E-form scan):
  * alpha = 1: no decay (chunk log-decays all zero);
  * beta = 0: nothing is written, the output reads the decayed initial state only;
  * b = 0: no state feedback (gated linear attention);
  * d = 0: no output correction;
  * alpha = 1e-3: decay so strong that gamma underflows inside a chunk (log-decays down to
    about -440), which the masked exp-of-difference form must survive without inf or NaN.

dalpha is reached through d log alpha_j = alpha_j dalpha_j, a sum of pair terms of the chunk
whose decay factors can be ~1 (tokens with alpha = 1 between them) and cancel pairwise; fp32
rounding of those O(1) terms is then amplified by 1 / alpha_j.  Where alpha_min < 0.1 the fp32
dalpha bound is max(1e-4, C u_32 / alpha_min) with C = 64 and u_32 = 2^-24 (3.8e-3 at 1e-3)."""
import numpy as np
import pytest

import oracle
from gpu_helpers import param_grad_errors, rel, tol, to_dev
from paper_2506_02475_gb300 import inputs
from test_gpu_chunk import GRADS, check_fwd, gpu_bwd

pytestmark = pytest.mark.gpu

CASES = {
    "no_decay": dict(alpha=1.0),
    "no_write": dict(beta=0.0),
    "no_feedback": dict(b=0.0),
    "no_correction": dict(d=0.0),
    "vanishing_decay": dict(alpha=1e-3),
    "mixed_extremes": dict(alpha="mixed"),
}


def _workload(dtype, dk, dv, case):
    w = inputs.make("custom", B=2, T=150, H=2, dk=dk, dv=dv, dtype=dtype, with_b=True, with_h0=True, with_grads=True,
                    seed_offset=29)
    for key, val in CASES[case].items():
        if key in ("alpha", "beta"):
            arr = getattr(w, key)
            if val == "mixed":   # per token either 1, 1e-3 or an ordinary gate
                rng = np.random.default_rng(3)
                pick = rng.integers(0, 3, arr.shape)
                arr = np.where(pick == 0, 1.0, np.where(pick == 1, 1e-3, arr)).astype(np.float32)
            else:
                arr = np.full_like(arr, val)
            setattr(w, key, arr)
        else:
            setattr(w, key, np.full_like(getattr(w, key), val))
    return w


@pytest.mark.parametrize("case", sorted(CASES))
@pytest.mark.parametrize("dtype,dk,dv", [("bf16", 128, 128), ("f32", 64, 64), ("bf16", 256, 128)])
def test_degenerate_gates(dtype, dk, dv, case):
    w = _workload(dtype, dk, dv, case)
    t = to_dev(w)
    check_fwd(w, t)
    g = gpu_bwd(t)
    r = oracle.bwd(w.q, w.k, w.v, w.alpha, w.beta, w.b, w.d, w.dO, h0=w.h0, dhT=w.dhT)
    errs = {key: rel(g[key], r[key]) for key in GRADS}
    for key in GRADS:
        assert np.all(np.isfinite(g[key])), key
    errs.update(param_grad_errors(g, r))
    if case == "no_write":
        # beta = 0: db is exactly zero on both sides
        assert np.array_equal(g["db"], r["db"])
    bound = {key: tol(w.dtype) for key in errs}
    amin = float(np.min(w.alpha))
    if w.dtype == "f32" and amin < 0.1:
        bound["dalpha"] = max(tol(w.dtype), 64 * 2.0 ** -24 / amin)
    bad = {key: e for key, e in errs.items() if not e <= bound[key]}
    assert not bad, (case, bad, errs)
