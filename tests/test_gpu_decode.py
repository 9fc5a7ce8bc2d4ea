"""GPU parity of the one-token recurrent step against the oracle."""
import numpy as np
import pytest
import torch

import oracle
from gpu_helpers import TOL_BF16, TOL_F32, np64, rel
from paper_2506_02475_gb300 import comba_recurrent_step, inputs

pytestmark = pytest.mark.gpu


def _tok(x, dtype):
    return torch.from_numpy(np.ascontiguousarray(x)).cuda().to(torch.bfloat16 if dtype == "bf16" else torch.float32)


def _f32(x):
    return torch.from_numpy(np.ascontiguousarray(x, np.float32)).cuda()


@pytest.mark.parametrize("dtype,dk,dv,with_b", [("f32", 64, 64, True), ("f32", 128, 128, False),
                                                 ("bf16", 128, 64, True), ("bf16", 64, 128, False),
                                                 ("bf16", 128, 128, True)])
def test_decode_steps_small(dtype, dk, dv, with_b):
    Bd, H, steps = 5, 3, 6
    state = inputs.decode_state(Bd, H, dk, dv, seed_offset=dk + dv)
    b = np.random.default_rng(1).uniform(0, 1, H).astype(np.float32) if with_b else None
    st_gpu = _f32(state)
    st_ref = state.astype(np.float64)
    for s in range(steps):
        q, k, v, a, be, d = inputs.decode_tokens(s, Bd, H, dk, dv, dtype)
        o = comba_recurrent_step(_tok(q, dtype), _tok(k, dtype), _tok(v, dtype), _f32(a), _f32(be), _f32(d), st_gpu,
                                 b=None if b is None else _f32(b))
        ro, st_ref = oracle.step(q, k, v, a, be, b, d, st_ref)
        torch.cuda.synchronize()
        tl = TOL_BF16 if dtype == "bf16" else TOL_F32
        assert rel(np64(o), ro) <= tl
        assert rel(np64(st_gpu), st_ref) <= tl


def test_decode_workload_1024_steps_sampled_rows():
    """Bd=256, H=16, d=128, bf16 tokens with an fp32 state, 1024 sequential steps on the
    GPU; rows 0 and 255 (all heads) follow the oracle step by step."""
    Bd, H, dk, dv, steps = 256, 16, 128, 128, 1024
    rows = [0, 255]
    state = inputs.decode_state(Bd, H, dk, dv)
    st_gpu = _f32(state)
    st_ref = state[rows].astype(np.float64)
    worst_o = 0.0
    for s in range(steps):
        q, k, v, a, be, d = inputs.decode_tokens(s, Bd, H, dk, dv, "bf16")
        o = comba_recurrent_step(_tok(q, "bf16"), _tok(k, "bf16"), _tok(v, "bf16"), _f32(a), _f32(be), _f32(d),
                                 st_gpu)
        ro, st_ref = oracle.step(q[rows], k[rows], v[rows], a[rows], be[rows], None, d, st_ref)
        if s % 64 == 0 or s == steps - 1:
            worst_o = max(worst_o, rel(np64(o[rows]), ro))
    torch.cuda.synchronize()
    assert worst_o <= TOL_BF16
    assert rel(np64(st_gpu[rows]), st_ref) <= TOL_BF16


@pytest.mark.parametrize("dtype,dk", [("f32", 128), ("bf16", 128), ("bf16", 256)])
def test_decode_steps_iplr(dtype, dk):
    """Comba-iplr decode (feedback strength 2 alpha b beta) against the oracle's iplr step."""
    Bd, H, dv, steps = 6, 2, 128, 5
    state = inputs.decode_state(Bd, H, dk, dv, seed_offset=7)
    b = np.random.default_rng(2).uniform(0, 1, H).astype(np.float32)
    st_gpu = _f32(state)
    st_ref = state.astype(np.float64)
    for s in range(steps):
        q, k, v, a, be, d = inputs.decode_tokens(s, Bd, H, dk, dv, dtype)
        o = comba_recurrent_step(_tok(q, dtype), _tok(k, dtype), _tok(v, dtype), _f32(a), _f32(be), _f32(d), st_gpu,
                                 b=_f32(b), iplr=True)
        ro, st_ref = oracle.step(q, k, v, a, be, b, d, st_ref, variant="iplr")
        torch.cuda.synchronize()
        tl = TOL_BF16 if dtype == "bf16" else TOL_F32
        assert rel(np64(o), ro) <= tl
        assert rel(np64(st_gpu), st_ref) <= tl
