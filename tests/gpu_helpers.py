"""Helpers shared by the GPU parity tests: move a seeded workload to the GPU,
run the library through its binding, and compare with the fp64 oracle.

Error metric (per output tensor): max-norm relative error
    rel = max_i |x_i - r_i| / max_i |r_i|.
Tolerances: 1e-4 for the fp32 storage path, 2e-2 for bf16 storage with fp32
state and accumulation.
"""
import numpy as np
import torch

TOL_F32 = 1e-4
TOL_BF16 = 2e-2


def rel(x, ref):
    x = np.asarray(x, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.abs(ref).max()
    return float(np.abs(x - ref).max() / den) if den > 0 else float(np.abs(x).max())


def tol(dtype):
    return TOL_BF16 if dtype == "bf16" else TOL_F32


def to_dev(w, device="cuda"):
    """Torch tensors for a Workload (token tensors in the workload's storage type)."""
    tdt = torch.bfloat16 if w.dtype == "bf16" else torch.float32

    def tok(x):
        return None if x is None else torch.from_numpy(np.ascontiguousarray(x)).to(device=device, dtype=tdt)

    def f32(x):
        return None if x is None else torch.from_numpy(np.ascontiguousarray(x, np.float32)).to(device)

    t = dict(q=tok(w.q), k=tok(w.k), v=tok(w.v), alpha=f32(w.alpha), beta=f32(w.beta), d=f32(w.d), b=f32(w.b),
             h0=f32(w.h0), dO=tok(w.dO), dhT=f32(w.dhT))
    t["cu_seqlens"] = None if w.cu_seqlens is None else torch.from_numpy(w.cu_seqlens.astype(np.int32)).to(device)
    return t


def np64(t):
    return t.detach().float().cpu().numpy().astype(np.float64)
