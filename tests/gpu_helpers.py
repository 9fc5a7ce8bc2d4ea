"""Helpers shared by the GPU parity tests: move a seeded workload to the GPU,
run the library through its binding, and compare with the fp64 oracle.

Error metric (per output tensor, every tensor alike): max-norm relative error
    rel = max_i |x_i - r_i| / max_i |r_i|.
Tolerances: 1e-4 for the fp32 storage path, 2e-2 for bf16 storage with fp32
state and accumulation.

The per-head parameter gradients db and dd are tensors [H] like any other and
take the same metric over their heads.  Each head's value is a sum over every
token of the batch of per-token contributions c_t (dd: -k_t . dq~_t, from the
output correction q~ = q - d k; db: beta_t dbtilde_t, from btilde = b beta),
and a head whose sum happens to cancel to near zero has a large error of its
own (its elementwise relative error), the same as a near-zero element of any
other tensor.  `param_grad_report` gives those per-head figures and the error
on the scale sum_t |c_t| of the contributions, for reporting next to the
metric: c_t(dd) = -k_t . dq_t, c_t(db) = (beta_t dbeta_t - v_t . dv_t) / b,
both from the oracle's outputs alone (dbeta = v . de + b dbtilde, dv = beta de).
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


def _heads_last(x):
    """[..., H] -> [tokens, H]."""
    return x.reshape(-1, x.shape[-1])


def param_grad_scales(k, v, beta, b, ref):
    """Per-head sums of |per-token contribution| to dd and db (see the module docstring)."""
    k, v, beta = (np.asarray(x, np.float64) for x in (k, v, beta))
    H = k.shape[-2]
    cdd = -np.einsum("...hd,...hd->...h", k, ref["dq"])
    bh = np.ones(H) if b is None else np.asarray(b, np.float64)
    cdb = (beta * ref["dbeta"] - np.einsum("...hd,...hd->...h", v, ref["dv"])) / bh
    return {"dd": np.abs(_heads_last(cdd)).sum(0), "db": np.abs(_heads_last(cdb)).sum(0)}


def rel_sum(x, ref, scale):
    """max_h |x_h - r_h| / scale_h for per-head sums over tokens."""
    x, ref, scale = (np.asarray(a, np.float64).reshape(-1) for a in (x, ref, scale))
    return float(np.max(np.abs(x - ref) / np.maximum(scale, 1e-300)))


def param_grad_errors(g, ref):
    """dd and db: the max-norm relative error over their heads, as for every tensor."""
    return {key: rel(g[key], ref[key]) for key in ("dd", "db")}


def param_grad_report(g, ref, k, v, beta, b):
    """Context for dd and db (not a bound): the worst per-head relative error, and the error
    on the summation scale sum_t |c_t|."""
    sc = param_grad_scales(k, v, beta, b, ref)
    out = {}
    for key in ("dd", "db"):
        x, r = (np.asarray(a, np.float64).reshape(-1) for a in (g[key], ref[key]))
        out[key + "_per_head_max"] = float(np.max(np.abs(x - r) / np.maximum(np.abs(r), 1e-300)))
        out[key + "_sum_scale"] = rel_sum(x, r, sc[key])
    return out


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
