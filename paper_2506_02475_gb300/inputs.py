"""Seeded synthetic inputs for the Comba chunk and decode paths.

This module holds no arithmetic of the method itself: it draws random
tensors with the shapes and value ranges of the paper's layer workloads and
rounds them to the storage precision.  Both the CUDA tests/benchmark and the
fp64 oracle consume exactly these values.

Value recipe (the paper's gate parameterisation, section 3.1 table of gates:
alpha = exp(-a*softplus(.)) close to 1, beta = sigmoid(.) in (0, 1);
keys/queries L2-normalised as in section 3, "SPLR" paragraph):
  * q, k ~ N(0,1), then L2-normalised per (token, head); v ~ N(0,1);
  * alpha = exp(-0.1*softplus(x)), beta = sigmoid(x), x ~ N(0,1) (fp32);
  * d per head ~ U(0,1) (the tiny fp32 workload uses d = 0.5);
  * optional b per head ~ U(0,1) (None means b = 1, i.e. btilde = beta);
  * optional initial state h0 ~ 0.1*N(0,1) fp32; gradients dO ~ N(0,1),
    dhT ~ 0.1*N(0,1);
  * bf16 workloads round q, k, v, dO to bf16 (round to nearest even) on the
    host; arrays are returned as float32 holding bf16-representable values;
  * Comba-pk feedback vectors (``feedback_vectors``): p = s * normalise(k + 0.5 n),
    n ~ N(0,1), s ~ U(0.5, 1) per (token, head): a perturbed, rescaled copy of
    the key (the appendix's p = b k plus a learned deviation), so that p . k > 0
    mostly and the transitions alpha I - btilde p k^T stay contracting over
    long sequences.

Seeds: numpy PCG64 with seed 42 (the paper's training seed) plus a fixed
per-workload offset.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import Optional

import numpy as np

SEED = 42


def round_bf16(x: np.ndarray) -> np.ndarray:
    """Round float32 values to the nearest bf16 (ties to even); returns float32."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).reshape(f.shape)


def _l2norm(x: np.ndarray) -> np.ndarray:
    return x / np.sqrt(np.sum(x * x, axis=-1, keepdims=True))


def _softplus(x):
    return np.logaddexp(0.0, x)


def _sigmoid(x):
    return 1.0 / (1.0 + np.exp(-x))


@dataclass
class Workload:
    """One synthetic problem.  Token arrays are [B,T,H,D] (dense) or [Ttot,H,D] (packed)."""
    name: str
    dtype: str                      # "f32" or "bf16": storage type of q, k, v, o, dO
    q: np.ndarray
    k: np.ndarray
    v: np.ndarray
    alpha: np.ndarray
    beta: np.ndarray
    d: np.ndarray
    b: Optional[np.ndarray] = None
    h0: Optional[np.ndarray] = None
    dO: Optional[np.ndarray] = None
    dhT: Optional[np.ndarray] = None
    cu_seqlens: Optional[np.ndarray] = None
    extra: dict = field(default_factory=dict)

    @property
    def packed(self) -> bool:
        return self.cu_seqlens is not None

    @property
    def H(self) -> int:
        return self.q.shape[-2]

    @property
    def dk(self) -> int:
        return self.q.shape[-1]

    @property
    def dv(self) -> int:
        return self.v.shape[-1]

    @property
    def tokens(self) -> int:
        return int(np.prod(self.q.shape[:-2]))

    @property
    def num_seqs(self) -> int:
        return len(self.cu_seqlens) - 1 if self.packed else self.q.shape[0]


def _gates(rng, shape):
    x = rng.standard_normal(shape)
    alpha = np.exp(-_softplus(x) * 0.1).astype(np.float32)
    x = rng.standard_normal(shape)
    beta = _sigmoid(x).astype(np.float32)
    return alpha, beta


def _tokens(rng, lead, H, dk, dv, dtype):
    q = _l2norm(rng.standard_normal(lead + (H, dk), dtype=np.float32))
    k = _l2norm(rng.standard_normal(lead + (H, dk), dtype=np.float32))
    v = rng.standard_normal(lead + (H, dv), dtype=np.float32)
    if dtype == "bf16":
        q, k, v = round_bf16(q), round_bf16(k), round_bf16(v)
    return q.astype(np.float32), k.astype(np.float32), v.astype(np.float32)


def varlen_lengths(rng, n=12, total=65536, lo=512, hi=16384) -> np.ndarray:
    """n lengths drawn log-uniformly in [lo, hi], rescaled to sum exactly to ``total``."""
    u = rng.uniform(np.log(lo), np.log(hi), size=n)
    x = np.exp(u)
    for _ in range(100):
        x = np.clip(x * (total / x.sum()), lo, hi)
        if abs(x.sum() - total) < 0.5:
            break
    lens = np.round(x).astype(np.int64)
    resid = total - int(lens.sum())
    order = np.argsort(-lens)
    for i in order:  # residual onto the longest sequences that stay within bounds
        if resid == 0:
            break
        step = min(resid, hi - lens[i]) if resid > 0 else max(resid, lo - lens[i])
        lens[i] += step
        resid -= step
    assert lens.sum() == total and lens.min() >= lo and lens.max() <= hi
    return lens


def make(name: str, *, B=None, T=None, H=None, dk=None, dv=None, dtype=None, seed_offset=0,
         with_b=False, with_h0=None, with_grads=None, lengths=None) -> Workload:
    """Build a named workload; keyword arguments shrink or vary it for tests.

    Names: ``tiny_fp32``, ``lm340m``, ``lm1p3b``, ``lm1p3b_v256`` (value heads twice as wide as the
    keys: dk = 128, dv = 256), ``lm1p3b_d256`` (head dim 256: dk = dv = 256, half the heads),
    ``varlen64k``, ``custom``.
    """
    presets = {
        # name: (B, T, H, dk, dv, dtype, h0, grads, offset)
        "tiny_fp32": (1, 256, 2, 64, 64, "f32", False, False, 1),
        "lm340m": (8, 2048, 8, 128, 128, "bf16", False, True, 2),
        "lm1p3b": (4, 4096, 16, 128, 128, "bf16", True, True, 3),
        "lm1p3b_v256": (4, 4096, 8, 128, 256, "bf16", True, True, 5),
        "lm1p3b_d256": (4, 4096, 8, 256, 256, "bf16", True, True, 6),
        "varlen64k": (1, 65536, 16, 128, 128, "bf16", False, True, 4),
        "custom": (1, 256, 2, 64, 64, "f32", False, True, 9),
    }
    pB, pT, pH, pdk, pdv, pdt, ph0, pgr, off = presets[name]
    B, T, H = B or pB, T or pT, H or pH
    dk, dv, dtype = dk or pdk, dv or pdv, dtype or pdt
    with_h0 = ph0 if with_h0 is None else with_h0
    with_grads = pgr if with_grads is None else with_grads
    rng = np.random.Generator(np.random.PCG64(SEED + 1000 * off + seed_offset))

    cu = None
    if name == "varlen64k" or lengths is not None:
        if lengths is None:
            lengths = varlen_lengths(rng, total=T)
        lengths = np.asarray(lengths, dtype=np.int64)
        cu = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
        lead = (int(cu[-1]),)
        N = len(lengths)
    else:
        lead = (B, T)
        N = B
    q, k, v = _tokens(rng, lead, H, dk, dv, dtype)
    alpha, beta = _gates(rng, lead + (H,))
    # per-head parameters come from their own generator: ranks of a data-parallel
    # run (different seed_offset) share d and b and differ only in their data
    prng = np.random.Generator(np.random.PCG64(SEED + 1000 * off + 500))
    if name == "tiny_fp32":
        d = np.full(H, 0.5, np.float32)
    else:
        d = prng.uniform(0.0, 1.0, size=H).astype(np.float32)
    b = prng.uniform(0.0, 1.0, size=H).astype(np.float32) if with_b else None
    h0 = (0.1 * rng.standard_normal((N, H, dk, dv))).astype(np.float32) if with_h0 else None
    dO = dhT = None
    if with_grads:
        dO = rng.standard_normal(lead + (H, dv), dtype=np.float32)
        if dtype == "bf16":
            dO = round_bf16(dO)
        dhT = (0.1 * rng.standard_normal((N, H, dk, dv))).astype(np.float32)
    return Workload(name=name, dtype=dtype, q=q, k=k, v=v, alpha=alpha, beta=beta, d=d, b=b, h0=h0,
                    dO=dO, dhT=dhT, cu_seqlens=cu)


def decode_state(Bd=256, H=16, dk=128, dv=128, seed_offset=0, state_std=0.05) -> np.ndarray:
    """fp32 decode state [Bd,H,dk,dv] ~ N(0, state_std^2)."""
    rng = np.random.Generator(np.random.PCG64(SEED + 6000 + seed_offset))
    return (state_std * rng.standard_normal((Bd, H, dk, dv), dtype=np.float32)).astype(np.float32)


def decode_tokens(step, Bd=256, H=16, dk=128, dv=128, dtype="bf16", seed_offset=0):
    """Token inputs of one decode step (its own seed, so long decode runs never materialise all steps).

    Returns q, k [Bd,H,dk], v [Bd,H,dv], alpha, beta [Bd,H] and d [H] (d is the same for every step)."""
    rng = np.random.Generator(np.random.PCG64([SEED + 7000 + seed_offset, step]))
    q, k, v = _tokens(rng, (Bd,), H, dk, dv, dtype)
    alpha, beta = _gates(rng, (Bd, H))
    drng = np.random.Generator(np.random.PCG64(SEED + 8000))   # a parameter: shared by every rank
    d = drng.uniform(0.0, 1.0, size=H).astype(np.float32)
    return q, k, v, alpha, beta, d


@dataclass
class GatedWorkload:
    """Raw inputs of the gate and normalisation prologue (q, k not normalised; gate pre-activations)."""
    dtype: str
    q: np.ndarray            # [B,T,H,dk] or packed [Ttot,H,dk]
    k: np.ndarray
    v: np.ndarray
    g_alpha: np.ndarray      # [B,T,H] or [Ttot,H]
    g_beta: np.ndarray
    a: np.ndarray            # [H]
    c: np.ndarray
    b_raw: np.ndarray
    d: np.ndarray
    h0: Optional[np.ndarray]
    dO: np.ndarray
    dhT: np.ndarray
    cu_seqlens: Optional[np.ndarray] = None


def make_gated(B=2, T=200, H=3, dk=128, dv=128, dtype="bf16", seed_offset=0, lengths=None, with_h0=True):
    """Seeded raw inputs: q, k ~ N(0, s^2) with a per-row scale s in [0.5, 2] (so the in-kernel L2
    norm has work to do), v ~ N(0,1), gate pre-activations ~ N(0,1), a ~ U(0.05, 0.3) (alpha near 1
    as the forgetting section asks), c, b_raw ~ U(-1, 1), d ~ U(0, 1); bf16 rounding on the host."""
    rng = np.random.Generator(np.random.PCG64(SEED + 9000 + seed_offset))
    cu = None
    if lengths is not None:
        lengths = np.asarray(lengths, dtype=np.int64)
        cu = np.concatenate([[0], np.cumsum(lengths)]).astype(np.int64)
        lead, N = (int(cu[-1]),), len(lengths)
    else:
        lead, N = (B, T), B
    q = rng.standard_normal(lead + (H, dk)) * rng.uniform(0.5, 2.0, lead + (H, 1))
    k = rng.standard_normal(lead + (H, dk)) * rng.uniform(0.5, 2.0, lead + (H, 1))
    v = rng.standard_normal(lead + (H, dv))
    dO = rng.standard_normal(lead + (H, dv))
    q, k, v, dO = (x.astype(np.float32) for x in (q, k, v, dO))
    if dtype == "bf16":
        q, k, v, dO = (round_bf16(x) for x in (q, k, v, dO))
    g_alpha = rng.standard_normal(lead + (H,)).astype(np.float32)
    g_beta = rng.standard_normal(lead + (H,)).astype(np.float32)
    prng = np.random.Generator(np.random.PCG64(SEED + 9500))
    a = prng.uniform(0.05, 0.3, H).astype(np.float32)
    c = prng.uniform(-1.0, 1.0, H).astype(np.float32)
    b_raw = prng.uniform(-1.0, 1.0, H).astype(np.float32)
    d = prng.uniform(0.0, 1.0, H).astype(np.float32)
    h0 = (0.1 * rng.standard_normal((N, H, dk, dv))).astype(np.float32) if with_h0 else None
    dhT = (0.1 * rng.standard_normal((N, H, dk, dv))).astype(np.float32)
    return GatedWorkload(dtype=dtype, q=q, k=k, v=v, g_alpha=g_alpha, g_beta=g_beta, a=a, c=c, b_raw=b_raw, d=d,
                         h0=h0, dO=dO, dhT=dhT, cu_seqlens=cu)


def feedback_vectors(k: np.ndarray, dtype: str = "bf16", seed_offset: int = 0) -> np.ndarray:
    """Comba-pk feedback vectors shaped like ``k``: s * normalise(k + 0.5 n), n ~ N(0,1),
    s ~ U(0.5, 1) per row; bf16-rounded for bf16 workloads."""
    rng = np.random.Generator(np.random.PCG64(SEED + 11000 + seed_offset))
    k = np.asarray(k, np.float32)
    n = rng.standard_normal(k.shape, dtype=np.float32)
    s = rng.uniform(0.5, 1.0, k.shape[:-1] + (1,)).astype(np.float32)
    p = (s * _l2norm(k + 0.5 * n)).astype(np.float32)
    return round_bf16(p) if dtype == "bf16" else p
