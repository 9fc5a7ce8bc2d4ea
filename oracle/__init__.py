"""Comba fp64 CPU oracle (test infrastructure only).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The CUDA library never calls it, and it
never calls the CUDA library.

``comba_oracle.c`` is the token-by-token recurrence of the paper (section 3,
Eq. "comba-S"; feedback strength of section 3.1; recurrent listing of
appendix B.1) in double precision, with exact back-propagation through time
for the gradients.  ``chunked.py`` is a separate fp64 NumPy statement of the
paper's chunk-wise algorithm (section 3.2: WY representation, UT transform,
inter-chunk state and output equations); it is used only to pin the paper's
chunk algebra against the recurrence.

Arrays are NumPy float64 in the packed layout ``[Ttot, H, D]`` with
``cu_seqlens`` (int64 ``[N+1]``); a dense ``[B, T, H, D]`` batch may be passed
as is (it is reshaped, with ``cu = {0, T, 2T, ...}``).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "comba_oracle.c")
_BUILD = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD, "libcomba_oracle.so")
_lib = None
_lock = threading.Lock()


def build(force: bool = False) -> str:
    """Compile ``comba_oracle.c`` with gcc into ``oracle/_build``; returns the path."""
    os.makedirs(_BUILD, exist_ok=True)
    stale = (not os.path.exists(_LIB_PATH)) or os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)
    if force or stale:
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", "-o", tmp, _SRC]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _bind(lib):
    P = ctypes.c_void_p
    I = ctypes.c_int
    lib.comba_oracle_fwd.argtypes = [I, P, I, I, I] + [P] * 11 + [I, I]
    lib.comba_oracle_fwd.restype = I
    lib.comba_oracle_bwd.argtypes = [I, P, I, I, I] + [P] * 9 + [P, P] + [P] * 9 + [I, I]
    lib.comba_oracle_bwd.restype = I
    lib.comba_oracle_step.argtypes = [I, I, I, I] + [P] * 10 + [I, I]
    lib.comba_oracle_step.restype = I
    return lib


def _load():
    global _lib
    with _lock:
        if _lib is None:
            _lib = _bind(ctypes.CDLL(build()))
        return _lib


def build_variant(source_text: str, out_dir: str) -> str:
    """Compile an edited copy of the oracle source (used by tests that plant mistakes)."""
    os.makedirs(out_dir, exist_ok=True)
    src = os.path.join(out_dir, "variant.c")
    lib = os.path.join(out_dir, "libvariant.so")
    with open(src, "w") as f:
        f.write(source_text)
    subprocess.run(["gcc", "-O2", "-std=c11", "-shared", "-fPIC", "-pthread", "-o", lib, src], check=True)
    return lib


def source_text() -> str:
    with open(_SRC) as f:
        return f.read()


def default_threads() -> int:
    return os.cpu_count() or 1


def _f64(x):
    return None if x is None else np.ascontiguousarray(x, dtype=np.float64)


def _ptr(x):
    return None if x is None else x.ctypes.data_as(ctypes.c_void_p)


def _packed(q, k, v, alpha, beta, cu_seqlens, p=None):
    """Return packed [Ttot,H,D] views plus int64 cu, and the original batch shape."""
    if q.ndim == 4:
        if cu_seqlens is not None:
            raise ValueError("cu_seqlens is only valid with packed [Ttot,H,D] inputs")
        B, T, H, _ = q.shape
        cu = np.arange(B + 1, dtype=np.int64) * T
        shape = (B, T)
        q, k, v = (x.reshape(B * T, H, x.shape[-1]) for x in (q, k, v))
        p = None if p is None else p.reshape(B * T, H, p.shape[-1])
        alpha, beta = alpha.reshape(B * T, H), beta.reshape(B * T, H)
    else:
        if cu_seqlens is None:
            cu = np.array([0, q.shape[0]], dtype=np.int64)
        else:
            cu = np.ascontiguousarray(cu_seqlens, dtype=np.int64)
        shape = None
    return q, k, v, alpha, beta, cu, shape, p


VARIANTS = {"splr": 0, "iplr": 1}


def fwd(q, k, v, alpha, beta, b, d, h0=None, cu_seqlens=None, threads=None, lib=None, variant="splr", p=None):
    """Token recurrence forward.  Returns ``(o, hT)`` in float64.

    ``variant="iplr"``: the Comba-iplr transition alpha (I - 2 btilde k k^T).
    ``p`` (shaped like k): the Comba-pk feedback vectors of appendix B.3, read
    back from the state and used in the output correction in place of k."""
    q, k, v, alpha, beta, b, d, h0, p = map(_f64, (q, k, v, alpha, beta, b, d, h0, p))
    q, k, v, alpha, beta, cu, shape, p = _packed(q, k, v, alpha, beta, cu_seqlens, p)
    Ttot, H, dk = q.shape
    dv = v.shape[-1]
    N = cu.shape[0] - 1
    q, k, v, alpha, beta = map(np.ascontiguousarray, (q, k, v, alpha, beta))
    p = None if p is None else np.ascontiguousarray(p)
    o = np.zeros((Ttot, H, dv), np.float64)
    hT = np.zeros((N, H, dk, dv), np.float64)
    rc = (lib or _load()).comba_oracle_fwd(N, _ptr(cu), H, dk, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(p), _ptr(alpha),
                                  _ptr(beta), _ptr(b), _ptr(d), _ptr(h0), _ptr(o), _ptr(hT),
                                  threads or default_threads(), VARIANTS[variant])
    if rc:
        raise MemoryError("oracle forward failed to allocate")
    if shape is not None:
        o = o.reshape(shape[0], shape[1], H, dv)
    return o, hT


def bwd(q, k, v, alpha, beta, b, d, dO, h0=None, dhT=None, cu_seqlens=None, threads=None, lib=None,
        variant="splr", p=None):
    """Exact BPTT.  Returns a dict with dq, dk, dv, dalpha, dbeta, db, dd, dh0 (and dp when
    the Comba-pk feedback vectors ``p`` are given)."""
    q, k, v, alpha, beta, b, d, h0, dO, dhT, p = map(_f64, (q, k, v, alpha, beta, b, d, h0, dO, dhT, p))
    batched = q.ndim == 4
    q, k, v, alpha, beta, cu, shape, p = _packed(q, k, v, alpha, beta, cu_seqlens, p)
    if batched:
        dO = dO.reshape(-1, dO.shape[-2], dO.shape[-1])
    Ttot, H, dk = q.shape
    dv = v.shape[-1]
    N = cu.shape[0] - 1
    q, k, v, alpha, beta, dO = map(np.ascontiguousarray, (q, k, v, alpha, beta, dO))
    p = None if p is None else np.ascontiguousarray(p)
    out = {
        "dq": np.zeros((Ttot, H, dk)), "dk": np.zeros((Ttot, H, dk)), "dv": np.zeros((Ttot, H, dv)),
        "dalpha": np.zeros((Ttot, H)), "dbeta": np.zeros((Ttot, H)),
        "db": np.zeros(H), "dd": np.zeros(H), "dh0": np.zeros((N, H, dk, dv)),
    }
    if p is not None:
        out["dp"] = np.zeros((Ttot, H, dk))
    rc = (lib or _load()).comba_oracle_bwd(
        N, _ptr(cu), H, dk, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(p), _ptr(alpha), _ptr(beta), _ptr(b), _ptr(d),
        _ptr(h0), _ptr(dO), _ptr(dhT), _ptr(out["dq"]), _ptr(out["dk"]), _ptr(out["dv"]), _ptr(out.get("dp")),
        _ptr(out["dalpha"]), _ptr(out["dbeta"]), _ptr(out["db"]), _ptr(out["dd"]), _ptr(out["dh0"]),
        threads or default_threads(), VARIANTS[variant])
    if rc:
        raise MemoryError("oracle backward failed to allocate")
    if shape is not None:
        B, T = shape
        for key in ("dq", "dk", "dv", "dp"):
            if key in out:
                out[key] = out[key].reshape(B, T, H, -1)
        for key in ("dalpha", "dbeta"):
            out[key] = out[key].reshape(B, T, H)
    return out


def step(q, k, v, alpha, beta, b, d, state, threads=None, lib=None, variant="splr", p=None):
    """One decode token.  ``state`` [Bd,H,dk,dv] is copied, updated and returned with ``o``.
    ``p`` [Bd,H,dk]: Comba-pk feedback vectors (default: k)."""
    q, k, v, alpha, beta, b, d, p = map(_f64, (q, k, v, alpha, beta, b, d, p))
    st = np.array(state, dtype=np.float64, copy=True, order="C")
    Bd, H, dk = q.shape
    dv = v.shape[-1]
    o = np.zeros((Bd, H, dv), np.float64)
    rc = (lib or _load()).comba_oracle_step(Bd, H, dk, dv, _ptr(q), _ptr(k), _ptr(v), _ptr(p), _ptr(alpha),
                                   _ptr(beta), _ptr(b), _ptr(d), _ptr(st), _ptr(o), threads or default_threads(),
                                   VARIANTS[variant])
    if rc:
        raise MemoryError("oracle step failed to allocate")
    return o, st


def load_variant(path):
    """ctypes handle of a compiled oracle variant, for the ``lib=`` argument of fwd/bwd/step."""
    return _bind(ctypes.CDLL(path))
