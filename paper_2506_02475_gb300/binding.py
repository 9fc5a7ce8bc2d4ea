"""Thin ctypes binding of ``libcomba.so`` (the C ABI in ``include/comba.h``).

Argument marshalling only: tensors are checked, outputs and the workspace are
allocated with torch (device memory plumbing), raw device pointers and the
current CUDA stream are passed to the C entry points, and a non-OK status is
raised as an exception.  Every arithmetic step runs inside the library's
CUDA kernels; there is no fallback path.  If the compiled library is missing
the import of any entry point fails loudly.
"""
from __future__ import annotations

import ctypes
import os
import threading

import torch

from . import build as _build

_lib = None
_lock = threading.Lock()

COMBA_F32, COMBA_BF16 = 0, 1
COMBA_SAVE_FACTORS, COMBA_REUSE_FACTORS, COMBA_IPLR, COMBA_GATED, COMBA_PK = 1, 2, 4, 8, 16
COMBA_ERR_TIMEOUT = 5
_STATUS = {0: "ok", 1: "invalid argument", 2: "unsupported configuration", 3: "workspace missing or too small",
           4: "CUDA error", 5: "device-side wait timed out"}


class CombaError(RuntimeError):
    def __init__(self, fn, status):
        super().__init__(f"{fn} failed: {_STATUS.get(status, status)} (status {status})")
        self.status = status


class _Shape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int), ("T", ctypes.c_int), ("H", ctypes.c_int), ("dk", ctypes.c_int),
                ("dv", ctypes.c_int), ("num_seqs", ctypes.c_int), ("cu_seqlens", ctypes.c_void_p),
                ("dtype", ctypes.c_int), ("chunk", ctypes.c_int), ("flags", ctypes.c_int),
                ("stage_events", ctypes.c_void_p),
                ("num_stage_events", ctypes.c_int), ("wait_limit_ns", ctypes.c_uint)]


def library_path() -> str:
    return _build.LIB


def lib():
    """Load libcomba.so (building it first if this checkout has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        path = _build.LIB
        if not os.path.exists(path) or not _build.up_to_date():
            _build.build()
        L = ctypes.CDLL(path)
        P, I, Z = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        SP = ctypes.POINTER(_Shape)
        L.comba_workspace_size.argtypes = [SP, I]
        L.comba_workspace_size.restype = Z
        L.comba_chunk_fwd.argtypes = [SP] + [P] * 10 + [P, Z, P]
        L.comba_chunk_fwd.restype = I
        L.comba_chunk_bwd.argtypes = [SP] + [P] * 10 + [P] * 8 + [P, Z, P]
        L.comba_chunk_bwd.restype = I
        L.comba_recurrent_step.argtypes = [I, I, I, I, I] + [P] * 9 + [I, P]
        L.comba_recurrent_step.restype = I
        L.comba_chunk_fwd_gated.argtypes = [SP] + [P] * 12 + [P, Z, P]
        L.comba_chunk_fwd_gated.restype = I
        L.comba_chunk_bwd_gated.argtypes = [SP] + [P] * 12 + [P] * 10 + [P, Z, P]
        L.comba_chunk_bwd_gated.restype = I
        L.comba_chunk_fwd_pk.argtypes = [SP] + [P] * 11 + [P, Z, P]
        L.comba_chunk_fwd_pk.restype = I
        L.comba_chunk_bwd_pk.argtypes = [SP] + [P] * 11 + [P] * 9 + [P, Z, P]
        L.comba_chunk_bwd_pk.restype = I
        L.comba_recurrent_step_pk.argtypes = [I, I, I, I, I] + [P] * 10 + [I, P]
        L.comba_recurrent_step_pk.restype = I
        L.comba_workspace_status.argtypes = [P, P]
        L.comba_workspace_status.restype = I
        L.comba_status_string.argtypes = [I]
        L.comba_status_string.restype = ctypes.c_char_p
        _lib = L
        return L


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _dtype_code(t):
    if t.dtype == torch.bfloat16:
        return COMBA_BF16
    if t.dtype == torch.float32:
        return COMBA_F32
    raise TypeError(f"q/k/v must be float32 or bfloat16, got {t.dtype}")


def _check(name, t, dtype=None, shape=None, device=None):
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")


def make_shape(q, v, cu_seqlens=None, stage_events=None, flags=0, wait_limit_ns=0):
    """Build the C shape struct from q [B,T,H,dk] (or packed [Ttot,H,dk]) and v.

    ``stage_events`` (optional): sequence of raw cudaEvent_t handles (ints) recorded at
    kernel boundaries (instrumentation; see include/comba.h).  ``wait_limit_ns``: limit of
    each device-side wait in nanoseconds (0: the library's default of one second)."""
    if q.dim() == 3:
        q = q.unsqueeze(0)
        v = v.unsqueeze(0)
    B, T, H, dk = q.shape
    dv = v.shape[-1]
    s = _Shape()
    s.B, s.T, s.H, s.dk, s.dv = B, T, H, dk, dv
    if cu_seqlens is not None:
        s.num_seqs = cu_seqlens.numel() - 1
        s.cu_seqlens = cu_seqlens.data_ptr()
    else:
        s.num_seqs = B
        s.cu_seqlens = None
    s.dtype = _dtype_code(q)
    s.chunk = 64
    s.flags = flags
    s.wait_limit_ns = wait_limit_ns
    if stage_events is not None:
        arr = (ctypes.c_void_p * len(stage_events))(*stage_events)
        s._events_keepalive = arr
        s.stage_events = ctypes.cast(arr, ctypes.c_void_p)
        s.num_stage_events = len(stage_events)
    return s


def comba_workspace_size(q, v, cu_seqlens=None, backward=False, flags=0) -> int:
    return int(lib().comba_workspace_size(ctypes.byref(make_shape(q, v, cu_seqlens, None, flags)),
                                          int(bool(backward))))


def _workspace(nbytes, device, workspace):
    if workspace is not None:
        if workspace.numel() * workspace.element_size() < nbytes:
            raise ValueError(f"workspace has {workspace.numel() * workspace.element_size()} bytes, need {nbytes}")
        return workspace
    return torch.empty(max(nbytes, 16), dtype=torch.uint8, device=device)


def _check_inputs(q, k, v, alpha, beta, b, d, h0, cu_seqlens):
    dev = q.device
    packed = q.dim() == 3
    lead = tuple(q.shape[:-1])
    H, dk, dv = q.shape[-2], q.shape[-1], v.shape[-1]
    _check("q", q, device=dev)
    _check("k", k, dtype=q.dtype, shape=q.shape, device=dev)
    _check("v", v, dtype=q.dtype, shape=lead + (dv,), device=dev)
    _check("alpha", alpha, torch.float32, lead, dev)
    _check("beta", beta, torch.float32, lead, dev)
    _check("b", b, torch.float32, (H,), dev)
    _check("d", d, torch.float32, (H,), dev)
    if cu_seqlens is not None:
        _check("cu_seqlens", cu_seqlens, torch.int32, None, dev)
        N = cu_seqlens.numel() - 1
        if not packed and q.shape[0] != 1:
            raise ValueError("cu_seqlens requires B == 1 (or packed [Ttot,H,D] inputs)")
    else:
        N = 1 if packed else q.shape[0]
    _check("h0", h0, torch.float32, (N, H, dk, dv), dev)
    return N, H, dk, dv


def comba_chunk_fwd(q, k, v, alpha, beta, d, b=None, h0=None, cu_seqlens=None, output_final_state=False,
                    o=None, hT=None, workspace=None, stream=None, stage_events=None, save_factors=False,
                    iplr=False, wait_limit_ns=0):
    """Chunk-parallel forward.  Returns ``(o, hT)`` (``hT`` is None unless requested).

    ``save_factors=True`` keeps the backward's chunk factors in ``workspace`` (which must
    then be sized for the backward) so that ``comba_chunk_bwd(..., reuse_factors=True)``
    with the same workspace skips recomputing them.  ``iplr=True``: the Comba-iplr
    transition alpha (I - 2 btilde k k^T)."""
    N, H, dk, dv = _check_inputs(q, k, v, alpha, beta, b, d, h0, cu_seqlens)
    shape = make_shape(q, v, cu_seqlens, stage_events,
                       (COMBA_SAVE_FACTORS if save_factors else 0) | (COMBA_IPLR if iplr else 0), wait_limit_ns)
    L = lib()
    nbytes = L.comba_workspace_size(ctypes.byref(shape), 1 if save_factors else 0)
    if nbytes == 0:
        raise CombaError("comba_workspace_size", 1)
    ws = _workspace(nbytes, q.device, workspace)
    if o is None:
        o = torch.empty_like(v)
    if hT is None and output_final_state:
        hT = torch.empty((N, H, dk, dv), dtype=torch.float32, device=q.device)
    st = L.comba_chunk_fwd(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(alpha), _ptr(beta), _ptr(b),
                           _ptr(d), _ptr(h0), _ptr(o), _ptr(hT), _ptr(ws), ws.numel() * ws.element_size(),
                           _stream(stream))
    if st != 0:
        raise CombaError("comba_chunk_fwd", st)
    return o, hT


def comba_chunk_bwd(q, k, v, alpha, beta, d, dO, b=None, h0=None, dhT=None, cu_seqlens=None, want_dh0=True,
                    want_db=True, out=None, workspace=None, stream=None, stage_events=None, reuse_factors=False,
                    iplr=False, wait_limit_ns=0):
    """Chunk-parallel backward.  Returns a dict with dq, dk, dv, dalpha, dbeta, dd, db, dh0.

    ``reuse_factors=True`` requires ``workspace`` to hold the factors of a
    ``comba_chunk_fwd(..., save_factors=True)`` call on the same inputs."""
    N, H, dk, dv = _check_inputs(q, k, v, alpha, beta, b, d, h0, cu_seqlens)
    _check("dO", dO, q.dtype, v.shape, q.device)
    _check("dhT", dhT, torch.float32, (N, H, dk, dv), q.device)
    if reuse_factors and workspace is None:
        raise ValueError("reuse_factors=True needs the workspace of the saving forward call")
    shape = make_shape(q, v, cu_seqlens, stage_events,
                       (COMBA_REUSE_FACTORS if reuse_factors else 0) | (COMBA_IPLR if iplr else 0), wait_limit_ns)
    L = lib()
    nbytes = L.comba_workspace_size(ctypes.byref(shape), 1)
    if nbytes == 0:
        raise CombaError("comba_workspace_size", 1)
    ws = _workspace(nbytes, q.device, workspace)
    g = out if out is not None else {}
    g.setdefault("dq", torch.empty_like(q))
    g.setdefault("dk", torch.empty_like(k))
    g.setdefault("dv", torch.empty_like(v))
    g.setdefault("dalpha", torch.empty_like(alpha))
    g.setdefault("dbeta", torch.empty_like(beta))
    g.setdefault("dd", torch.empty_like(d))
    if want_db:
        g.setdefault("db", torch.empty((H,), dtype=torch.float32, device=q.device))
    if want_dh0:
        g.setdefault("dh0", torch.empty((N, H, dk, dv), dtype=torch.float32, device=q.device))
    st = L.comba_chunk_bwd(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(alpha), _ptr(beta), _ptr(b),
                           _ptr(d), _ptr(h0), _ptr(dO), _ptr(dhT), _ptr(g["dq"]), _ptr(g["dk"]), _ptr(g["dv"]),
                           _ptr(g["dalpha"]), _ptr(g["dbeta"]), _ptr(g.get("db")), _ptr(g["dd"]),
                           _ptr(g.get("dh0")), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream))
    if st != 0:
        raise CombaError("comba_chunk_bwd", st)
    return g


def comba_workspace_status(workspace=None, stream=None) -> int:
    """Status word of the calls that last used ``workspace`` (None: the static scratch of the
    allocation-free forward): 0 (COMBA_OK), or 5 (COMBA_ERR_TIMEOUT) when a device-side wait of
    one of their kernels gave up.  Waits for ``stream`` first."""
    st = lib().comba_workspace_status(_ptr(workspace), _stream(stream))
    if st not in (0, COMBA_ERR_TIMEOUT):
        raise CombaError("comba_workspace_status", st)
    return st


def comba_recurrent_step(q, k, v, alpha, beta, d, state, b=None, o=None, stream=None, iplr=False):
    """One decode token; ``state`` [Bd,H,dk,dv] fp32 is updated in place.  Returns ``o``."""
    Bd, H, dk = q.shape
    dv = v.shape[-1]
    dev = q.device
    _check("q", q, device=dev)
    _check("k", k, q.dtype, q.shape, dev)
    _check("v", v, q.dtype, (Bd, H, dv), dev)
    _check("alpha", alpha, torch.float32, (Bd, H), dev)
    _check("beta", beta, torch.float32, (Bd, H), dev)
    _check("b", b, torch.float32, (H,), dev)
    _check("d", d, torch.float32, (H,), dev)
    _check("state", state, torch.float32, (Bd, H, dk, dv), dev)
    if o is None:
        o = torch.empty_like(v)
    st = lib().comba_recurrent_step(Bd, H, dk, dv, _dtype_code(q), _ptr(q), _ptr(k), _ptr(v), _ptr(alpha),
                                    _ptr(beta), _ptr(b), _ptr(d), _ptr(state), _ptr(o), COMBA_IPLR if iplr else 0,
                                    _stream(stream))
    if st != 0:
        raise CombaError("comba_recurrent_step", st)
    return o


def _check_gated(q, k, v, g_alpha, g_beta, a, c, b_raw, d, h0, cu_seqlens):
    N, H, dk, dv = _check_inputs(q, k, v, g_alpha, g_beta, None, d, h0, cu_seqlens)
    for name, t in (("a", a), ("c", c), ("b_raw", b_raw)):
        if t is None:
            raise ValueError(f"{name} is required")
        _check(name, t, torch.float32, (H,), q.device)
    return N, H, dk, dv


def comba_chunk_fwd_gated(q, k, v, g_alpha, g_beta, a, c, b_raw, d, h0=None, cu_seqlens=None,
                          output_final_state=False, o=None, hT=None, workspace=None, stream=None, stage_events=None,
                          save_factors=False, iplr=False):
    """Forward with the gate and normalisation prologue: raw q, k; alpha = exp(-a softplus(g_alpha + c)),
    beta = sigmoid(g_beta), b = sigmoid(b_raw); q, k L2-normalised in the kernels.  Returns ``(o, hT)``."""
    N, H, dk, dv = _check_gated(q, k, v, g_alpha, g_beta, a, c, b_raw, d, h0, cu_seqlens)
    flags = COMBA_GATED | (COMBA_SAVE_FACTORS if save_factors else 0) | (COMBA_IPLR if iplr else 0)
    shape = make_shape(q, v, cu_seqlens, stage_events, flags)
    L = lib()
    nbytes = L.comba_workspace_size(ctypes.byref(shape), 1 if save_factors else 0)
    if nbytes == 0:
        raise CombaError("comba_workspace_size", 1)
    ws = _workspace(nbytes, q.device, workspace)
    if o is None:
        o = torch.empty_like(v)
    if hT is None and output_final_state:
        hT = torch.empty((N, H, dk, dv), dtype=torch.float32, device=q.device)
    st = L.comba_chunk_fwd_gated(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(g_alpha), _ptr(g_beta),
                                 _ptr(a), _ptr(c), _ptr(b_raw), _ptr(d), _ptr(h0), _ptr(o), _ptr(hT), _ptr(ws),
                                 ws.numel() * ws.element_size(), _stream(stream))
    if st != 0:
        raise CombaError("comba_chunk_fwd_gated", st)
    return o, hT


def comba_chunk_bwd_gated(q, k, v, g_alpha, g_beta, a, c, b_raw, d, dO, h0=None, dhT=None, cu_seqlens=None,
                          want_dh0=True, out=None, workspace=None, stream=None, stage_events=None,
                          reuse_factors=False, iplr=False):
    """Gradients w.r.t. the raw inputs: dq, dk, dv, dg_alpha, dg_beta, da, dc, db_raw, dd, dh0."""
    N, H, dk, dv = _check_gated(q, k, v, g_alpha, g_beta, a, c, b_raw, d, h0, cu_seqlens)
    _check("dO", dO, q.dtype, v.shape, q.device)
    _check("dhT", dhT, torch.float32, (N, H, dk, dv), q.device)
    if reuse_factors and workspace is None:
        raise ValueError("reuse_factors=True needs the workspace of the saving forward call")
    flags = COMBA_GATED | (COMBA_REUSE_FACTORS if reuse_factors else 0) | (COMBA_IPLR if iplr else 0)
    shape = make_shape(q, v, cu_seqlens, stage_events, flags)
    L = lib()
    nbytes = L.comba_workspace_size(ctypes.byref(shape), 1)
    if nbytes == 0:
        raise CombaError("comba_workspace_size", 1)
    ws = _workspace(nbytes, q.device, workspace)
    g = out if out is not None else {}
    g.setdefault("dq", torch.empty_like(q))
    g.setdefault("dk", torch.empty_like(k))
    g.setdefault("dv", torch.empty_like(v))
    g.setdefault("dg_alpha", torch.empty_like(g_alpha))
    g.setdefault("dg_beta", torch.empty_like(g_beta))
    for key in ("da", "dc", "db_raw", "dd"):
        g.setdefault(key, torch.empty((H,), dtype=torch.float32, device=q.device))
    if want_dh0:
        g.setdefault("dh0", torch.empty((N, H, dk, dv), dtype=torch.float32, device=q.device))
    st = L.comba_chunk_bwd_gated(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(g_alpha), _ptr(g_beta),
                                 _ptr(a), _ptr(c), _ptr(b_raw), _ptr(d), _ptr(h0), _ptr(dO), _ptr(dhT),
                                 _ptr(g["dq"]), _ptr(g["dk"]), _ptr(g["dv"]), _ptr(g["dg_alpha"]),
                                 _ptr(g["dg_beta"]), _ptr(g["da"]), _ptr(g["dc"]), _ptr(g["db_raw"]), _ptr(g["dd"]),
                                 _ptr(g.get("dh0")), _ptr(ws), ws.numel() * ws.element_size(), _stream(stream))
    if st != 0:
        raise CombaError("comba_chunk_bwd_gated", st)
    return g


def comba_chunk_fwd_pk(q, k, v, p, alpha, beta, d, b=None, h0=None, cu_seqlens=None, output_final_state=False,
                       o=None, hT=None, workspace=None, stream=None, stage_events=None, save_factors=False,
                       iplr=False):
    """Comba-pk forward: feedback vectors ``p`` (shaped like k) read back from the state and used in
    the correction q - d p, while k writes the state.  Returns ``(o, hT)``."""
    N, H, dk, dv = _check_inputs(q, k, v, alpha, beta, b, d, h0, cu_seqlens)
    _check("p", p, q.dtype, q.shape, q.device)
    flags = COMBA_PK | (COMBA_SAVE_FACTORS if save_factors else 0) | (COMBA_IPLR if iplr else 0)
    shape = make_shape(q, v, cu_seqlens, stage_events, flags)
    L = lib()
    nbytes = L.comba_workspace_size(ctypes.byref(shape), 1 if save_factors else 0)
    if nbytes == 0:
        raise CombaError("comba_workspace_size", 1)
    ws = _workspace(nbytes, q.device, workspace)
    if o is None:
        o = torch.empty_like(v)
    if hT is None and output_final_state:
        hT = torch.empty((N, H, dk, dv), dtype=torch.float32, device=q.device)
    st = L.comba_chunk_fwd_pk(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(p), _ptr(alpha), _ptr(beta),
                              _ptr(b), _ptr(d), _ptr(h0), _ptr(o), _ptr(hT), _ptr(ws), ws.numel() * ws.element_size(),
                              _stream(stream))
    if st != 0:
        raise CombaError("comba_chunk_fwd_pk", st)
    return o, hT


def comba_chunk_bwd_pk(q, k, v, p, alpha, beta, d, dO, b=None, h0=None, dhT=None, cu_seqlens=None, want_dh0=True,
                       want_db=True, out=None, workspace=None, stream=None, stage_events=None, reuse_factors=False,
                       iplr=False):
    """Comba-pk backward.  Returns a dict with dq, dk, dv, dp, dalpha, dbeta, dd, db, dh0."""
    N, H, dk, dv = _check_inputs(q, k, v, alpha, beta, b, d, h0, cu_seqlens)
    _check("p", p, q.dtype, q.shape, q.device)
    _check("dO", dO, q.dtype, v.shape, q.device)
    _check("dhT", dhT, torch.float32, (N, H, dk, dv), q.device)
    if reuse_factors and workspace is None:
        raise ValueError("reuse_factors=True needs the workspace of the saving forward call")
    flags = COMBA_PK | (COMBA_REUSE_FACTORS if reuse_factors else 0) | (COMBA_IPLR if iplr else 0)
    shape = make_shape(q, v, cu_seqlens, stage_events, flags)
    L = lib()
    nbytes = L.comba_workspace_size(ctypes.byref(shape), 1)
    if nbytes == 0:
        raise CombaError("comba_workspace_size", 1)
    ws = _workspace(nbytes, q.device, workspace)
    g = out if out is not None else {}
    g.setdefault("dq", torch.empty_like(q))
    g.setdefault("dk", torch.empty_like(k))
    g.setdefault("dv", torch.empty_like(v))
    g.setdefault("dp", torch.empty_like(p))
    g.setdefault("dalpha", torch.empty_like(alpha))
    g.setdefault("dbeta", torch.empty_like(beta))
    g.setdefault("dd", torch.empty_like(d))
    if want_db:
        g.setdefault("db", torch.empty((H,), dtype=torch.float32, device=q.device))
    if want_dh0:
        g.setdefault("dh0", torch.empty((N, H, dk, dv), dtype=torch.float32, device=q.device))
    st = L.comba_chunk_bwd_pk(ctypes.byref(shape), _ptr(q), _ptr(k), _ptr(v), _ptr(p), _ptr(alpha), _ptr(beta),
                              _ptr(b), _ptr(d), _ptr(h0), _ptr(dO), _ptr(dhT), _ptr(g["dq"]), _ptr(g["dk"]),
                              _ptr(g["dv"]), _ptr(g["dp"]), _ptr(g["dalpha"]), _ptr(g["dbeta"]), _ptr(g.get("db")),
                              _ptr(g["dd"]), _ptr(g.get("dh0")), _ptr(ws), ws.numel() * ws.element_size(),
                              _stream(stream))
    if st != 0:
        raise CombaError("comba_chunk_bwd_pk", st)
    return g


def comba_recurrent_step_pk(q, k, v, p, alpha, beta, d, state, b=None, o=None, stream=None, iplr=False):
    """One Comba-pk decode token (feedback vector ``p`` [Bd,H,dk]); ``state`` is updated in place."""
    Bd, H, dk = q.shape
    dv = v.shape[-1]
    dev = q.device
    _check("q", q, device=dev)
    _check("k", k, q.dtype, q.shape, dev)
    _check("p", p, q.dtype, q.shape, dev)
    _check("v", v, q.dtype, (Bd, H, dv), dev)
    _check("alpha", alpha, torch.float32, (Bd, H), dev)
    _check("beta", beta, torch.float32, (Bd, H), dev)
    _check("b", b, torch.float32, (H,), dev)
    _check("d", d, torch.float32, (H,), dev)
    _check("state", state, torch.float32, (Bd, H, dk, dv), dev)
    if o is None:
        o = torch.empty_like(v)
    st = lib().comba_recurrent_step_pk(Bd, H, dk, dv, _dtype_code(q), _ptr(q), _ptr(k), _ptr(v), _ptr(p),
                                       _ptr(alpha), _ptr(beta), _ptr(b), _ptr(d), _ptr(state), _ptr(o),
                                       COMBA_IPLR if iplr else 0, _stream(stream))
    if st != 0:
        raise CombaError("comba_recurrent_step_pk", st)
    return o
