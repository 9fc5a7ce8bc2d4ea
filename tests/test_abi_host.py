"""Host-side checks of the C ABI that need no GPU.

The library loads and exports every entry point declared in include/comba.h;
workspace sizing and argument validation answer on the host.  Every call here
returns an error before anything would be launched (validation runs before
the first CUDA call), so fake but well-aligned addresses are safe to pass.
"""
import ctypes
import os
import re

import pytest

from paper_2506_02475_gb300 import binding
from paper_2506_02475_gb300 import build as cbuild

HEADER = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include", "comba.h")
OK, INVALID, UNSUPPORTED, WORKSPACE = 0, 1, 2, 3
FAKE = 0x100000  # aligned, never dereferenced


@pytest.fixture(scope="module")
def L():
    return binding.lib()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(comba_[a-z_0-9]+)\s*\(", text)))


def test_library_exports_every_declared_symbol(L):
    names = declared_functions()
    assert set(names) >= {"comba_chunk_fwd", "comba_chunk_bwd", "comba_recurrent_step", "comba_workspace_size",
                          "comba_status_string"}
    for name in names:
        assert hasattr(L, name), name


def test_library_is_built_for_sm103a():
    assert any("compute_103a" in a for a in cbuild.ARCH)
    assert os.path.exists(binding.library_path())


def test_status_strings(L):
    for code, text in [(0, b"ok"), (1, b"invalid argument"), (3, b"workspace missing or too small")]:
        assert L.comba_status_string(code) == text
    assert L.comba_status_string(99) == b"unknown status"


def shape(B=2, T=300, H=4, dk=128, dv=128, N=None, cu=None, dtype=1, chunk=64, flags=0):
    s = binding._Shape()
    s.B, s.T, s.H, s.dk, s.dv = B, T, H, dk, dv
    s.num_seqs = B if N is None else N
    s.cu_seqlens = cu
    s.dtype, s.chunk, s.flags = dtype, chunk, flags
    return s


def ws(L, s, backward=0):
    return L.comba_workspace_size(ctypes.byref(s), backward)


def test_workspace_size_counts_chunks_and_heads(L):
    a = ws(L, shape(T=256))
    b = ws(L, shape(T=257))      # one more (ragged) chunk per sequence
    c = ws(L, shape(T=256, H=8))
    assert 0 < a < b and c > a
    assert ws(L, shape(), 1) > ws(L, shape(), 0)
    # bf16 needs less than fp32 storage
    assert ws(L, shape(dtype=1)) < ws(L, shape(dtype=0))
    # packed varlen: bound covers T/64 + N chunk slots
    assert ws(L, shape(B=1, T=65536, N=12, cu=FAKE)) > ws(L, shape(B=1, T=65536, N=1))


def test_workspace_per_unit_on_the_tcgen05_path(L):
    """bf16 dk = dv = 128, one (chunk, head) unit per 64 tokens: the forward keeps W^T, U^T,
    U_s^T (16 KB each), the log-decays (256 B), Atilde and the chunk state H^T (32 KB each) per
    unit, and no B^T (its scan forms B^T = U_s^T K itself); the backward adds E (16 KB), M
    (8 KB), Z^T (16 KB, for the C term its scan forms), dH'^T (32 KB) and two per-unit floats,
    and no C^T.  32 more units (and their 16-byte slot records) keep every sub-buffer a whole
    number of 256-byte alignment steps, so the differences are exact."""
    fwd_unit = 3 * 16384 + 256 + 2 * 32768
    bwd_unit = fwd_unit + 16384 + 8192 + 16384 + 32768 + 8
    for backward, unit in ((0, fwd_unit), (1, bwd_unit)):
        d = ws(L, shape(B=1, T=64 * 64, H=1), backward) - ws(L, shape(B=1, T=64 * 32, H=1), backward)
        assert d == 32 * (unit + 16), (backward, d)


@pytest.mark.parametrize("kw", [dict(dk=96), dict(dv=192), dict(dv=256, dk=64), dict(dv=256, dtype=0), dict(dv=640),
                                dict(chunk=32), dict(H=0), dict(B=0), dict(dtype=7),
                                dict(B=2, N=3), dict(B=2, cu=FAKE, N=2), dict(T=-1), dict(cu=FAKE + 4, B=1, N=1)])
def test_invalid_shapes_have_no_workspace(L, kw):
    assert ws(L, shape(**kw)) == 0


def test_fp32_backward_is_limited_to_head_dim_64(L):
    assert ws(L, shape(dtype=0, dk=64, dv=64), 1) > 0
    assert ws(L, shape(dtype=0, dk=128, dv=128), 1) == 0
    assert ws(L, shape(dtype=0, dk=128, dv=128), 0) > 0


def fwd(L, s, q=FAKE, k=FAKE, v=FAKE, alpha=FAKE, beta=FAKE, b=None, d=FAKE, h0=None, o=FAKE, hT=None,
        work=None, nbytes=0):
    return L.comba_chunk_fwd(ctypes.byref(s), q, k, v, alpha, beta, b, d, h0, o, hT, work, nbytes, None)


def test_forward_argument_validation(L):
    s = shape()
    assert fwd(L, s, q=None) == INVALID
    assert fwd(L, s, d=None) == INVALID
    assert fwd(L, s, o=None) == INVALID
    assert fwd(L, s, k=FAKE + 8) == INVALID          # misaligned
    assert fwd(L, s, b=FAKE + 4) == INVALID          # optional but misaligned
    assert fwd(L, s, work=None, nbytes=1 << 40) == WORKSPACE
    need = ws(L, s)
    assert fwd(L, s, work=FAKE, nbytes=need - 1) == WORKSPACE
    assert fwd(L, shape(dk=80)) == UNSUPPORTED
    # saving the backward's factors needs the backward-sized workspace
    sv = shape(flags=1)
    assert fwd(L, sv, work=FAKE, nbytes=ws(L, shape(), 0)) == WORKSPACE
    assert fwd(L, shape(flags=2)) == INVALID            # reuse is a backward flag
    assert fwd(L, shape(flags=8)) == INVALID            # unknown bit
    assert fwd(L, shape(flags=4), q=None) == INVALID    # iplr is a valid forward flag; q still required


def test_backward_argument_validation(L):
    s = shape()
    args = [FAKE] * 10 + [FAKE] * 8
    base = dict(zip(["q", "k", "v", "alpha", "beta", "b", "d", "h0", "dO", "dhT", "dq", "dk", "dv", "dalpha",
                     "dbeta", "db", "dd", "dh0"], args))

    def call(nbytes=0, work=None, **over):
        a = dict(base, **over)
        return L.comba_chunk_bwd(ctypes.byref(s), *[a[n] for n in base], work, nbytes, None)

    assert call(dO=None) == INVALID
    assert call(dalpha=None) == INVALID
    assert call(dd=None) == INVALID
    assert call() == WORKSPACE                       # db, dh0, dhT, h0, b may be NULL; workspace may not
    assert call(db=None, dh0=None, dhT=None, h0=None, b=None) == WORKSPACE
    assert call(work=FAKE, nbytes=ws(L, s, 1) - 256) == WORKSPACE
    s.flags = 1                                          # save is a forward flag
    assert call() == INVALID
    s.flags = 4 | 2                                      # iplr + reuse: valid flags, workspace still missing
    assert call() == WORKSPACE
    s.flags = 0


def test_recurrent_step_validation(L):
    def call(Bd=4, H=2, dk=128, dv=128, dtype=1, flags=0, **over):
        a = dict(q=FAKE, k=FAKE, v=FAKE, alpha=FAKE, beta=FAKE, b=None, d=FAKE, state=FAKE, o=FAKE)
        a.update(over)
        return L.comba_recurrent_step(Bd, H, dk, dv, dtype, a["q"], a["k"], a["v"], a["alpha"], a["beta"], a["b"],
                                      a["d"], a["state"], a["o"], flags, None)

    assert call(flags=8) == INVALID                  # only COMBA_IPLR is a step flag
    assert call(flags=1) == INVALID

    assert call(Bd=0) == INVALID
    assert call(dk=32) == UNSUPPORTED
    assert call(dtype=3) == INVALID
    assert call(state=None) == INVALID
    assert call(q=FAKE + 2) == INVALID


def test_gated_flag_rules(L):
    """COMBA_GATED selects the gated entry points; the plain ones reject it, and the gated
    workspace is larger (it holds the prologue's outputs)."""
    plain, gated_ws = ws(L, shape(), 1), ws(L, shape(flags=8), 1)
    assert gated_ws > plain
    assert fwd(L, shape(flags=8)) == INVALID
    s = shape(flags=0)
    args = [FAKE] * 12
    # the gated forward without COMBA_GATED in the shape is invalid
    assert L.comba_chunk_fwd_gated(ctypes.byref(s), *args, FAKE, 1 << 40, None) == INVALID
    s.flags = 8
    assert L.comba_chunk_fwd_gated(ctypes.byref(s), *args, None, 0, None) == WORKSPACE
    args[5] = None   # a is required
    assert L.comba_chunk_fwd_gated(ctypes.byref(s), *args, None, 0, None) == INVALID


def test_pk_flag_rules(L):
    """COMBA_PK selects the Comba-pk entry points; the plain and gated ones reject it, its
    workspace also holds q - d p, and p (and dp) are required."""
    plain, pk_ws = ws(L, shape(), 1), ws(L, shape(flags=16), 1)
    assert pk_ws > plain
    assert fwd(L, shape(flags=16)) == INVALID
    s = shape(flags=0)
    args = [FAKE] * 11   # q k v p alpha beta b d h0 o hT
    assert L.comba_chunk_fwd_pk(ctypes.byref(s), *args, FAKE, 1 << 40, None) == INVALID   # flag missing
    s.flags = 16 | 8
    assert L.comba_chunk_fwd_pk(ctypes.byref(s), *args, FAKE, 1 << 40, None) == INVALID   # not with gated
    s.flags = 16
    assert L.comba_chunk_fwd_pk(ctypes.byref(s), *args, None, 0, None) == WORKSPACE
    args[3] = None   # p is required
    assert L.comba_chunk_fwd_pk(ctypes.byref(s), *args, None, 0, None) == INVALID
    s.flags = 16 | 2
    bargs = [FAKE] * 20   # q k v p alpha beta b d h0 dO dhT dq dk dv dp dalpha dbeta db dd dh0
    assert L.comba_chunk_bwd_pk(ctypes.byref(s), *bargs, None, 0, None) == WORKSPACE
    bargs[14] = None   # dp is required
    assert L.comba_chunk_bwd_pk(ctypes.byref(s), *bargs, None, 0, None) == INVALID
    s.flags = 16 | 1   # the saving flag belongs to the forward
    assert L.comba_chunk_bwd_pk(ctypes.byref(s), *([FAKE] * 20), None, 0, None) == INVALID

    def step(flags=0, **over):
        a = dict(q=FAKE, k=FAKE, v=FAKE, p=FAKE, alpha=FAKE, beta=FAKE, b=None, d=FAKE, state=FAKE, o=FAKE)
        a.update(over)
        return L.comba_recurrent_step_pk(4, 2, 128, 128, 1, a["q"], a["k"], a["v"], a["p"], a["alpha"], a["beta"],
                                         a["b"], a["d"], a["state"], a["o"], flags, None)

    assert step(p=None) == INVALID
    assert step(flags=16) == INVALID
    assert step(p=FAKE + 4) == INVALID


def test_value_head_groups(L):
    """dv = 256 / 384 / 512 with dk = 128 (bf16) runs as groups of 128-wide value heads: the
    workspace grows with the value heads (and the backward's per-value-head key-side gradients)."""
    w128, w256, w512 = (ws(L, shape(dv=d), 1) for d in (128, 256, 512))
    assert 0 < w128 < w256 < w512
    assert ws(L, shape(dv=384), 0) > 0
    # the gated and pk forms take value-head groups too
    assert ws(L, shape(dv=256, flags=8), 1) > w256
    assert ws(L, shape(dv=256, flags=16), 1) > w256
    assert ws(L, shape(dv=256, H=65535 // 2 + 1)) == 0   # value heads H * 2 beyond the head limit

    def step(dv, dk=128, dtype=1):
        return L.comba_recurrent_step(4, 2, dk, dv, dtype, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, FAKE, FAKE, 0,
                                      None)
    assert step(256, dk=64) == UNSUPPORTED
    assert step(384) == UNSUPPORTED


def test_head_dim_256(L):
    """dk = 256 (bf16; plain, iplr, pk or gated form) runs as value heads 64 wide: dv = 64 .. 256 in steps of 64."""
    w64, w128, w256 = (ws(L, shape(dk=256, dv=d), 1) for d in (64, 128, 256))
    assert 0 < w64 < w128 < w256
    assert ws(L, shape(dk=256, dv=192), 0) > 0
    assert ws(L, shape(dk=256, dv=64, flags=4), 1) > 0
    for kw in (dict(dv=320), dict(dv=32), dict(dv=96), dict(dtype=0)):
        assert ws(L, shape(dk=256, **kw)) == 0, kw
    assert ws(L, shape(dk=256, dv=256, flags=8), 1) > ws(L, shape(dk=256, dv=256), 1)   # gated: the prologue's outputs
    # Comba-pk at head dim 256: the workspace also holds q - d p and, with value-head groups, the
    # per-value-head dp
    assert ws(L, shape(dk=256, dv=128, flags=16), 1) > ws(L, shape(dk=256, dv=128), 1)

    def step(dv, dk=256):
        return L.comba_recurrent_step(4, 2, dk, dv, 1, FAKE, FAKE, FAKE, FAKE, FAKE, None, FAKE, FAKE, FAKE, 0,
                                      None)
    assert step(384) == UNSUPPORTED
    assert step(256, dk=64) == UNSUPPORTED


def test_noalloc_forward_takes_only_the_plain_and_iplr_forms(L):
    """The allocation-free forward rejects flags it cannot honour (saved factors would sit in the
    shared static array out of the caller's reach; gated and pk have entry points of their own)
    before any CUDA call."""
    fn = L.comba_chunk_fwd_noalloc
    for flags in (1, 2, 8, 16, 1 | 4):
        s = shape(flags=flags)
        assert fn(ctypes.byref(s), *([FAKE] * 7), None, FAKE, None, None) == INVALID, flags
    s = shape(B=8, T=4096, H=16)
    assert fn(ctypes.byref(s), *([FAKE] * 7), None, FAKE, None, None) == WORKSPACE


def test_diagnostic_stall_flag_is_accepted_only_by_the_plain_chunk_calls(L):
    """COMBA_DIAG_STALL (32) is a flag of comba_chunk_fwd / comba_chunk_bwd: with it, validation goes
    on to the workspace check (it is accepted); an unknown bit next to it, and the allocation-free
    forward, reject it before any CUDA call."""
    assert fwd(L, shape(flags=32)) == WORKSPACE
    assert fwd(L, shape(flags=1 | 32)) == WORKSPACE
    assert fwd(L, shape(flags=32 | 64)) == INVALID
    fn = L.comba_chunk_fwd_noalloc
    s = shape(flags=32)
    assert fn(ctypes.byref(s), *([FAKE] * 7), None, FAKE, None, None) == INVALID


def test_header_compiles_as_c_and_takes_a_cuda_stream(tmp_path):
    """include/comba.h is plain C (C99, no CUDA include), and in C++ next to the CUDA runtime's
    header a cudaStream_t passes as the entry points' stream argument without a cast."""
    import shutil
    import subprocess
    inc = os.path.dirname(HEADER)
    gcc, gxx = shutil.which("gcc"), shutil.which("g++")
    if not gcc or not gxx:
        pytest.skip("no host compiler")
    c_src = tmp_path / "t.c"
    c_src.write_text('#include "comba.h"\nint main(void) { comba_stream_t s = 0; (void)s; return 0; }\n')
    r = subprocess.run([gcc, "-std=c99", "-Wall", "-Werror", "-I" + inc, "-c", str(c_src), "-o",
                        str(tmp_path / "t.o")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    cuda_inc = next((d for d in ("/usr/local/cuda/include",) if os.path.exists(os.path.join(d, "cuda_runtime_api.h"))),
                    None)
    if cuda_inc is None:
        pytest.skip("no CUDA runtime header")
    cc_src = tmp_path / "t.cc"
    cc_src.write_text('#include <cuda_runtime_api.h>\n#include "comba.h"\n'
                      'comba_status_t f(const comba_shape_t* s, cudaStream_t st) {\n'
                      '  return comba_chunk_fwd(s, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 0, st);\n}\n')
    r = subprocess.run([gxx, "-std=c++17", "-Wall", "-Werror", "-I" + inc, "-I" + cuda_inc, "-c", str(cc_src), "-o",
                        str(tmp_path / "t2.o")], capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
