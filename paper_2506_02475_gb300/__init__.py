"""GB300-native (sm_103a) Comba chunk-parallel library.

Comba (arXiv 2506.02475) is a bilinear RNN with a scalar-plus-low-rank state
transition, state feedback and output feedback.  This package is the hot path
of its training and inference: ``libcomba.so`` (C ABI in ``include/comba.h``,
CUDA kernels under ``csrc/``) and a thin ctypes binding with the same names.
"""
from .binding import (  # noqa: F401
    CombaError,
    comba_chunk_bwd,
    comba_chunk_bwd_gated,
    comba_chunk_bwd_pk,
    comba_chunk_fwd,
    comba_chunk_fwd_gated,
    comba_chunk_fwd_pk,
    comba_recurrent_step,
    comba_recurrent_step_pk,
    comba_workspace_size,
    comba_workspace_status,
    lib,
    library_path,
)
