"""GB300-native Sparse Delta Memory (arXiv 2607.07386) hot path.

A thin ctypes binding of ``libsdm.so`` (C ABI in ``include/sdm.h``): argument
marshalling only; every step runs in the library's sm_103a kernels.  The
library is built in-tree by ``paper_2607_07386_gb300.build.build()``; using any
entry point without it raises ``RuntimeError`` (there is no fallback).
"""
from ._binding import (  # noqa: F401
    ADDR_DIRECT, ADDR_PROJECTED, DTYPE_BF16, DTYPE_F32, SdmError, SdmShape, abi_version, address,
    decode_step, device_stats, device_status, forward, forward_m0, init_memory, last_error, lib, lib_path, recur, recur_noalloc,
    recur_workspace_bytes, workspace_bytes, RECUR_NOALLOC_SCRATCH_BYTES, forward_lazy, lazy_workspace_bytes,
    materialize, touched_words, access_stats, access_stats_workspace_bytes, gates, norm_gate, gates_tensor_cores, head_mix,
    undo_log_bytes, recur_undo, recur_backward, undo_code_bytes, undo_quantize, recur_backward_q, recur_chunkwise, recur_plan, test_recur_wait_timeout,
    RECUR_PLAN_FIELDS, test_scores,
)
