"""ctypes binding of libsdm.so.  Functions take torch CUDA tensors (or raw integer
device pointers) and pass their addresses, sizes and the current CUDA stream."""
from __future__ import annotations

import ctypes
import os
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
_LIB_PATH = os.path.join(HERE, "lib", "libsdm.so")

DTYPE_F32, DTYPE_BF16 = 0, 1
ADDR_PROJECTED, ADDR_DIRECT = 0, 1
_STATUS = {0: "SDM_OK", 1: "SDM_ERR_INVALID_ARG", 2: "SDM_ERR_UNSUPPORTED", 4: "SDM_ERR_CUDA",
           5: "SDM_ERR_TIMEOUT", 6: "SDM_ERR_DEVICE"}


class SdmError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{_STATUS.get(status, status)}: {message}")
        self.status = status


class SdmShape(ctypes.Structure):
    _fields_ = [("B", ctypes.c_int32), ("H", ctypes.c_int32), ("T", ctypes.c_int32),
                ("d_k", ctypes.c_int32), ("d_v", ctypes.c_int32), ("N", ctypes.c_int64),
                ("k_write", ctypes.c_int32), ("k_read", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("addr", ctypes.c_int32)]

    @classmethod
    def make(cls, B, H, T, d_k, d_v, N, k_write, k_read, dtype="bf16", addr="projected") -> "SdmShape":
        dt = {"f32": DTYPE_F32, "bf16": DTYPE_BF16}[dtype] if isinstance(dtype, str) else int(dtype)
        ad = {"projected": ADDR_PROJECTED, "direct": ADDR_DIRECT}[addr] if isinstance(addr, str) else int(addr)
        return cls(B, H, T, d_k, d_v, N, k_write, k_read, dt, ad)

    def replace(self, **kw) -> "SdmShape":
        vals = {f: getattr(self, f) for f, _ in self._fields_}
        vals.update(kw)
        return SdmShape(**vals)


_lib = None
_lock = threading.Lock()
_VP, _SZ, _I32P = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p
_SHP = ctypes.POINTER(SdmShape)


def lib_path() -> str:
    return _LIB_PATH


def lib():
    """Load libsdm.so (built in-tree); raises if it has not been built."""
    global _lib
    with _lock:
        if _lib is None:
            if not os.path.exists(_LIB_PATH):
                raise RuntimeError(f"libsdm.so not found at {_LIB_PATH}: build it with "
                                   "paper_2607_07386_gb300.build.build() (no fallback exists)")
            L = ctypes.CDLL(_LIB_PATH)
            L.sdm_abi_version.restype = ctypes.c_int
            L.sdm_last_error.restype = ctypes.c_char_p
            L.sdm_workspace_bytes.restype = ctypes.c_size_t
            L.sdm_workspace_bytes.argtypes = [_SHP]
            L.sdm_init_memory.argtypes = [_SHP, _VP, _VP, _VP]
            fwd = [_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _I32P, _VP, _I32P, _VP, _VP, _SZ, _VP]
            L.sdm_forward.argtypes = fwd
            L.sdm_forward_m0.argtypes = [fwd[0], _VP] + fwd[1:]
            L.sdm_forward_m0.restype = ctypes.c_int
            L.sdm_decode_step.argtypes = fwd
            L.sdm_forward_lazy.argtypes = [fwd[0], _VP, _VP] + fwd[1:]
            L.sdm_forward_lazy.restype = ctypes.c_int
            L.sdm_lazy_workspace_bytes.restype = ctypes.c_size_t
            L.sdm_lazy_workspace_bytes.argtypes = [_SHP]
            L.sdm_materialize.argtypes = [_SHP, _VP, _VP, _VP, _VP]
            L.sdm_materialize.restype = ctypes.c_int
            L.sdm_recur_chunkwise.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _VP, _VP, _VP, ctypes.c_int32, _VP]
            L.sdm_recur_chunkwise.restype = ctypes.c_int
            L.sdm_undo_log_bytes.restype = ctypes.c_size_t
            L.sdm_undo_log_bytes.argtypes = [_SHP]
            L.sdm_recur_undo.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]
            L.sdm_recur_undo.restype = ctypes.c_int
            L.sdm_recur_backward.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP,
                                             _VP, _VP, _VP, _VP, _VP]
            L.sdm_recur_backward.restype = ctypes.c_int
            L.sdm_undo_code_bytes.restype = ctypes.c_size_t
            L.sdm_undo_code_bytes.argtypes = [_SHP, ctypes.c_int]
            L.sdm_undo_quantize.argtypes = [_SHP, _VP, ctypes.c_int, _VP, _VP, _VP]
            L.sdm_undo_quantize.restype = ctypes.c_int
            L.sdm_recur_backward_q.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _VP, _VP, ctypes.c_int, _VP,
                                               _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP]
            L.sdm_recur_backward_q.restype = ctypes.c_int
            L.sdm_gates.argtypes = [_SHP, ctypes.c_int32, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _VP]
            L.sdm_gates.restype = ctypes.c_int
            L.sdm_norm_gate.argtypes = [_SHP, _VP, _VP, _VP, ctypes.c_float, _VP, _VP]
            L.sdm_norm_gate.restype = ctypes.c_int
            L.sdm_gates_tensor_cores.argtypes = [_SHP, ctypes.c_int32]
            L.sdm_gates_tensor_cores.restype = ctypes.c_int
            L.sdm_head_mix.argtypes = [_SHP, ctypes.c_int32, _VP, _VP, _VP, _VP]
            L.sdm_head_mix.restype = ctypes.c_int
            L.sdm_access_stats_workspace_bytes.restype = ctypes.c_size_t
            L.sdm_access_stats_workspace_bytes.argtypes = [_SHP]
            L.sdm_access_stats.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _SZ, _VP]
            L.sdm_access_stats.restype = ctypes.c_int
            L.sdm_address.argtypes = [_SHP, _VP, _VP, _VP, _VP, _I32P, _VP, _I32P, _VP, _VP, _SZ, _VP]
            L.sdm_recur.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]
            L.sdm_recur_workspace_bytes.restype = ctypes.c_size_t
            L.sdm_recur_workspace_bytes.argtypes = [_SHP]
            L.sdm_device_status.argtypes = [ctypes.POINTER(ctypes.c_int32), _VP]
            L.sdm_recur_noalloc.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _VP, _VP, _VP, _VP]
            L.sdm_recur_noalloc.restype = ctypes.c_int
            L.sdm_device_stats.argtypes = [ctypes.POINTER(ctypes.c_uint32), ctypes.c_int, _VP]
            L.sdm_device_stats.restype = ctypes.c_int
            L.sdm_test_scores.argtypes = [_SHP, _VP, _VP, _VP, _VP, _VP, _VP, _SZ, _VP]
            L.sdm_test_scores.restype = ctypes.c_int
            L.sdm_recur_plan.argtypes = [_SHP, ctypes.POINTER(ctypes.c_int32), ctypes.c_int]
            L.sdm_recur_plan.restype = ctypes.c_int
            L.sdm_test_recur_wait_timeout.argtypes = [_SHP, _I32P, _VP, _I32P, _VP, _VP, _VP, _VP, _VP, _VP, _VP,
                                                      _SZ, ctypes.c_int64, _VP]
            L.sdm_test_recur_wait_timeout.restype = ctypes.c_int
            for f in ("sdm_init_memory", "sdm_forward", "sdm_decode_step", "sdm_address", "sdm_recur",
                      "sdm_device_status"):
                getattr(L, f).restype = ctypes.c_int
            _lib = L
    return _lib


def abi_version() -> int:
    return lib().sdm_abi_version()


def last_error() -> str:
    return lib().sdm_last_error().decode()


def _check(status: int):
    if status != 0:
        raise SdmError(status, last_error())


def _ptr(x):
    """Address of a tensor (must be contiguous), an int, or None."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if not x.is_contiguous():
        raise ValueError("tensors passed to libsdm must be contiguous")
    if x.device.type != "cuda":
        raise ValueError("tensors passed to libsdm must live on a CUDA device")
    return x.data_ptr()


def _stream(stream):
    if stream is None:
        import torch
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _nbytes(x):
    return x.numel() * x.element_size() if x is not None and not isinstance(x, int) else None


def workspace_bytes(shape: SdmShape) -> int:
    n = lib().sdm_workspace_bytes(ctypes.byref(shape))
    if n == 0:
        raise SdmError(1, last_error())
    return n


def init_memory(shape: SdmShape, M0, mem, stream=None):
    _check(lib().sdm_init_memory(ctypes.byref(shape), _ptr(M0), _ptr(mem), _stream(stream)))


def address(shape: SdmShape, P_q, P_k, q, k, idx_w, w_w, idx_r, w_r, workspace, stream=None, workspace_nbytes=None):
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_address(ctypes.byref(shape), _ptr(P_q), _ptr(P_k), _ptr(q), _ptr(k), _ptr(idx_w), _ptr(w_w),
                             _ptr(idx_r), _ptr(w_r), _ptr(workspace), nb, _stream(stream)))


def forward(shape: SdmShape, P_q, P_k, q, k, v, alpha, beta, mem, y, workspace, idx_w=None, w_w=None,
            idx_r=None, w_r=None, stream=None, workspace_nbytes=None):
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_forward(ctypes.byref(shape), _ptr(P_q), _ptr(P_k), _ptr(q), _ptr(k), _ptr(v), _ptr(alpha),
                             _ptr(beta), _ptr(mem), _ptr(y), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r),
                             _ptr(workspace), nb, _stream(stream)))


def forward_m0(shape: SdmShape, M0, P_q, P_k, q, k, v, alpha, beta, mem, y, workspace, idx_w=None, w_w=None,
               idx_r=None, w_r=None, stream=None, workspace_nbytes=None):
    """sdm_forward_m0: mem = M0 broadcast (overlapping the addressing), then the forward pass."""
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_forward_m0(ctypes.byref(shape), _ptr(M0), _ptr(P_q), _ptr(P_k), _ptr(q), _ptr(k), _ptr(v),
                                _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), _ptr(idx_w), _ptr(w_w), _ptr(idx_r),
                                _ptr(w_r), _ptr(workspace), nb, _stream(stream)))


def lazy_workspace_bytes(shape: SdmShape) -> int:
    n = lib().sdm_lazy_workspace_bytes(ctypes.byref(shape))
    if n == 0:
        raise SdmError(1, last_error())
    return n


def touched_words(shape: SdmShape) -> int:
    """uint32 words of one chain's touched bitmap (ceil(N / 32))."""
    return (shape.N + 31) // 32


def forward_lazy(shape: SdmShape, M0, touched, P_q, P_k, q, k, v, alpha, beta, mem, y, workspace, idx_w=None,
                 w_w=None, idx_r=None, w_r=None, stream=None, workspace_nbytes=None):
    """sdm_forward_lazy: the forward pass on a copy-on-write memory seeded from M0; touched is
    the [B, H, ceil(N/32)] uint32 (int32 tensors work too) bitmap of written slots."""
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_forward_lazy(ctypes.byref(shape), _ptr(M0), _ptr(touched), _ptr(P_q), _ptr(P_k), _ptr(q), _ptr(k),
                                  _ptr(v), _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), _ptr(idx_w), _ptr(w_w),
                                  _ptr(idx_r), _ptr(w_r), _ptr(workspace), nb, _stream(stream)))


def materialize(shape: SdmShape, M0, touched, mem, stream=None):
    """sdm_materialize: write M0's rows into the untouched slots of mem."""
    _check(lib().sdm_materialize(ctypes.byref(shape), _ptr(M0), _ptr(touched), _ptr(mem), _stream(stream)))


def recur_chunkwise(shape: SdmShape, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, chunk: int, stream=None):
    """sdm_recur_chunkwise: the recurrence in chunkwise (WY) form, chunks of `chunk` <= 32 tokens."""
    _check(lib().sdm_recur_chunkwise(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r), _ptr(v),
                                     _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), int(chunk), _stream(stream)))


def undo_log_bytes(shape: SdmShape) -> int:
    n = lib().sdm_undo_log_bytes(ctypes.byref(shape))
    if n == 0 and shape.B * shape.H * shape.T * shape.k_write > 0:
        raise SdmError(1, last_error())
    return n


def recur_undo(shape: SdmShape, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, undo, workspace, stream=None,
               workspace_nbytes=None):
    """sdm_recur_undo: sdm_recur plus the undo log [B, H, T, k_write, d_v] of the backward."""
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_recur_undo(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r), _ptr(v),
                                _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), _ptr(undo), _ptr(workspace), nb,
                                _stream(stream)))


def recur_backward(shape: SdmShape, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, undo, dy, dv, dalpha, dbeta,
                   dw_w, dw_r, dM, stream=None):
    """sdm_recur_backward: gradients of sum <dy, y>; restores mem from M_T to M_0 with the undo log."""
    _check(lib().sdm_recur_backward(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r), _ptr(v),
                                    _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(undo), _ptr(dy), _ptr(dv),
                                    _ptr(dalpha), _ptr(dbeta), _ptr(dw_w), _ptr(dw_r), _ptr(dM), _stream(stream)))


UNDO_KINDS = {"fp8": 1, "int4": 2}


def undo_code_bytes(shape: SdmShape, kind: str) -> int:
    """Bytes of the codes of a quantised undo log ("fp8" or "int4"); the scales are
    B*H*T*k_write float32 more."""
    n = lib().sdm_undo_code_bytes(ctypes.byref(shape), UNDO_KINDS[kind])
    if n == 0 and shape.B * shape.H * shape.T * shape.k_write > 0:
        raise SdmError(1, last_error())
    return n


def undo_quantize(shape: SdmShape, undo, kind: str, codes, scales, stream=None):
    """sdm_undo_quantize: fp8 / int4 snapshot of the undo log, one float32 scale per row."""
    _check(lib().sdm_undo_quantize(ctypes.byref(shape), _ptr(undo), UNDO_KINDS[kind], _ptr(codes), _ptr(scales),
                                   _stream(stream)))


def recur_backward_q(shape: SdmShape, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, kind: str, codes, scales, dy, dv,
                     dalpha, dbeta, dw_w, dw_r, dM, stream=None):
    """sdm_recur_backward_q: sdm_recur_backward reading the log from a quantised snapshot."""
    _check(lib().sdm_recur_backward_q(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r), _ptr(v),
                                      _ptr(alpha), _ptr(beta), _ptr(mem), UNDO_KINDS[kind], _ptr(codes), _ptr(scales),
                                      _ptr(dy), _ptr(dv), _ptr(dalpha), _ptr(dbeta), _ptr(dw_w), _ptr(dw_r), _ptr(dM),
                                      _stream(stream)))


def gates(shape: SdmShape, d_model: int, x, W_a, W_b, b_dt, A, alpha, beta, stream=None):
    """sdm_gates: alpha, beta [B, H, T] from the layer input x [B, T, d_model]."""
    _check(lib().sdm_gates(ctypes.byref(shape), int(d_model), _ptr(x), _ptr(W_a), _ptr(W_b), _ptr(b_dt), _ptr(A),
                           _ptr(alpha), _ptr(beta), _stream(stream)))


def gates_tensor_cores(shape: SdmShape, d_model: int) -> bool:
    """Whether sdm_gates runs its projections on the tensor cores for this shape."""
    return bool(lib().sdm_gates_tensor_cores(ctypes.byref(shape), int(d_model)))


def head_mix(shape: SdmShape, d_model: int, z, W_o, out, stream=None):
    """sdm_head_mix: out [B*T, d_model] = z [B*T, H*d_v] W_o^T on the tensor cores (bf16)."""
    _check(lib().sdm_head_mix(ctypes.byref(shape), int(d_model), _ptr(z), _ptr(W_o), _ptr(out), _stream(stream)))


def norm_gate(shape: SdmShape, y, g, gamma, eps: float, z, stream=None):
    """sdm_norm_gate: z [B, T, H, d_v] = g * gamma * RMSNorm(y) per head."""
    _check(lib().sdm_norm_gate(ctypes.byref(shape), _ptr(y), _ptr(g), _ptr(gamma), float(eps), _ptr(z), _stream(stream)))


def access_stats_workspace_bytes(shape: SdmShape) -> int:
    n = lib().sdm_access_stats_workspace_bytes(ctypes.byref(shape))
    if n == 0:
        raise SdmError(1, last_error())
    return n


def access_stats(shape: SdmShape, idx_w, w_w, idx_r, w_r, out, workspace, stream=None, workspace_nbytes=None):
    """sdm_access_stats: float64 sums of the access diagnostics into the device tensor out
    (4 + k_write + k_read entries)."""
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_access_stats(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r), _ptr(out),
                                  _ptr(workspace), nb, _stream(stream)))


def decode_step(shape: SdmShape, P_q, P_k, q, k, v, alpha, beta, mem, y, workspace, idx_w=None, w_w=None,
                idx_r=None, w_r=None, stream=None, workspace_nbytes=None):
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_decode_step(ctypes.byref(shape), _ptr(P_q), _ptr(P_k), _ptr(q), _ptr(k), _ptr(v),
                                 _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), _ptr(idx_w), _ptr(w_w), _ptr(idx_r),
                                 _ptr(w_r), _ptr(workspace), nb, _stream(stream)))


def recur_workspace_bytes(shape: SdmShape) -> int:
    n = lib().sdm_recur_workspace_bytes(ctypes.byref(shape))
    if n == 0:
        raise SdmError(1, last_error())
    return n


def recur(shape: SdmShape, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, workspace, stream=None,
          workspace_nbytes=None):
    nb = workspace_nbytes if workspace_nbytes is not None else (_nbytes(workspace) or 0)
    _check(lib().sdm_recur(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r), _ptr(v),
                           _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), _ptr(workspace), nb, _stream(stream)))


# Fixed device scratch behind recur_noalloc (SDM_RECUR_NOALLOC_SCRATCH_BYTES in include/sdm.h).
RECUR_NOALLOC_SCRATCH_BYTES = 16 << 20


def recur_noalloc(shape: SdmShape, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, stream=None):
    """sdm_recur_noalloc: the recurrence without a workspace (fixed device scratch, no allocation)."""
    _check(lib().sdm_recur_noalloc(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r), _ptr(v),
                                   _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), _stream(stream)))


def device_status(stream=None) -> int:
    """Read and clear the device status word (0 = clean; bit 2 = a bounded wait gave up).
    Raises SdmError only if reading it failed."""
    code = ctypes.c_int32(0)
    st = lib().sdm_device_status(ctypes.byref(code), _stream(stream))
    if st not in (0, 5, 6):
        _check(st)
    return int(code.value)


def test_scores(shape: SdmShape, P_q, P_k, q, k, scores, workspace, stream=None):
    """sdm_test_scores: raw tensor-core scores [2, H, B*T, 2 sqrt(N)] float32 into `scores`."""
    _check(lib().sdm_test_scores(ctypes.byref(shape), _ptr(P_q), _ptr(P_k), _ptr(q), _ptr(k), _ptr(scores),
                                 _ptr(workspace), _nbytes(workspace) or 0, _stream(stream)))


RECUR_PLAN_FIELDS = ("dch", "nsplit", "spt", "la", "w", "p")


def recur_plan(shape: SdmShape) -> dict:
    """sdm_recur_plan: the recurrence's launch plan for `shape` (host only)."""
    arr = (ctypes.c_int32 * len(RECUR_PLAN_FIELDS))()
    _check(lib().sdm_recur_plan(ctypes.byref(shape), arr, len(RECUR_PLAN_FIELDS)))
    return {name: int(arr[i]) for i, name in enumerate(RECUR_PLAN_FIELDS)}


def test_recur_wait_timeout(shape: SdmShape, idx_w, w_w, idx_r, w_r, v, alpha, beta, mem, y, workspace,
                            wait_cycles: int, stream=None):
    """sdm_test_recur_wait_timeout: the token-interleaved recurrence with a withheld progress
    word and a short wait limit (the bounded waits must run out and set status bit 2)."""
    _check(lib().sdm_test_recur_wait_timeout(ctypes.byref(shape), _ptr(idx_w), _ptr(w_w), _ptr(idx_r), _ptr(w_r),
                                             _ptr(v), _ptr(alpha), _ptr(beta), _ptr(mem), _ptr(y), _ptr(workspace),
                                             _nbytes(workspace) or 0, int(wait_cycles), _stream(stream)))


STAT_NAMES = ("half_band", "half_full", "comb_band", "comb_full", "select_retry", "comb_merge", "band_f64", "serial",
              "half_band_entries", "comb_band_entries")


def device_stats(stream=None) -> dict:
    """Read and clear the selection event counters (see sdm_device_stats in include/sdm.h)."""
    n = len(STAT_NAMES)
    arr = (ctypes.c_uint32 * n)()
    _check(lib().sdm_device_stats(arr, n, _stream(stream)))
    return {name: int(arr[i]) for i, name in enumerate(STAT_NAMES)}
