"""Host-side checks of libsdm.so: it builds, loads, exports every entry point that
include/sdm.h declares, and rejects bad arguments before launching anything.

No call here reaches a kernel launch: every argument set fails validation first
(the fake device addresses below are never dereferenced)."""
import ctypes
import os
import re
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sdm.h")


@pytest.fixture(scope="module")
def sdm():
    import paper_2607_07386_gb300 as sdm
    from paper_2607_07386_gb300 import build as B
    if not os.path.exists(sdm.lib_path()):
        if shutil.which("nvcc") is None and not os.path.exists("/usr/local/cuda/bin/nvcc"):
            pytest.skip("nvcc not available to build libsdm.so")
        B.build()
    return sdm


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:sdm_status|int|size_t|const\s+char\s*\*)\s+(sdm_\w+)\s*\(", text, flags=re.M)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for required in ("sdm_abi_version", "sdm_last_error", "sdm_workspace_bytes", "sdm_init_memory",
                     "sdm_forward", "sdm_decode_step", "sdm_recur", "sdm_address", "sdm_device_status",
                     "sdm_recur_workspace_bytes", "sdm_device_stats", "sdm_forward_m0"):
        assert required in names


def test_library_exports_every_declared_symbol(sdm):
    L = sdm.lib()
    for name in declared_functions():
        assert hasattr(L, name), name
    assert sdm.abi_version() == 2


def test_shape_struct_layout_matches_header(sdm):
    S = sdm.SdmShape
    assert ctypes.sizeof(S) == 48
    assert S.N.offset == 24 and S.k_write.offset == 32 and S.addr.offset == 44


def _shape(sdm, **kw):
    base = dict(B=2, H=2, T=16, d_k=32, d_v=32, N=1024, k_write=8, k_read=8, dtype="bf16", addr="projected")
    base.update(kw)
    return sdm.SdmShape.make(**base)


@pytest.mark.parametrize("kw,frag", [
    (dict(N=1000), "perfect square"),
    (dict(k_write=33), "sqrt(N)"),
    (dict(k_read=0), "[1, 64]"),
    (dict(d_v=3), "multiple of 16"),
    (dict(addr="direct"), "DIRECT"),
    (dict(B=-1), ">= 0"),
    (dict(d_k=300), "d_k > 256"),
])
def test_workspace_bytes_rejects_bad_shapes(sdm, kw, frag):
    n = sdm.lib().sdm_workspace_bytes(ctypes.byref(_shape(sdm, **kw)))
    assert n == 0
    assert frag in sdm.last_error()


def test_workspace_bytes_covers_selection_buffers(sdm):
    s = sdm.SdmShape.make(8, 16, 4096, 128, 128, 262144, 32, 32, "bf16")
    n = sdm.workspace_bytes(s)
    assert n >= 4 * 8 * 16 * 4096 * 32 * 4
    assert sdm.workspace_bytes(s) == n   # deterministic


FAKE = 0x7F0000000000   # never dereferenced: each call below fails validation first


def _fwd(sdm, shape, **over):
    L = sdm.lib()
    args = dict(P_q=FAKE, P_k=FAKE + 0x100000, q=FAKE + 0x200000, k=FAKE + 0x300000, v=FAKE + 0x400000,
                alpha=FAKE + 0x500000, beta=FAKE + 0x600000, mem=FAKE + 0x10000000, y=FAKE + 0x700000,
                ws=FAKE + 0x40000000, ws_bytes=0)
    args.update(over)
    return L.sdm_forward(ctypes.byref(shape), args["P_q"], args["P_k"], args["q"], args["k"], args["v"],
                         args["alpha"], args["beta"], args["mem"], args["y"], None, None, None, None, args["ws"],
                         args["ws_bytes"], None)


def test_forward_rejects_null_misaligned_small_workspace_and_aliasing(sdm):
    s = _shape(sdm)
    assert _fwd(sdm, s, q=None) == 1 and "q is NULL" in sdm.last_error()
    assert _fwd(sdm, s, q=FAKE + 1) == 1 and "aligned" in sdm.last_error()
    assert _fwd(sdm, s, v=FAKE + 8) == 1 and "v is not 16-byte aligned" in sdm.last_error()
    assert _fwd(sdm, s, ws_bytes=16) == 1 and "workspace too small" in sdm.last_error()
    need = sdm.workspace_bytes(s)
    assert _fwd(sdm, s, ws_bytes=need, y=FAKE + 0x10000000 + 4096) == 1 and "mem overlaps y" in sdm.last_error()
    assert _fwd(sdm, s, ws_bytes=need, ws=FAKE + 0x10000000) == 1 and "overlaps workspace" in sdm.last_error()
    assert sdm.lib().sdm_forward(None, *([None] * 14), 0, None) == 1


def test_lazy_workspace_covers_first_writer_table(sdm):
    s = sdm.SdmShape.make(8, 16, 4096, 128, 128, 262144, 32, 32, "bf16")
    assert sdm.lazy_workspace_bytes(s) >= sdm.workspace_bytes(s) + 8 * 16 * 262144 * 4
    assert sdm.touched_words(s) == 8192


def test_forward_lazy_and_materialize_reject_bad_bitmaps(sdm):
    s = _shape(sdm)
    L = sdm.lib()
    need = sdm.lazy_workspace_bytes(s)
    mem = FAKE + 0x10000000

    def lazy(touched, M0=FAKE + 0x800000):
        return L.sdm_forward_lazy(ctypes.byref(s), M0, touched, FAKE, FAKE + 0x100000, FAKE + 0x200000,
                                  FAKE + 0x300000, FAKE + 0x400000, FAKE + 0x500000, FAKE + 0x600000, mem,
                                  FAKE + 0x700000, None, None, None, None, FAKE + 0x40000000, need, None)
    assert lazy(None) == 1 and "touched is NULL" in sdm.last_error()
    assert lazy(FAKE + 0x900002) == 1 and "touched is not 4-byte aligned" in sdm.last_error()
    assert lazy(mem + 4096) == 1 and "mem overlaps touched" in sdm.last_error()
    assert lazy(FAKE + 0x700000) == 1 and "touched overlaps y" in sdm.last_error()
    assert lazy(FAKE + 0x900000, M0=None) == 1 and "M0 is NULL" in sdm.last_error()
    assert L.sdm_forward_lazy(ctypes.byref(s), FAKE + 0x800000, FAKE + 0x900000, *([FAKE] * 9), None, None, None,
                              None, FAKE + 0x40000000, 16, None) == 1 and "too small" in sdm.last_error()
    assert L.sdm_materialize(ctypes.byref(s), FAKE, mem + 64, mem, None) == 1 and "overlaps" in sdm.last_error()
    assert L.sdm_materialize(ctypes.byref(s), None, FAKE, mem, None) == 1 and "M0 is NULL" in sdm.last_error()


def test_access_stats_rejects_bad_arguments(sdm):
    s = _shape(sdm)
    L = sdm.lib()
    need = sdm.access_stats_workspace_bytes(s)
    assert need >= 2 * 2 * 2 * (1024 // 32) * 4
    args = [FAKE, FAKE + 0x100000, FAKE + 0x200000, FAKE + 0x300000]
    assert L.sdm_access_stats(ctypes.byref(s), *args, None, FAKE + 0x400000, need, None) == 1
    assert "out is NULL" in sdm.last_error()
    assert L.sdm_access_stats(ctypes.byref(s), *args, FAKE + 0x500004, FAKE + 0x400000, need, None) == 1
    assert "8-byte aligned" in sdm.last_error()
    assert L.sdm_access_stats(ctypes.byref(s), *args, FAKE + 0x500000, FAKE + 0x400000, 16, None) == 1
    assert "too small" in sdm.last_error()
    assert L.sdm_access_stats(ctypes.byref(s), *args, FAKE + 0x400000, FAKE + 0x400000, need, None) == 1
    assert "out overlaps workspace" in sdm.last_error()


def test_gates_and_norm_gate_reject_bad_arguments(sdm):
    s = _shape(sdm)
    L = sdm.lib()
    gate_args = lambda **o: [o.get(k, v) for k, v in (("x", FAKE), ("W_a", FAKE + 0x100000), ("W_b", FAKE + 0x200000),
                                                       ("b_dt", FAKE + 0x300000), ("A", FAKE + 0x400000),
                                                       ("alpha", FAKE + 0x500000), ("beta", FAKE + 0x600000))]
    assert L.sdm_gates(ctypes.byref(s), 12, *gate_args(), None) == 2 and "multiple of 16" in sdm.last_error()
    assert L.sdm_gates(ctypes.byref(s), 64, *gate_args(x=None), None) == 1 and "x is NULL" in sdm.last_error()
    assert L.sdm_gates(ctypes.byref(s), 64, *gate_args(alpha=FAKE + 8), None) == 1 and "overlaps x" in sdm.last_error()
    assert L.sdm_gates(ctypes.byref(s), 64, *gate_args(beta=FAKE + 0x500000), None) == 1
    assert "alpha overlaps beta" in sdm.last_error()
    big = _shape(sdm, H=33, N=4096, k_write=8, k_read=8)
    assert L.sdm_gates(ctypes.byref(big), 64, *gate_args(), None) == 2 and "H > 32" in sdm.last_error()
    ng = lambda **o: L.sdm_norm_gate(ctypes.byref(o.pop("shape", s)), o.get("y", FAKE), o.get("g", FAKE + 0x100000),
                                     o.get("gamma", FAKE + 0x200000), ctypes.c_float(o.get("eps", 1e-6)),
                                     o.get("z", FAKE + 0x300000), None)
    assert ng(z=None) == 1 and "z is NULL" in sdm.last_error()
    assert ng(z=FAKE + 0x100000 + 64) == 1 and "z overlaps g" in sdm.last_error()
    assert ng(eps=-1.0) == 1 and "eps" in sdm.last_error()
    assert ng(shape=_shape(sdm, d_v=1024)) == 2 and "1024 bytes" in sdm.last_error()


def test_backward_entry_points_reject_bad_arguments(sdm):
    s = _shape(sdm)
    L = sdm.lib()
    assert sdm.undo_log_bytes(s) == 2 * 2 * 16 * 8 * 32 * 2
    base = [FAKE, FAKE + 0x100000, FAKE + 0x200000, FAKE + 0x300000, FAKE + 0x400000, FAKE + 0x500000,
            FAKE + 0x600000, FAKE + 0x10000000, FAKE + 0x700000]
    assert L.sdm_recur_undo(ctypes.byref(s), *base, None, FAKE + 0x40000000, 1 << 30, None) == 1
    assert "undo is NULL" in sdm.last_error()
    assert L.sdm_recur_undo(ctypes.byref(s), *base, FAKE + 0x10000000 + 256, FAKE + 0x40000000, 1 << 30, None) == 1
    assert "undo overlaps" in sdm.last_error()
    outs = [FAKE + 0x20000000 + i * 0x1000000 for i in range(6)]
    bw = lambda shape, **o: L.sdm_recur_backward(ctypes.byref(shape), *base[:8], o.get("undo", FAKE + 0x800000),
                                                 FAKE + 0x900000, *outs, None)
    assert bw(_shape(sdm, d_v=48)) == 2 and "multiple of 32" in sdm.last_error()
    assert bw(s, undo=None) == 1 and "undo is NULL" in sdm.last_error()
    assert bw(s, undo=FAKE + 0x10000000) == 1 and "mem overlaps undo" in sdm.last_error()


def test_snapshot_entry_points_size_and_reject_bad_arguments(sdm):
    s = _shape(sdm)
    L = sdm.lib()
    rows = 2 * 2 * 16 * 8
    assert sdm.undo_code_bytes(s, "fp8") == rows * 32 and sdm.undo_code_bytes(s, "int4") == rows * 16
    assert L.sdm_undo_code_bytes(ctypes.byref(s), 3) == 0
    q = lambda shape, kind, **o: L.sdm_undo_quantize(ctypes.byref(shape), o.get("undo", FAKE), kind,
                                                     o.get("codes", FAKE + 0x100000), o.get("scales", FAKE + 0x200000),
                                                     None)
    assert q(s, 3) == 1 and "kind" in sdm.last_error()
    assert q(_shape(sdm, d_v=48), 1) == 2 and "multiple of 32" in sdm.last_error()
    assert q(s, 1, codes=FAKE + 0x100) == 1 and "overlap" in sdm.last_error()
    assert q(s, 2, scales=None) == 1 and "scales is NULL" in sdm.last_error()
    base = [FAKE, FAKE + 0x100000, FAKE + 0x200000, FAKE + 0x300000, FAKE + 0x400000, FAKE + 0x500000,
            FAKE + 0x600000, FAKE + 0x10000000]
    outs = [FAKE + 0x20000000 + i * 0x1000000 for i in range(6)]
    bq = lambda shape, kind, **o: L.sdm_recur_backward_q(ctypes.byref(shape), *base, kind, o.get("codes", FAKE + 0x800000),
                                                         o.get("scales", FAKE + 0x880000), FAKE + 0x900000, *outs, None)
    assert bq(s, 0) == 1 and "kind" in sdm.last_error()
    assert bq(s, 1, scales=None) == 1 and "scales is NULL" in sdm.last_error()
    assert bq(s, 2, codes=FAKE + 0x10000000) == 1 and "mem overlaps codes" in sdm.last_error()
    assert bq(_shape(sdm, N=4096, k_write=40), 1) == 2 and "at most 32" in sdm.last_error()


def test_head_mix_and_tensor_core_gates_reject_or_route(sdm):
    L = sdm.lib()
    s = _shape(sdm, H=16, d_v=128)
    hm = lambda shape, d_model, **o: L.sdm_head_mix(ctypes.byref(shape), d_model, o.get("z", FAKE),
                                                    o.get("W_o", FAKE + 0x1000000), o.get("out", FAKE + 0x2000000), None)
    assert hm(_shape(sdm, H=16, d_v=128, dtype="f32"), 2048) == 2 and "bf16" in sdm.last_error()
    assert hm(s, 48) == 2 and "multiple of 32" in sdm.last_error()
    assert hm(s, 2048, out=FAKE + 0x10) == 1 and "out overlaps z" in sdm.last_error()
    assert hm(s, 2048, W_o=None) == 1 and "W_o is NULL" in sdm.last_error()
    # the gates take the tensor cores for bf16 storage with H = 16 or 32 and d_model % 8 == 0
    assert sdm.gates_tensor_cores(s, 2048) and sdm.gates_tensor_cores(_shape(sdm, H=32), 64)
    assert not sdm.gates_tensor_cores(_shape(sdm, H=8), 64)
    assert not sdm.gates_tensor_cores(_shape(sdm, H=16, dtype="f32"), 64)
    assert not sdm.gates_tensor_cores(s, 2044)


def test_chunkwise_rejects_bad_chunks_and_rows(sdm):
    s = _shape(sdm)
    L = sdm.lib()
    args = [FAKE, FAKE + 0x100000, FAKE + 0x200000, FAKE + 0x300000, FAKE + 0x400000, FAKE + 0x500000,
            FAKE + 0x600000, FAKE + 0x10000000, FAKE + 0x700000]
    assert L.sdm_recur_chunkwise(ctypes.byref(s), *args, 0, None) == 1 and "[1, 32]" in sdm.last_error()
    assert L.sdm_recur_chunkwise(ctypes.byref(s), *args, 33, None) == 1 and "[1, 32]" in sdm.last_error()
    wide = _shape(sdm, d_v=512)
    assert L.sdm_recur_chunkwise(ctypes.byref(wide), *args, 8, None) == 2 and "d_v > 256" in sdm.last_error()
    assert L.sdm_recur_chunkwise(ctypes.byref(s), *args[:7], FAKE + 0x100000, FAKE + 0x700000, 8, None) == 1
    assert "mem overlaps" in sdm.last_error()


def test_decode_step_requires_T_equal_1(sdm):
    s = _shape(sdm, T=2)
    L = sdm.lib()
    st = L.sdm_decode_step(ctypes.byref(s), *([FAKE] * 9), None, None, None, None, FAKE, 1 << 30, None)
    assert st == 1 and "T == 1" in sdm.last_error()


def test_init_memory_and_recur_reject_overlap(sdm):
    s = _shape(sdm)
    L = sdm.lib()
    assert L.sdm_init_memory(ctypes.byref(s), FAKE, FAKE + 64, None) == 1 and "overlaps" in sdm.last_error()
    assert L.sdm_init_memory(ctypes.byref(s), None, FAKE, None) == 1
    st = L.sdm_recur(ctypes.byref(s), FAKE + 0x10000000, FAKE + 0x100000, FAKE + 0x200000, FAKE + 0x300000,
                     FAKE + 0x400000, FAKE + 0x500000, FAKE + 0x600000, FAKE + 0x10000000, FAKE + 0x700000,
                     FAKE + 0x40000000, 1 << 30, None)
    assert st == 1 and "mem overlaps idx_w" in sdm.last_error()


def test_binding_fails_loudly_without_library(tmp_path, monkeypatch):
    import paper_2607_07386_gb300._binding as b
    monkeypatch.setattr(b, "_LIB_PATH", str(tmp_path / "missing.so"))
    monkeypatch.setattr(b, "_lib", None)
    with pytest.raises(RuntimeError, match="not found"):
        b.lib()


def test_recur_plan_reports_the_launch_shape(sdm):
    """sdm_recur_plan is host-only: the short-T parity shapes of the GPU tests reach the kernel
    variant the bench runs at full size (the plan depends on T only through T == 1)."""
    import synth
    full = synth.LAYER_1P4B
    mk = lambda c, T: sdm.SdmShape.make(c.B, c.H, T, c.d_k, c.d_v, c.N, c.k_write, c.k_read, c.dtype)
    bench_plan = sdm.recur_plan(mk(full, full.T))
    assert sdm.recur_plan(mk(full, 128)) == bench_plan
    assert set(bench_plan) == set(sdm.RECUR_PLAN_FIELDS)
    assert sdm.recur_plan(mk(full, 1))["la"] == 1 and bench_plan["la"] > 1
    arr = (ctypes.c_int32 * 8)()
    assert sdm.lib().sdm_recur_plan(ctypes.byref(mk(full, 16)), arr, 7) == 1 and "[0, 6]" in sdm.last_error()


def test_wait_timeout_hook_rejects_shapes_without_interleaved_warps(sdm):
    L = sdm.lib()
    args = [FAKE, FAKE + 0x100000, FAKE + 0x200000, FAKE + 0x300000, FAKE + 0x400000, FAKE + 0x500000,
            FAKE + 0x600000, FAKE + 0x10000000, FAKE + 0x700000, FAKE + 0x40000000, 1 << 30]
    one = _shape(sdm, B=8, H=16, T=1, d_k=128, d_v=128, N=262144, k_write=32, k_read=32)
    assert sdm.recur_plan(one)["w"] == 0
    assert L.sdm_test_recur_wait_timeout(ctypes.byref(one), *args, 1000, None) == 2
    assert "token-interleaved" in sdm.last_error()
    many = _shape(sdm, B=1, H=2, T=8, d_v=64, N=4096, k_write=8, k_read=8)
    assert sdm.recur_plan(many)["w"] >= 2
    assert L.sdm_test_recur_wait_timeout(ctypes.byref(many), *args, 0, None) == 1 and "wait_cycles" in sdm.last_error()


def test_noalloc_size_check_cannot_wrap(sdm):
    """A shape whose entry count B*H*T*k overflows 64 bits is still rejected as too large."""
    huge = sdm.SdmShape.make(2 ** 31 - 1, 2 ** 31 - 1, 2 ** 31 - 1, 8, 64, 4096, 64, 64, "bf16")
    st = sdm.lib().sdm_recur_noalloc(ctypes.byref(huge), *[FAKE + i * 0x10000000 for i in range(9)], None)
    assert st == 2 and "fixed scratch" in sdm.last_error()
    neg = sdm.SdmShape.make(-1, 1, 1, 8, 64, 4096, 8, 8, "bf16")
    assert sdm.lib().sdm_recur_noalloc(ctypes.byref(neg), *[FAKE] * 9, None) == 1


def test_score_hook_rejects_shapes_off_the_tensor_core_path(sdm):
    s = _shape(sdm, dtype="f32")
    st = sdm.lib().sdm_test_scores(ctypes.byref(s), FAKE, FAKE + 0x100000, FAKE + 0x200000, FAKE + 0x300000,
                                   FAKE + 0x400000, FAKE + 0x40000000, 1 << 30, None)
    assert st == 2 and "tensor-core" in sdm.last_error()
