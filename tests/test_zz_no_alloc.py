"""sdm_recur_noalloc (fixed device scratch, no workspace) against sdm_recur.

Some callers cannot allocate device memory for the library (a runtime whose own pool
owns the device, a serving loop that must not call an allocator); this entry point
takes its scratch from an array the library reserves statically.  It runs the same
kernels as sdm_recur, so the results must be identical bit for bit.

Collected last on purpose: it must give the same results whether it runs alone in a
fresh process (first use of its scratch) or after every other test."""
import ctypes

import pytest

import synth
from oracle import sdm_oracle as O
from oracle.reference_run import rel_fro

TOL = {"bf16": 2e-3, "f32": 1e-5}


@pytest.fixture(scope="module")
def sdm():
    import paper_2607_07386_gb300 as sdm
    from paper_2607_07386_gb300 import build as B
    B.build()
    return sdm


def test_rejects_shapes_beyond_the_fixed_scratch(sdm):
    """Needs B*H*T*max(k_write,k_read)*4 bytes <= the fixed scratch; larger shapes are
    rejected before any CUDA call (the fake addresses are never dereferenced)."""
    cap = sdm.RECUR_NOALLOC_SCRATCH_BYTES // 4
    k = 32
    T = cap // k + 1                   # one token more than fits
    shape = sdm.SdmShape.make(1, 1, T, 8, 64, 4096, k, k, "bf16")
    fake = 0x7F0000000000
    st = sdm.lib().sdm_recur_noalloc(ctypes.byref(shape), *[fake + i * 0x10000000 for i in range(9)], None)
    assert st == 2 and "fixed scratch" in sdm.last_error()
    assert sdm.lib().sdm_recur_noalloc(None, *([None] * 9), None) == 1


@pytest.mark.gpu
@pytest.mark.parametrize("name", ["tiny_fp32", "small_bf16"])
def test_noalloc_matches_workspace_entry_on_two_calls(sdm, name):
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from tests import gpu_harness as G
    from synth.torch_io import torch_dtype
    cfg = synth.CONFIGS[name]
    B, H, T, N, dv = cfg.B, cfg.H, cfg.T, cfg.N, cfg.d_v
    dt = torch_dtype(cfg.dtype)
    dev = G.device_inputs(cfg)
    full_shape = G.shape_of(cfg)
    idx_w = torch.empty((B, H, T, cfg.k_write), dtype=torch.int32, device="cuda")
    w_w = torch.empty((B, H, T, cfg.k_write), dtype=torch.float32, device="cuda")
    idx_r = torch.empty((B, H, T, cfg.k_read), dtype=torch.int32, device="cuda")
    w_r = torch.empty((B, H, T, cfg.k_read), dtype=torch.float32, device="cuda")
    sdm.address(full_shape, dev.get("P_q"), dev.get("P_k"), dev["q"], dev["k"], idx_w, w_w, idx_r, w_r,
                G.workspace(full_shape))
    mems = []
    for _ in range(2):
        m = torch.empty((B, H, N, dv), dtype=dt, device="cuda")
        sdm.init_memory(full_shape, dev["M0"], m)
        mems.append(m)
    mem_ws, mem_na = mems
    cut = T // 2 + 3                   # two calls in a row: tokens [0, cut) then [cut, T)
    for t0, t1 in ((0, cut), (cut, T)):
        shape = G.shape_of(cfg, t1 - t0)
        sl = lambda x: x[:, :, t0:t1].contiguous()
        args = [sl(idx_w), sl(w_w), sl(idx_r), sl(w_r), sl(dev["v"]), sl(dev["alpha"]), sl(dev["beta"])]
        y_ws = torch.empty((B, H, t1 - t0, dv), dtype=dt, device="cuda")
        y_na = torch.empty_like(y_ws)
        ws = torch.empty(sdm.recur_workspace_bytes(shape), dtype=torch.uint8, device="cuda")
        sdm.recur(shape, *args, mem_ws, y_ws, ws)
        sdm.recur_noalloc(shape, *args, mem_na, y_na)
        torch.cuda.synchronize()
        assert sdm.device_status() == 0
        # same kernels on the same inputs: only the scratch differs, so the results must be
        # identical bit for bit (a tolerance could hide a scratch-aliasing fault)
        assert torch.equal(y_na, y_ws), t0
        ya, yb = (O.to_f64(G.host(x, cfg.dtype), cfg.dtype) for x in (y_ws, y_na))
        for b in range(B):
            for h in range(H):
                assert rel_fro(yb[b, h], ya[b, h]) <= TOL[cfg.dtype], (t0, b, h)
    assert torch.equal(mem_na, mem_ws)
