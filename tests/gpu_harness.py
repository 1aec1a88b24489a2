"""GPU-side helpers for the parity tests: build device inputs from the seeded
generator, run the library through its C ABI, fetch results."""
from __future__ import annotations

import numpy as np

import synth
from synth.torch_io import from_torch, to_torch, torch_dtype


def shape_of(cfg: synth.SdmConfig, T: int | None = None):
    import paper_2607_07386_gb300 as sdm
    return sdm.SdmShape.make(cfg.B, cfg.H, cfg.T if T is None else T, cfg.d_k, cfg.d_v, cfg.N, cfg.k_write,
                             cfg.k_read, cfg.dtype, cfg.addr)


def device_inputs(cfg: synth.SdmConfig, full: dict | None = None) -> dict:
    full = full if full is not None else synth.full_inputs(cfg)
    return {name: to_torch(a, cfg.dtype) for name, a in full.items()}


def alloc_outputs(cfg: synth.SdmConfig, T: int):
    import torch
    dt = torch_dtype(cfg.dtype)
    o = {
        "y": torch.empty((cfg.B, cfg.H, T, cfg.d_v), dtype=dt, device="cuda"),
        "idx_w": torch.empty((cfg.B, cfg.H, T, cfg.k_write), dtype=torch.int32, device="cuda"),
        "w_w": torch.empty((cfg.B, cfg.H, T, cfg.k_write), dtype=torch.float32, device="cuda"),
        "idx_r": torch.empty((cfg.B, cfg.H, T, cfg.k_read), dtype=torch.int32, device="cuda"),
        "w_r": torch.empty((cfg.B, cfg.H, T, cfg.k_read), dtype=torch.float32, device="cuda"),
    }
    return o


def workspace(shape):
    import torch
    import paper_2607_07386_gb300 as sdm
    return torch.empty(sdm.workspace_bytes(shape), dtype=torch.uint8, device="cuda")


def run_forward(cfg: synth.SdmConfig, dev: dict, T0: int = 0, T1: int | None = None, mem=None, ws=None):
    """sdm_forward over tokens [T0, T1) (memory initialised from M0 unless `mem` is given)."""
    import torch
    import paper_2607_07386_gb300 as sdm
    T1 = cfg.tokens_per_seq if T1 is None else T1
    T = T1 - T0
    shape = shape_of(cfg, T)
    if mem is None:
        mem = torch.empty((cfg.B, cfg.H, cfg.N, cfg.d_v), dtype=torch_dtype(cfg.dtype), device="cuda")
        sdm.init_memory(shape, dev["M0"], mem)
    sl = lambda name: dev[name][:, :, T0:T1].contiguous()
    out = alloc_outputs(cfg, T)
    ws = ws if ws is not None else workspace(shape)
    sdm.forward(shape, dev.get("P_q"), dev.get("P_k"), sl("q"), sl("k"), sl("v"), sl("alpha"), sl("beta"), mem,
                out["y"], ws, idx_w=out["idx_w"], w_w=out["w_w"], idx_r=out["idx_r"], w_r=out["w_r"])
    out["mem"] = mem
    return out


def run_forward_lazy(cfg: synth.SdmConfig, dev: dict, T0: int = 0, T1: int | None = None, mem=None, touched=None):
    """sdm_forward_lazy over tokens [T0, T1); a fresh sequence (all touched bits clear, mem
    filled with a value no slot holds) unless `mem` and `touched` continue one."""
    import torch
    import paper_2607_07386_gb300 as sdm
    T1 = cfg.tokens_per_seq if T1 is None else T1
    T = T1 - T0
    shape = shape_of(cfg, T)
    if mem is None:
        mem = torch.full((cfg.B, cfg.H, cfg.N, cfg.d_v), 7.0, dtype=torch_dtype(cfg.dtype), device="cuda")
        touched = torch.zeros((cfg.B, cfg.H, sdm.touched_words(shape)), dtype=torch.int32, device="cuda")
    sl = lambda name: dev[name][:, :, T0:T1].contiguous()
    out = alloc_outputs(cfg, T)
    ws = torch.empty(sdm.lazy_workspace_bytes(shape), dtype=torch.uint8, device="cuda")
    sdm.forward_lazy(shape, dev["M0"], touched, dev.get("P_q"), dev.get("P_k"), sl("q"), sl("k"), sl("v"),
                     sl("alpha"), sl("beta"), mem, out["y"], ws, idx_w=out["idx_w"], w_w=out["w_w"],
                     idx_r=out["idx_r"], w_r=out["w_r"])
    out["mem"] = mem
    out["touched"] = touched
    return out


def touched_bits(touched, N: int) -> np.ndarray:
    """[B, H, ceil(N/32)] int32 bitmaps -> bool [B, H, N] (bit s % 32 of word s // 32)."""
    w = touched.cpu().numpy().astype(np.int64) & 0xFFFFFFFF
    bits = (w[..., :, None] >> np.arange(32)) & 1
    return bits.reshape(w.shape[0], w.shape[1], -1)[..., :N].astype(bool)


def host(t, dtype: str) -> np.ndarray:
    return from_torch(t, dtype)


# ------------------------------------------------------------------ elementwise comparison

def storage_ulp(x: np.ndarray, dtype: str) -> np.ndarray:
    """Unit in the last place of the storage dtype at |x| (bf16: 8 significant bits, fp32: 24)."""
    mant = 7 if dtype == "bf16" else 23
    ax = np.abs(np.asarray(x, np.float64))
    e = np.floor(np.log2(np.where(ax > 0, ax, 1.0)))
    return np.where(ax > 0, 2.0 ** (e - mant), 2.0 ** (-126 - mant))


def elementwise(got: np.ndarray, ref: np.ndarray, dtype: str) -> dict:
    """Per-element distance of stored values `got` from the oracle's stored values `ref` (both
    float64 of storage numbers), rows along the last axis:
      max_row_ulps  max |got - ref| in units of the ulp of the row's largest |ref|;
      frac_gt1      fraction of elements more than one ulp of their own value apart (the
                    ulp taken at max(|ref|, 2^-8 * row max), so that near-zero elements of a
                    row are measured at the row's own resolution);
      max_rel_row   max |got - ref| / row max of |ref|."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    rowmax = np.max(np.abs(ref), axis=-1, keepdims=True)
    d = np.abs(got - ref)
    u_row = storage_ulp(rowmax, dtype)
    u_own = storage_ulp(np.maximum(np.abs(ref), rowmax * 2.0 ** -8), dtype)
    return {"max_row_ulps": float(np.max(d / u_row)) if d.size else 0.0,
            "frac_gt1": float(np.mean(d > u_own)) if d.size else 0.0,
            "max_rel_row": float(np.max(d / np.where(rowmax > 0, rowmax, 1.0))) if d.size else 0.0}
