"""Storage arrays (numpy) <-> torch tensors; plumbing for tests and the benchmark."""
from __future__ import annotations

import numpy as np


def to_torch(a: np.ndarray, dtype: str, device="cuda"):
    import torch
    a = np.ascontiguousarray(a)
    if dtype == "bf16":
        t = torch.from_numpy(a.view(np.int16)).view(torch.bfloat16)
    elif dtype == "f32":
        t = torch.from_numpy(a.astype(np.float32, copy=False))
    else:
        t = torch.from_numpy(a)
    return t.to(device) if device is not None else t


def from_torch(t, dtype: str) -> np.ndarray:
    import torch
    t = t.detach().cpu().contiguous()
    if dtype == "bf16":
        assert t.dtype == torch.bfloat16
        return t.view(torch.int16).numpy().view(np.uint16)
    return t.numpy()


def torch_dtype(dtype: str):
    import torch
    return {"bf16": torch.bfloat16, "f32": torch.float32}[dtype]
