"""Seeded synthetic inputs for the Sparse Delta Memory hot path.

This package is shared by the float64 oracle (``oracle/``) and the CUDA path
(``paper_2607_07386_gb300``).  It draws random numbers and rounds them to the
storage dtype; it holds none of the method's arithmetic.
"""
from .configs import SdmConfig, CONFIGS, TINY_FP32, SMALL_BF16, LAYER_1P4B, LONG_CTX, DECODE, get_config
from .gen import (TensorId, slice_inputs, head_inputs, full_inputs, decode_step_inputs, storage_to_f64,
                  round_f64_to_storage, storage_np_dtype)

__all__ = [
    "SdmConfig", "CONFIGS", "TINY_FP32", "SMALL_BF16", "LAYER_1P4B", "LONG_CTX", "DECODE",
    "get_config", "TensorId", "slice_inputs", "head_inputs", "full_inputs", "decode_step_inputs",
    "storage_to_f64", "round_f64_to_storage", "storage_np_dtype",
]
