"""The five synthetic SDM workloads (shapes, dtypes, distributions, seeds).

Each workload is one global SDM layer's recurrence at the paper's scale:
per-head memory of N slots x d_v (Sec. 3.1), k slots read and written per
token (Sec. 4 uses W = R = 64; these workloads use k = 8..32), PKM addressing
with sqrt(N) x sqrt(N) product keys (Sec. 2, Product Key Memory).

Distributions (drawn in float64, then rounded to the storage dtype):
  q, k  ~ N(0, 1) per element, then each token row L2-normalised
  v     ~ N(0, 1)
  alpha = sigmoid(N(alpha_mu, 1)),  beta = sigmoid(N(0, 1))
  M0    ~ N(0, mem_std^2), one initial memory per head shared by all sequences
  P_q, P_k ~ N(0, 1), per head [2*sqrt(N), d_k] (PROJECTED addressing)
"""
from __future__ import annotations

import math
from dataclasses import dataclass, replace


@dataclass(frozen=True)
class SdmConfig:
    name: str
    B: int
    H: int
    T: int
    d_k: int
    d_v: int
    N: int
    k_write: int
    k_read: int
    dtype: str          # "f32" or "bf16": storage / I/O dtype of every tensor
    seed: int
    alpha_mu: float     # alpha = sigmoid(N(alpha_mu, 1))
    mem_std: float = 0.02
    addr: str = "projected"   # "projected" (s = P x) or "direct" (s = x, needs d_k == 2 sqrt(N))
    prefill_steps: int = 0    # decode workload: untimed decode steps before the timed ones
    decode_steps: int = 0     # decode workload: timed decode steps (0 = prefill/scan workload)

    @property
    def S(self) -> int:
        s = math.isqrt(self.N)
        assert s * s == self.N, "N must be a perfect square"
        return s

    @property
    def is_decode(self) -> bool:
        return self.decode_steps > 0

    @property
    def tokens_per_seq(self) -> int:
        """Tokens each sequence sees in total (decode: prefill + timed steps)."""
        return self.prefill_steps + self.decode_steps if self.is_decode else self.T

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def with_(self, **kw) -> "SdmConfig":
        return replace(self, **kw)

    def algorithmic_bytes_per_token_head(self) -> int:
        """Bytes the method itself must move per (b, h, t): write-gather, scatter and
        read-gather of k rows, the q and k vectors, v, alpha and beta, and y."""
        s = self.elem_bytes
        return (2 * self.k_write + self.k_read) * self.d_v * s + 2 * self.d_k * s + 2 * self.d_v * s + 2 * s

    def recurrence_bytes_per_token_head(self) -> int:
        """Algorithmic bytes of the fused recurrence alone: rows gathered/scattered, v, alpha, beta, y,
        and the slot lists it is given (int32 index + fp32 weight per write and per read slot)."""
        s = self.elem_bytes
        return ((2 * self.k_write + self.k_read) * self.d_v * s + 2 * self.d_v * s + 2 * s
                + (self.k_write + self.k_read) * 8)


TINY_FP32 = SdmConfig("tiny_fp32", B=1, H=1, T=256, d_k=64, d_v=64, N=4096, k_write=8, k_read=8,
                      dtype="f32", seed=0, alpha_mu=3.0)
SMALL_BF16 = SdmConfig("small_bf16", B=4, H=8, T=2048, d_k=128, d_v=128, N=65536, k_write=16, k_read=16,
                       dtype="bf16", seed=1, alpha_mu=3.0)
LAYER_1P4B = SdmConfig("layer_1p4b", B=8, H=16, T=4096, d_k=128, d_v=128, N=262144, k_write=32, k_read=32,
                       dtype="bf16", seed=2, alpha_mu=4.0)
LONG_CTX = SdmConfig("long_ctx", B=2, H=16, T=65536, d_k=128, d_v=128, N=1 << 20, k_write=32, k_read=32,
                     dtype="bf16", seed=3, alpha_mu=4.0)
DECODE = SdmConfig("decode", B=256, H=16, T=1, d_k=128, d_v=128, N=262144, k_write=32, k_read=32,
                   dtype="bf16", seed=4, alpha_mu=4.0, prefill_steps=1024, decode_steps=1000)

CONFIGS = {c.name: c for c in (TINY_FP32, SMALL_BF16, LAYER_1P4B, LONG_CTX, DECODE)}


def get_config(name: str) -> SdmConfig:
    return CONFIGS[name]
