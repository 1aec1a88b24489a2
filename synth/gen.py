"""Seeded, slice-addressable synthetic inputs.

Every tensor is drawn in float64 from a PCG64 stream keyed by
``SeedSequence([seed, tensor_id, *coords])`` and rounded (round-to-nearest-even)
to the storage dtype, so any (b, h) slice or head can be regenerated alone:

* per head h:        M0 [N, d_v], P_q / P_k [2 sqrt(N), d_k]
* per slice (b, h):  q, k [T_seq, d_k], v [T_seq, d_v], alpha, beta [T_seq]
* layer side (the gate preparation and output epilogue around the path), with
  d_model = H * d_v:  x [B, T, d_model]; W_a, W_b [H, d_model]; b_dt, A [H]; g
  [B, H, T, d_v]; gamma [d_v]

For the decode workload T_seq = prefill + timed steps and step s uses token s
of every slice.  Storage format: ``np.float32`` for "f32"; ``np.uint16``
holding the bfloat16 bit pattern for "bf16".
"""
from __future__ import annotations

import enum

import numpy as np

from .configs import SdmConfig


class TensorId(enum.IntEnum):
    M0 = 1
    P_Q = 2
    P_K = 3
    Q = 4
    K = 5
    V = 6
    ALPHA = 7
    BETA = 8
    X = 9
    W_A = 10
    W_B = 11
    B_DT = 12
    A_LOG = 13
    G = 14
    GAMMA = 15


def _rng(seed: int, tid: TensorId, *coords: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(np.random.SeedSequence([int(seed), int(tid), *map(int, coords)])))


def storage_np_dtype(dtype: str):
    return np.float32 if dtype == "f32" else np.uint16


def round_f64_to_storage(x: np.ndarray, dtype: str) -> np.ndarray:
    """float64 -> storage dtype, round-to-nearest-even, in one rounding step."""
    x = np.asarray(x, dtype=np.float64)
    if dtype == "f32":
        return x.astype(np.float32)
    if dtype != "bf16":
        raise ValueError(dtype)
    _, e = np.frexp(x)
    quantum = np.ldexp(1.0, np.maximum(e - 8, -133))   # 8 significant bits; bf16 subnormal step 2^-133
    r = np.rint(x / quantum) * quantum                  # exact scaling, ties-to-even
    return (r.astype(np.float32).view(np.uint32) >> 16).astype(np.uint16)


def storage_to_f64(a: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "f32":
        return np.asarray(a, dtype=np.float32).astype(np.float64)
    return (np.asarray(a, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _unit_rows(x: np.ndarray) -> np.ndarray:
    return x / np.sqrt(np.sum(x * x, axis=-1, keepdims=True))


def _sigmoid(z: np.ndarray) -> np.ndarray:
    return 1.0 / (1.0 + np.exp(-z))


def head_inputs(cfg: SdmConfig, h: int, which=("M0", "P_q", "P_k")) -> dict:
    """Per-head parameters: initial memory M0[h] and the PKM projections P_q[h], P_k[h]."""
    out = {}
    if "M0" in which:
        m = _rng(cfg.seed, TensorId.M0, h).standard_normal((cfg.N, cfg.d_v)) * cfg.mem_std
        out["M0"] = round_f64_to_storage(m, cfg.dtype)
    if cfg.addr == "projected":
        if "P_q" in which:
            out["P_q"] = round_f64_to_storage(_rng(cfg.seed, TensorId.P_Q, h).standard_normal((2 * cfg.S, cfg.d_k)), cfg.dtype)
        if "P_k" in which:
            out["P_k"] = round_f64_to_storage(_rng(cfg.seed, TensorId.P_K, h).standard_normal((2 * cfg.S, cfg.d_k)), cfg.dtype)
    return out


def slice_inputs(cfg: SdmConfig, b: int, h: int) -> dict:
    """Per-sequence inputs of slice (b, h) for all of its tokens."""
    T = cfg.tokens_per_seq
    q = _unit_rows(_rng(cfg.seed, TensorId.Q, b, h).standard_normal((T, cfg.d_k)))
    k = _unit_rows(_rng(cfg.seed, TensorId.K, b, h).standard_normal((T, cfg.d_k)))
    v = _rng(cfg.seed, TensorId.V, b, h).standard_normal((T, cfg.d_v))
    alpha = _sigmoid(_rng(cfg.seed, TensorId.ALPHA, b, h).standard_normal(T) + cfg.alpha_mu)
    beta = _sigmoid(_rng(cfg.seed, TensorId.BETA, b, h).standard_normal(T))
    r = lambda x: round_f64_to_storage(x, cfg.dtype)
    return {"q": r(q), "k": r(k), "v": r(v), "alpha": r(alpha), "beta": r(beta)}


def full_inputs(cfg: SdmConfig, b0: int = 0) -> dict:
    """Whole-workload inputs as storage arrays: M0 [H,N,dv], P_* [H,2S,dk], q/k [B,H,T,dk],
    v [B,H,T,dv], alpha/beta [B,H,T] (T = tokens per sequence).  Sequence b of the result
    is global sequence b0 + b (a rank's shard of a larger batch)."""
    T = cfg.tokens_per_seq
    nd = storage_np_dtype(cfg.dtype)
    out = {"M0": np.empty((cfg.H, cfg.N, cfg.d_v), nd)}
    if cfg.addr == "projected":
        out["P_q"] = np.empty((cfg.H, 2 * cfg.S, cfg.d_k), nd)
        out["P_k"] = np.empty((cfg.H, 2 * cfg.S, cfg.d_k), nd)
    for h in range(cfg.H):
        for name, arr in head_inputs(cfg, h).items():
            out[name][h] = arr
    shapes = {"q": (cfg.d_k,), "k": (cfg.d_k,), "v": (cfg.d_v,), "alpha": (), "beta": ()}
    for name, tail in shapes.items():
        out[name] = np.empty((cfg.B, cfg.H, T) + tail, nd)
    for b in range(cfg.B):
        for h in range(cfg.H):
            for name, arr in slice_inputs(cfg, b0 + b, h).items():
                out[name][b, h] = arr
    return out


def decode_step_inputs(full: dict, s: int) -> dict:
    """Inputs of decode step s for every (b, h) (token s of each sequence), from ``full_inputs``."""
    return {name: np.ascontiguousarray(full[name][:, :, s]) for name in ("q", "k", "v", "alpha", "beta")}


def layer_inputs(cfg: SdmConfig) -> dict:
    """Inputs of the steps around the path for the whole workload, with d_model = H * d_v:

    * x [B, T, d_model] ~ N(0, 1), the layer input;
    * W_a, W_b [H, d_model] ~ N(0, 1 / d_model), the gate projections;
    * A [H] ~ U(0, 16) and b_dt [H] = inv_softplus(U(0.001, 0.1)), the initialisation the
      paper states (Sec. 4, "SDM Configuration");
    * g [B, H, T, d_v] = sigmoid(N(0, 1)), the output gate;
    * gamma [d_v] ~ 1 + 0.1 N(0, 1), the RMSNorm scale.

    x, W_a, W_b and g are rounded to the storage dtype; A, b_dt and gamma stay float32.
    """
    d = cfg.H * cfg.d_v
    T = cfg.tokens_per_seq
    r = lambda a: round_f64_to_storage(a, cfg.dtype)
    x = _rng(cfg.seed, TensorId.X).standard_normal((cfg.B, T, d))
    wa = _rng(cfg.seed, TensorId.W_A).standard_normal((cfg.H, d)) / np.sqrt(d)
    wb = _rng(cfg.seed, TensorId.W_B).standard_normal((cfg.H, d)) / np.sqrt(d)
    A = _rng(cfg.seed, TensorId.A_LOG).uniform(0.0, 16.0, cfg.H)
    u = _rng(cfg.seed, TensorId.B_DT).uniform(0.001, 0.1, cfg.H)
    b_dt = np.log(np.expm1(u))                      # inv_softplus(u)
    g = _sigmoid(_rng(cfg.seed, TensorId.G).standard_normal((cfg.B, cfg.H, T, cfg.d_v)))
    gamma = 1.0 + 0.1 * _rng(cfg.seed, TensorId.GAMMA).standard_normal(cfg.d_v)
    return {"x": r(x), "W_a": r(wa), "W_b": r(wb), "A": A.astype(np.float32), "b_dt": b_dt.astype(np.float32),
            "g": r(g), "gamma": gamma.astype(np.float32)}
