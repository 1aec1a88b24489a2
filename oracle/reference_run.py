"""Run the float64 oracle on seeded synthetic slices (test infrastructure only).

Inputs come from ``synth`` (the shared generator); everything else here is the
oracle of ``sdm_oracle``.  Slices (b, h) are independent, so several can run in
a ``spawn`` process pool.
"""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np

import synth
from . import sdm_oracle as O


def slice_f64(cfg: synth.SdmConfig, b: int, h: int, head: dict | None = None) -> dict:
    """float64 views of slice (b, h)'s inputs and head h's parameters."""
    head = head if head is not None else synth.head_inputs(cfg, h)
    sl = synth.slice_inputs(cfg, b, h)
    f = lambda a: O.to_f64(a, cfg.dtype)
    out = {name: f(a) for name, a in sl.items()}
    out["M0"] = f(head["M0"])
    out["P_q"] = f(head["P_q"]) if "P_q" in head else None
    out["P_k"] = f(head["P_k"]) if "P_k" in head else None
    return out


def oracle_slice(cfg: synth.SdmConfig, b: int, h: int, T: int | None = None, head: dict | None = None) -> dict:
    """Oracle forward of slice (b, h) over its first T tokens (all by default), from M0."""
    x = slice_f64(cfg, b, h, head)
    T = x["v"].shape[0] if T is None else T
    cut = lambda a: a[:T]
    return O.forward_slice(x["M0"], x["P_q"], x["P_k"], cut(x["q"]), cut(x["k"]), cut(x["v"]), cut(x["alpha"]),
                           cut(x["beta"]), cfg.N, cfg.k_write, cfg.k_read, cfg.dtype)


def _worker(args):
    cfg, b, h, T = args
    r = oracle_slice(cfg, b, h, T)
    touched = np.unique(r["idx_w"])
    return (b, h, {"y": r["y"], "idx_w": r["idx_w"], "idx_r": r["idx_r"], "w_w": r["w_w"], "w_r": r["w_r"],
                   "touched": touched, "M_touched": r["M"][touched]})


def oracle_slices(cfg: synth.SdmConfig, slices, T: int | None = None, workers: int | None = None):
    """Oracle results for several (b, h) slices; returns {(b, h): result} (final memory kept
    only for the rows the slice wrote)."""
    jobs = [(cfg, b, h, T) for b, h in slices]
    workers = workers or min(len(jobs), os.cpu_count() or 1)
    if workers <= 1 or len(jobs) == 1:
        res = [_worker(j) for j in jobs]
    else:
        with mp.get_context("spawn").Pool(workers) as pool:
            res = pool.map(_worker, jobs)
    return {(b, h): r for b, h, r in res}


def rel_fro(got: np.ndarray, ref: np.ndarray) -> float:
    """||got - ref||_F / ||ref||_F (0 when both are zero)."""
    got = np.asarray(got, np.float64)
    ref = np.asarray(ref, np.float64)
    den = np.linalg.norm(ref)
    num = np.linalg.norm(got - ref)
    return float(num / den) if den > 0 else float(num)


def timed_worker(args) -> float:
    """Oracle forward of one slice over its first T tokens; returns the compute seconds
    (input generation and float64 conversion excluded)."""
    import time
    cfg, b, h, T = args
    x = slice_f64(cfg, b, h)
    cut = lambda a: a[:T]
    t0 = time.perf_counter()
    O.forward_slice(x["M0"], x["P_q"], x["P_k"], cut(x["q"]), cut(x["k"]), cut(x["v"]), cut(x["alpha"]),
                    cut(x["beta"]), cfg.N, cfg.k_write, cfg.k_read, cfg.dtype)
    return time.perf_counter() - t0
