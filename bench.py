"""Benchmark of the Sparse Delta Memory hot path on GB300.

One step = one pass of the whole hot path over the 1.4B-scale global-layer
workload (B=8, H=16, T=4096, d_k=d_v=128, N=262144 slots/head, k=32, bf16):
learned-initial-state broadcast (sdm_init_memory), then sdm_forward (PKM
addressing for the write keys and read queries of every token, then the fused
recurrence), all inputs resident in HBM.  Prints one JSON line.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

--impl reference times the float64 CPU oracle on this machine's cores on a
bounded sample of the same workload (the comparison arm; no GPU use).
Multi-GPU (torchrun): every rank runs an independent shard of sequences (weak
scaling); only the timing uses a collective.
"""
from __future__ import annotations

import argparse
import datetime
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402

import synth  # noqa: E402

METRIC = "SDM recurrence tokens/s per layer (1 GB300) and achieved HBM GB/s vs ~8 TB/s"
UNIT = "tokens/s"


# DRAM bytes per token-head moved by the recurrence phase (hazard pass + recurrence), from an
# ncu capture of dram__bytes_read.sum + dram__bytes_write.sum of the hazard pass and the
# recurrence on the layer_1p4b workload itself (one launch, one pass per kernel):
# (134.40 MB + 39.86 MB) + (10.37 GB + 4.35 GB) over 524,288 token-heads.
RECUR_DRAM_BYTES_PER_TOKEN_HEAD = (134.40e6 + 39.86e6 + 10.37e9 + 4.35e9) / 524288


def _peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "bf16_tflops": float(p.get("bf16_tflops", 1931.2)),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "source": "fallback"}


def _workload_desc(cfg) -> str:
    return (f"{cfg.name}: B={cfg.B} H={cfg.H} T={cfg.T} d_k={cfg.d_k} d_v={cfg.d_v} N={cfg.N} "
            f"k_write={cfg.k_write} k_read={cfg.k_read} {cfg.dtype} seed={cfg.seed}")


# ----------------------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region.

    The sampler is started before the region and waited for until it writes, so that its
    start-up does not fall into the region; samples are kept by their timestamps."""

    Q = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str):
        self.idx = gpu_id
        self.proc = None
        self.path = None
        self.t0 = self.t1 = None

    def __enter__(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={self.idx}", f"--query-gpu={self.Q}",
                                          "--format=csv,noheader,nounits", "-lms", "50", "-f", self.path],
                                         stdout=subprocess.DEVNULL, stderr=subprocess.DEVNULL)
            deadline = time.time() + 5.0
            while time.time() < deadline and os.path.getsize(self.path) == 0:
                time.sleep(0.02)
        except Exception:
            self.proc = None
        return self

    def mark_start(self):
        self.t0 = time.time()

    def mark_end(self):
        self.t1 = time.time()

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.06)                 # one more sample after the region
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if not self.path or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        rows = []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 10:
                    continue
                try:
                    ts = datetime.datetime.strptime(parts[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                    rows.append((ts, float(parts[2]), float(parts[3]),
                                 {n for n, v in zip(names, parts[6:10]) if v.lower().startswith("active")}))
                except ValueError:
                    continue
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        inside = [r for r in rows if self.t0 is not None and self.t0 <= r[0] <= self.t1]
        use = inside or sorted(rows, key=lambda r: abs(r[0] - (self.t0 or r[0])))[:1]
        sm = sorted(r[1] for r in use)
        reasons = set().union(*(r[3] for r in use))
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(r[2] for r in use),
                "reasons": sorted(reasons), "samples": len(use), "samples_in_region": len(inside)}


# ----------------------------------------------------------------------------- CPU oracle arm

def _oracle_pool(n):
    import multiprocessing as mp
    return mp.get_context("spawn").Pool(n)


def _oracle_step(pool, cfg, slices, T):
    """Slices run one per worker in parallel; the step time is the slowest worker's
    oracle compute time (input generation excluded)."""
    from oracle.reference_run import timed_worker
    return max(pool.map(timed_worker, [(cfg, b, h, T) for b, h in slices]))


# The oracle sample, the same unit of work for the cpu_baseline key and the reference arm: one
# (b, h) slice per host core over the slice's first ORACLE_T tokens.  Both legs time this unit
# (the oracle's per-slice set-up, a float64 copy of the head's M0, is amortised over the same
# number of tokens), so their tokens/s agree; the cpu_baseline key repeats it CPU_REPEATS
# times for a 10-30 s sample, the reference arm once per step.
ORACLE_T = 1024
CPU_REPEATS = 12


def _oracle_sample(cfg, pool, cores, steps, seed):
    rng = np.random.default_rng(seed)
    times = []
    for _ in range(steps):
        slices = [(int(rng.integers(cfg.B)), int(rng.integers(cfg.H))) for _ in range(cores)]
        times.append(_oracle_step(pool, cfg, slices, ORACLE_T))
    return cores * ORACLE_T / cfg.H * len(times) / sum(times), times


def cpu_baseline(cfg):
    """Oracle throughput on a bounded sample: CPU_REPEATS rounds of one (b, h) slice x ORACLE_T
    tokens per core; tokens/s per layer = slice-tokens / H / time (slices are independent, so
    per-core work adds up)."""
    cores = os.cpu_count() or 1
    with _oracle_pool(cores) as pool:
        value, times = _oracle_sample(cfg, pool, cores, CPU_REPEATS, 0)
    return {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{CPU_REPEATS} rounds of {cores} (b,h) slices x first {ORACLE_T} tokens of {cfg.name}, one "
                      f"float64 worker per core, {sum(times):.1f} s (slowest worker per round, input generation "
                      "excluded); the reference arm times the same unit"}


def run_reference(args, cfg):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cores = os.cpu_count() or 1
    T = ORACLE_T
    with _oracle_pool(cores) as pool:
        for _ in range(args.warmup):
            _oracle_step(pool, cfg, [(0, 0)], 32)
        value, times = _oracle_sample(cfg, pool, cores, args.steps, 1)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * sum(times) / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": _workload_desc(cfg), "global_batch": cfg.B,
                                            "seq_len": cfg.T, "parallelism": "none (host cores)"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle",
                             "sample": f"each step: {cores} (b,h) slices x first {T} tokens, float64 oracle, "
                                       "one worker per core, input generation excluded"},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------------- GPU arm

def tokens_step_of(B: int, T: int, world: int) -> int:
    return B * T * world


def shard_b0(rank: int, B: int) -> int:
    """First global sequence of a rank's shard: each rank owns B whole sequences (their (b, h)
    chains are independent), so per-rank work is fixed as ranks are added (weak scaling)."""
    return rank * B


def reduce_max(x: float, dist=None, device="cpu") -> float:
    """Max of x over all ranks (x itself on one rank): the job's time is its slowest rank's."""
    if dist is None or not dist.is_initialized() or dist.get_world_size() == 1:
        return x
    import torch
    t = torch.tensor([x], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_value(B: int, T: int, world: int, ms_max: float) -> float:
    """Whole-job tokens/s: every rank's B*T tokens over the slowest rank's step time."""
    return tokens_step_of(B, T, world) / (ms_max * 1e-3)


# ----------------------------------------------------------------------------- other workloads

def device_inputs(cfg, seed: int):
    """Inputs of a workload's shapes and value distributions (the generator recipe of synth),
    drawn on the device with torch's generator: the bench legs of the other workloads time
    the kernels on them; their parity with the oracle is covered by the tests on synth's
    inputs."""
    import torch
    from synth.torch_io import torch_dtype
    dt = torch_dtype(cfg.dtype)
    g = torch.Generator(device="cuda").manual_seed(seed)
    rn = lambda *sh: torch.randn(sh, generator=g, device="cuda", dtype=torch.float32)
    B, H, T, dk, dv, S = cfg.B, cfg.H, cfg.T, cfg.d_k, cfg.d_v, cfg.S
    unit = lambda x: x / x.norm(dim=-1, keepdim=True)
    out = {"q": unit(rn(B, H, T, dk)).to(dt), "k": unit(rn(B, H, T, dk)).to(dt), "v": rn(B, H, T, dv).to(dt),
           "alpha": torch.sigmoid(rn(B, H, T) + cfg.alpha_mu).to(dt), "beta": torch.sigmoid(rn(B, H, T)).to(dt),
           "P_q": rn(H, 2 * S, dk).to(dt), "P_k": rn(H, 2 * S, dk).to(dt)}
    M0 = torch.empty((H, cfg.N, dv), dtype=dt, device="cuda")
    for h in range(H):                      # in per-head pieces: bounded fp32 temporaries
        M0[h] = (rn(cfg.N, dv) * cfg.mem_std).to(dt)
    out["M0"] = M0
    return out


def leg_scan(name: str, steps: int, warmup: int) -> dict:
    """A scan workload's step (sdm_forward_m0: M0 broadcast beside the addressing, then the
    recurrence) and its phases, on device-drawn inputs; inputs larger than L2."""
    import torch
    import paper_2607_07386_gb300 as sdm
    from synth.torch_io import torch_dtype
    cfg = synth.get_config(name)
    dev = device_inputs(cfg, seed=cfg.seed)
    B, H, T, N, dv = cfg.B, cfg.H, cfg.T, cfg.N, cfg.d_v
    dt = torch_dtype(cfg.dtype)
    shape = sdm.SdmShape.make(B, H, T, cfg.d_k, dv, N, cfg.k_write, cfg.k_read, cfg.dtype)
    mem = torch.empty((B, H, N, dv), dtype=dt, device="cuda")
    y = torch.empty((B, H, T, dv), dtype=dt, device="cuda")
    ws = torch.empty(sdm.workspace_bytes(shape), dtype=torch.uint8, device="cuda")
    lists = {n: torch.empty((B, H, T, k), dtype=tt, device="cuda")
             for n, k, tt in (("idx_w", cfg.k_write, torch.int32), ("w_w", cfg.k_write, torch.float32),
                              ("idx_r", cfg.k_read, torch.int32), ("w_r", cfg.k_read, torch.float32))}
    st = torch.cuda.current_stream()

    def step():
        sdm.forward_m0(shape, dev["M0"], dev["P_q"], dev["P_k"], dev["q"], dev["k"], dev["v"], dev["alpha"],
                       dev["beta"], mem, y, ws, stream=st)

    def timed(fn, n):
        for _ in range(warmup):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        for _ in range(n):
            fn()
        e1.record(st)
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / n

    ms = timed(step, steps)
    ms_addr = timed(lambda: sdm.address(shape, dev["P_q"], dev["P_k"], dev["q"], dev["k"], lists["idx_w"], lists["w_w"],
                                        lists["idx_r"], lists["w_r"], ws, stream=st), steps)
    ms_rec = timed(lambda: sdm.recur(shape, lists["idx_w"], lists["w_w"], lists["idx_r"], lists["w_r"], dev["v"],
                                     dev["alpha"], dev["beta"], mem, y, ws, stream=st), steps)
    ms_init = timed(lambda: sdm.init_memory(shape, dev["M0"], mem, st), steps)
    if sdm.device_status(st) != 0:
        raise RuntimeError(f"device status word set in the {name} leg")
    peaks = _peaks()
    rec_bytes = cfg.recurrence_bytes_per_token_head() * B * H * T
    gbs = rec_bytes / (ms_rec * 1e-3) / 1e9
    return {"workload": _workload_desc(cfg), "data": "synthetic (device-drawn, the workload's distributions)",
            "tokens_per_s": B * T / (ms * 1e-3), "ms_per_step": ms,
            "step": "sdm_forward_m0 (M0 broadcast beside the addressing, then the recurrence)",
            "phase_ms": {"init_memory": ms_init, "address": ms_addr, "recurrence": ms_rec},
            "recurrence_gbs": gbs, "recurrence_frac_of_measured": gbs / peaks["hbm_gbs"],
            "recurrence_frac_of_8tbs": gbs / 8000.0, "recurrence_bytes": rec_bytes, "gpu_launches_per_step": 8}


def leg_decode(steps: int, warmup: int) -> dict:
    """The decode workload: B=256 sequences x H=16 heads, one token per call on the 275 GB
    state, per-sequence memories pre-filled by 1024 decode steps from M0, then `steps`
    consecutive steps replayed as one CUDA graph.  Each step has its own inputs (a pool of 64
    input sets cycled, so no step re-reads the previous steps' rows from L2)."""
    import torch
    import paper_2607_07386_gb300 as sdm
    cfg = synth.DECODE
    B, H, N, dv, dk = cfg.B, cfg.H, cfg.N, cfg.d_v, cfg.d_k
    pool = 64
    dev = device_inputs(cfg.with_(T=pool), seed=cfg.seed)
    shape = sdm.SdmShape.make(B, H, 1, dk, dv, N, cfg.k_write, cfg.k_read, cfg.dtype)
    mem = torch.empty((B, H, N, dv), dtype=torch.bfloat16, device="cuda")
    y = torch.empty((B, H, dv), dtype=torch.bfloat16, device="cuda")
    ws = torch.empty(sdm.workspace_bytes(shape), dtype=torch.uint8, device="cuda")
    per = [{n: dev[n][:, :, i].contiguous() for n in ("q", "k", "v", "alpha", "beta")} for i in range(pool)]
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        sdm.init_memory(shape, dev["M0"], mem, st)

        def one(i):
            x = per[i % pool]
            sdm.decode_step(shape, dev["P_q"], dev["P_k"], x["q"], x["k"], x["v"], x["alpha"], x["beta"], mem, y, ws,
                            stream=st)

        for i in range(cfg.prefill_steps):
            one(i)
        for i in range(warmup):
            one(i)
        st.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        for i in range(steps):
            one(i)
        e1.record(st)
        st.synchronize()
        direct_us = e0.elapsed_time(e1) / steps * 1e3
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=st):
            for i in range(steps):
                one(i)
        graph.replay()
        st.synchronize()
        e0.record(st)
        graph.replay()
        e1.record(st)
        st.synchronize()
        graph_us = e0.elapsed_time(e1) / steps * 1e3
    if sdm.device_status(st) != 0:
        raise RuntimeError("device status word set in the decode leg")
    per_step = cfg.algorithmic_bytes_per_token_head() * B * H
    peaks = _peaks()
    return {"workload": _workload_desc(cfg) + f" prefill={cfg.prefill_steps} timed={steps}",
            "data": "synthetic (device-drawn, the workload's distributions)",
            "us_per_step": graph_us, "us_per_step_direct_calls": direct_us,
            "tokens_per_s": B / (graph_us * 1e-6), "algorithmic_bytes_per_step": per_step,
            "gbs": per_step / (graph_us * 1e-6) / 1e9, "frac_of_measured": per_step / (graph_us * 1e-6) / 1e9 / peaks["hbm_gbs"],
            "timing": f"{steps} consecutive steps captured in one CUDA graph, one replay timed with CUDA events"}


def leg_next(steps: int, warmup: int) -> dict:
    """The rows beyond the token-serial forward, timed at the layer_1p4b geometry on the same
    device-drawn inputs: the chunkwise (WY) forward (App. A.1) at C = 16 and 32, the forward
    that also writes the undo log, and the backward that walks the tokens in reverse and
    restores the memory from that log (App. A.3).  Each call is bracketed by its own CUDA
    events; the zeroing of dM between backward calls is outside them."""
    import torch
    import paper_2607_07386_gb300 as sdm
    from synth.torch_io import torch_dtype
    cfg = synth.LAYER_1P4B
    dev = device_inputs(cfg, seed=cfg.seed)
    B, H, T, N, dv = cfg.B, cfg.H, cfg.T, cfg.N, cfg.d_v
    dt = torch_dtype(cfg.dtype)
    shape = sdm.SdmShape.make(B, H, T, cfg.d_k, dv, N, cfg.k_write, cfg.k_read, cfg.dtype)
    st = torch.cuda.current_stream()
    mem = torch.empty((B, H, N, dv), dtype=dt, device="cuda")
    y = torch.empty((B, H, T, dv), dtype=dt, device="cuda")
    ws = torch.empty(max(sdm.workspace_bytes(shape), sdm.recur_workspace_bytes(shape)), dtype=torch.uint8, device="cuda")
    lists = {n: torch.empty((B, H, T, k), dtype=tt, device="cuda")
             for n, k, tt in (("idx_w", cfg.k_write, torch.int32), ("w_w", cfg.k_write, torch.float32),
                              ("idx_r", cfg.k_read, torch.int32), ("w_r", cfg.k_read, torch.float32))}
    sdm.address(shape, dev["P_q"], dev["P_k"], dev["q"], dev["k"], lists["idx_w"], lists["w_w"], lists["idx_r"],
                lists["w_r"], ws, stream=st)
    sdm.init_memory(shape, dev["M0"], mem, st)
    L = (lists["idx_w"], lists["w_w"], lists["idx_r"], lists["w_r"], dev["v"], dev["alpha"], dev["beta"])

    def timed(fn, n, between=None):
        tot = 0.0
        for i in range(warmup + n):
            if between is not None:
                between()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(st)
            fn()
            e1.record(st)
            e1.synchronize()
            if i >= warmup:
                tot += e0.elapsed_time(e1)
        return tot / n

    out = {"workload": _workload_desc(cfg), "data": "synthetic (device-drawn, the workload's distributions)"}
    rec_bytes = cfg.recurrence_bytes_per_token_head() * B * H * T
    for C in (16, 32):
        ms = timed(lambda: sdm.recur_chunkwise(shape, *L, mem, y, C, stream=st), steps)
        out[f"chunkwise_c{C}"] = {"ms": ms, "tokens_per_s": B * T / (ms * 1e-3),
                                  "gbs_of_recurrence_bytes": rec_bytes / (ms * 1e-3) / 1e9}
    undo = torch.empty(sdm.undo_log_bytes(shape), dtype=torch.uint8, device="cuda")
    ms_u = timed(lambda: sdm.recur_undo(shape, *L, mem, y, undo, ws, stream=st), steps)
    dy = torch.randn((B, H, T, dv), device="cuda").to(dt)
    grads = {"dv": torch.empty((B, H, T, dv), device="cuda"), "dalpha": torch.empty((B, H, T), device="cuda"),
             "dbeta": torch.empty((B, H, T), device="cuda"), "dw_w": torch.empty((B, H, T, cfg.k_write), device="cuda"),
             "dw_r": torch.empty((B, H, T, cfg.k_read), device="cuda")}
    dM = torch.empty((B, H, N, dv), device="cuda")
    # each backward restores mem to the state before the forward: one undo forward before each
    def fwd_then_zero():
        sdm.recur_undo(shape, *L, mem, y, undo, ws, stream=st)
        dM.zero_()
    ms_b = timed(lambda: sdm.recur_backward(shape, *L, mem, undo, dy, grads["dv"], grads["dalpha"], grads["dbeta"],
                                            grads["dw_w"], grads["dw_r"], dM, stream=st), steps, between=fwd_then_zero)
    undo_bytes = undo.numel()
    out["forward_with_undo_log"] = {"ms": ms_u, "tokens_per_s": B * T / (ms_u * 1e-3), "undo_log_bytes": undo_bytes}
    out["backward"] = {"ms": ms_b, "tokens_per_s": B * T / (ms_b * 1e-3)}
    rows = B * H * T * cfg.k_write
    scales = torch.empty(rows, dtype=torch.float32, device="cuda")
    for kind in ("fp8", "int4"):
        codes = torch.empty(sdm.undo_code_bytes(shape, kind), dtype=torch.uint8, device="cuda")
        sdm.recur_undo(shape, *L, mem, y, undo, ws, stream=st)
        ms_q = timed(lambda: sdm.undo_quantize(shape, undo, kind, codes, scales, stream=st), steps)
        q_bytes = undo_bytes + codes.numel() + rows * 4
        sdm.recur_backward_q(shape, *L, mem, kind, codes, scales, dy, grads["dv"], grads["dalpha"], grads["dbeta"],
                             grads["dw_w"], grads["dw_r"], dM, stream=st)     # back to M_0

        def fwd_quant_zero():
            sdm.recur_undo(shape, *L, mem, y, undo, ws, stream=st)
            sdm.undo_quantize(shape, undo, kind, codes, scales, stream=st)
            dM.zero_()
        ms_bq = timed(lambda: sdm.recur_backward_q(shape, *L, mem, kind, codes, scales, dy, grads["dv"], grads["dalpha"],
                                                   grads["dbeta"], grads["dw_w"], grads["dw_r"], dM, stream=st),
                      steps, between=fwd_quant_zero)
        out[f"snapshot_{kind}"] = {"quantize_ms": ms_q, "quantize_gbs": q_bytes / (ms_q * 1e-3) / 1e9,
                                   "snapshot_bytes": codes.numel() + rows * 4, "backward_ms": ms_bq}
        del codes
    if sdm.device_status(st) != 0:
        raise RuntimeError("device status word set in the next-rows leg")
    out["timing"] = f"{warmup} untimed + {steps} timed calls each, CUDA events around each call"
    return out


def run_leg(args):
    """`bench.py --leg NAME`: one workload leg in its own process, printing one JSON object."""
    import torch
    from paper_2607_07386_gb300.build import build
    torch.cuda.set_device(0)
    build()
    if args.leg == "decode":
        res = leg_decode(args.steps, args.warmup)
    elif args.leg == "next_rows":
        res = leg_next(args.steps, args.warmup)
    else:
        res = leg_scan(args.leg, args.steps, args.warmup)
    print(json.dumps(res), flush=True)


def legs_in_subprocesses(names, warmup: int) -> dict:
    """Each (leg, steps) in a child process (its own CUDA context and memory), after the main
    leg has released its memory; a leg that fails reports its error instead of a result."""
    out = {}
    for name, st in names:
        cmd = [sys.executable, os.path.abspath(__file__), "--leg", name, "--steps", str(st), "--warmup", str(warmup)]
        try:
            r = subprocess.run(cmd, capture_output=True, text=True, timeout=900)
            lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
            out[name] = json.loads(lines[-1]) if r.returncode == 0 and lines else {
                "error": f"exit {r.returncode}: " + (r.stderr.strip().splitlines() or ["?"])[-1][:300]}
        except Exception as e:          # timeout or a crashed child: report it, keep the main line
            out[name] = {"error": repr(e)[:300]}
    return out


def run_ours(args, cfg):
    import torch
    import paper_2607_07386_gb300 as sdm
    from paper_2607_07386_gb300.build import build
    from synth.torch_io import to_torch, torch_dtype

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    if rank == 0:
        build()
    if world > 1:
        dist.barrier()
    build()   # no-op when up to date; loads in every rank

    # ---- inputs (rank r owns sequences [r*B, (r+1)*B) of the global batch), resident in HBM
    full = synth.full_inputs(cfg, b0=shard_b0(rank, cfg.B))
    dt = torch_dtype(cfg.dtype)
    dev = {n: to_torch(a, cfg.dtype) for n, a in full.items()}
    host_pinned = {n: torch.from_numpy(np.ascontiguousarray(full[n]).view(np.int16 if cfg.dtype == "bf16" else np.float32))
                   .view(dt).pin_memory() for n in ("q", "k", "v", "alpha", "beta")}
    del full
    B, H, T, N, dv = cfg.B, cfg.H, cfg.T, cfg.N, cfg.d_v
    shape = sdm.SdmShape.make(B, H, T, cfg.d_k, dv, N, cfg.k_write, cfg.k_read, cfg.dtype)
    mem = torch.empty((B, H, N, dv), dtype=dt, device="cuda")
    y = torch.empty((B, H, T, dv), dtype=dt, device="cuda")
    ws = torch.empty(sdm.workspace_bytes(shape), dtype=torch.uint8, device="cuda")
    idx_w = torch.empty((B, H, T, cfg.k_write), dtype=torch.int32, device="cuda")
    w_w = torch.empty((B, H, T, cfg.k_write), dtype=torch.float32, device="cuda")
    idx_r = torch.empty((B, H, T, cfg.k_read), dtype=torch.int32, device="cuda")
    w_r = torch.empty((B, H, T, cfg.k_read), dtype=torch.float32, device="cuda")
    stream = torch.cuda.current_stream()

    def step():   # mem = M0 broadcast (overlapping the addressing), then the forward pass
        sdm.forward_m0(shape, dev["M0"], dev["P_q"], dev["P_k"], dev["q"], dev["k"], dev["v"], dev["alpha"],
                       dev["beta"], mem, y, ws, stream=stream)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    def max_over_ranks(x: float) -> float:
        return reduce_max(x, dist if world > 1 else None, device="cuda")

    for _ in range(args.warmup):
        step()
    barrier()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(local).uuid)
    except Exception:
        gpu_id = str(local)
    with ClockSampler(gpu_id) as clk:
        barrier()
        clk.mark_start()
        ev0.record(stream)
        for _ in range(args.steps):
            step()
        ev1.record(stream)
        barrier()
        clk.mark_end()
    ms_total = max_over_ranks(ev0.elapsed_time(ev1))
    ms_step = ms_total / args.steps
    clocks = clk.summary()
    if sdm.device_status(stream) != 0:
        raise RuntimeError("device status word set during the benchmark")

    # ---- per-phase timing (same work split at the C ABI: init / addressing / recurrence)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(args.steps)]
    barrier()
    for s in range(args.steps):
        e = evs[s]
        e[0].record(stream)
        sdm.init_memory(shape, dev["M0"], mem, stream)
        e[1].record(stream)
        sdm.address(shape, dev["P_q"], dev["P_k"], dev["q"], dev["k"], idx_w, w_w, idx_r, w_r, ws, stream=stream)
        e[2].record(stream)
        sdm.recur(shape, idx_w, w_w, idx_r, w_r, dev["v"], dev["alpha"], dev["beta"], mem, y, ws, stream=stream)
        e[3].record(stream)
    barrier()
    ph = {"init_memory": 0.0, "address": 0.0, "recurrence": 0.0}
    for e in evs:
        ph["init_memory"] += e[0].elapsed_time(e[1]) / args.steps
        ph["address"] += e[1].elapsed_time(e[2]) / args.steps
        ph["recurrence"] += e[2].elapsed_time(e[3]) / args.steps

    # ---- the same step on the copy-on-write memory (sdm_forward_lazy, no broadcast): every
    # step is a fresh sequence, so its touched bitmaps are cleared first
    lazy = None
    if T > 1:
        ws_l = torch.empty(sdm.lazy_workspace_bytes(shape), dtype=torch.uint8, device="cuda")
        touched = torch.empty((B, H, sdm.touched_words(shape)), dtype=torch.int32, device="cuda")

        def lazy_step():
            touched.zero_()
            sdm.forward_lazy(shape, dev["M0"], touched, dev["P_q"], dev["P_k"], dev["q"], dev["k"], dev["v"],
                             dev["alpha"], dev["beta"], mem, y, ws_l, stream=stream)

        for _ in range(args.warmup):
            lazy_step()
        barrier()
        ev0.record(stream)
        for _ in range(args.steps):
            lazy_step()
        ev1.record(stream)
        barrier()
        ms_lazy = max_over_ranks(ev0.elapsed_time(ev1)) / args.steps
        if sdm.device_status(stream) != 0:
            raise RuntimeError("device status word set during the lazy-M0 benchmark")
        lazy = {"value": tokens_step_of(B, T, world) / (ms_lazy * 1e-3), "unit": UNIT, "ms_per_step": ms_lazy,
                "step": "bitmap clear + sdm_forward_lazy: addressing + first-writer table + recurrence gathering "
                        "unwritten rows from M0 (no broadcast; same y and memory state as the broadcast step)",
                "gpu_launches": 10 * args.steps}
        del ws_l, touched

    # ---- the steps around the path (gate preparation, output epilogue), timed apart from the step
    around = None
    if T > 1:
        from synth.gen import layer_inputs
        li = layer_inputs(cfg)
        d_model = H * dv
        lx, lwa, lwb, lg = (to_torch(li[n], cfg.dtype) for n in ("x", "W_a", "W_b", "g"))
        lbdt, lA, lgam = (torch.from_numpy(li[n]).cuda() for n in ("b_dt", "A", "gamma"))
        del li
        a_o = torch.empty((B, H, T), dtype=dt, device="cuda")
        b_o = torch.empty_like(a_o)
        z = torch.empty((B, T, H, dv), dtype=dt, device="cuda")
        W_o = (torch.randn(d_model, H * dv, device="cuda") / (H * dv) ** 0.5).to(dt)
        o_mix = torch.empty((B * T, d_model), dtype=dt, device="cuda")
        runs = {"gates": lambda: sdm.gates(shape, d_model, lx, lwa, lwb, lbdt, lA, a_o, b_o, stream=stream),
                "norm_gate": lambda: sdm.norm_gate(shape, y, lg, lgam, 1e-6, z, stream=stream),
                "head_mix": lambda: sdm.head_mix(shape, d_model, z.view(B * T, H * dv), W_o, o_mix, stream=stream),
                "w_o_gemm": lambda: torch.matmul(z.view(B * T, H * dv), W_o.t())}
        ms = {}
        for name, fn in runs.items():
            for _ in range(args.warmup):
                fn()
            barrier()
            ev0.record(stream)
            for _ in range(args.steps):
                fn()
            ev1.record(stream)
            barrier()
            ms[name] = max_over_ranks(ev0.elapsed_time(ev1)) / args.steps
        es = cfg.elem_bytes
        g_bytes = B * T * d_model * es + 2 * H * d_model * es + 2 * B * H * T * es
        n_bytes = 3 * B * H * T * dv * es + dv * 4
        w_flop = 2.0 * B * T * (H * dv) * d_model
        around = {
            "note": "sdm_gates, sdm_norm_gate and sdm_head_mix (library kernels; the gates and the head mix on "
                    "the tensor cores), each timed alone, with cuBLAS's GEMM of the same head mix beside them for "
                    "comparison; inputs larger than L2",
            "d_model": d_model,
            "gates": {"ms": ms["gates"], "gbs": g_bytes / (ms["gates"] * 1e-3) / 1e9,
                      "gflops": 4.0 * B * T * H * d_model / (ms["gates"] * 1e-3) / 1e9},
            "norm_gate": {"ms": ms["norm_gate"], "gbs": n_bytes / (ms["norm_gate"] * 1e-3) / 1e9,
                          "frac_of_measured_hbm": n_bytes / (ms["norm_gate"] * 1e-3) / 1e9 / _peaks()["hbm_gbs"]},
            "head_mix": {"ms": ms["head_mix"], "tflops": w_flop / (ms["head_mix"] * 1e-3) / 1e12,
                         "frac_of_measured_bf16": w_flop / (ms["head_mix"] * 1e-3) / 1e12 / _peaks()["bf16_tflops"]},
            "gates_tensor_cores": sdm.gates_tensor_cores(shape, d_model),
            "w_o_gemm_cublas": {"ms": ms["w_o_gemm"], "tflops": w_flop / (ms["w_o_gemm"] * 1e-3) / 1e12},
        }
        del lx, lwa, lwb, lg, a_o, b_o, z, W_o, o_mix

    # ---- end to end through the public API with host buffers (pinned), copies inside the region
    h2d = sum(t.numel() * t.element_size() for t in host_pinned.values())
    y_host = torch.empty(y.shape, dtype=dt, pin_memory=True)
    d2h = y_host.numel() * y_host.element_size()

    # Two input sets and two outputs: the copy stream brings step i+1's inputs in and takes
    # step i-1's y out while step i computes; every step's copies are inside the timed region.
    names = ("q", "k", "v", "alpha", "beta")
    bufs = [{n: dev[n] for n in names}, {n: torch.empty_like(dev[n]) for n in names}]
    ys = [y, torch.empty_like(y)]
    y_hosts = [y_host, torch.empty(y.shape, dtype=dt, pin_memory=True)]
    cs = torch.cuda.Stream()

    def step_on(inp, yo):
        sdm.forward_m0(shape, dev["M0"], dev["P_q"], dev["P_k"], inp["q"], inp["k"], inp["v"], inp["alpha"],
                       inp["beta"], mem, yo, ws, stream=stream)

    def e2e_run(nsteps, start_event):
        ev = lambda: torch.cuda.Event()
        h2d_done, comp_done, d2h_done = [ev(), ev()], [None] * nsteps, [None, None]
        cs.wait_event(start_event)
        with torch.cuda.stream(cs):
            for n in names:
                bufs[0][n].copy_(host_pinned[n], non_blocking=True)
        h2d_done[0].record(cs)
        for i in range(nsteps):
            sb = i % 2
            stream.wait_event(h2d_done[sb])
            if d2h_done[sb] is not None:
                stream.wait_event(d2h_done[sb])      # y buffer free again
            step_on(bufs[sb], ys[sb])
            comp_done[i] = ev()
            comp_done[i].record(stream)
            if i + 1 < nsteps:
                nb = (i + 1) % 2
                if i >= 1:
                    cs.wait_event(comp_done[i - 1])  # inputs of step i-1 consumed
                with torch.cuda.stream(cs):
                    for n in names:
                        bufs[nb][n].copy_(host_pinned[n], non_blocking=True)
                h2d_done[nb].record(cs)
            cs.wait_event(comp_done[i])
            with torch.cuda.stream(cs):
                y_hosts[sb].copy_(ys[sb], non_blocking=True)
            d2h_done[sb] = ev()
            d2h_done[sb].record(cs)
        for e in d2h_done:
            if e is not None:
                stream.wait_event(e)

    e2e_run(2, torch.cuda.Event())
    barrier()
    ev0.record(stream)
    e2e_run(args.steps, ev0)
    ev1.record(stream)
    barrier()
    ms_e2e = max_over_ranks(ev0.elapsed_time(ev1)) / args.steps

    tokens_step = B * T * world
    peaks = _peaks()
    rec_bytes = cfg.recurrence_bytes_per_token_head() * B * H * T
    rec_ms = max_over_ranks(ph["recurrence"])
    achieved = rec_bytes / (rec_ms * 1e-3) / 1e9
    step_bytes = cfg.algorithmic_bytes_per_token_head() * B * H * T + (1 + B) * H * N * dv * cfg.elem_bytes
    kernels_per_step = 8   # init, P row norms, scores, finalize (3 passes), hazard pass, recurrence
    line = {
        "metric": METRIC, "value": weak_scaling_value(B, T, world, ms_step), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": cfg.dtype, "data": "synthetic",
        "config": {"workload": _workload_desc(cfg), "global_batch": B * world, "seq_len": T,
                   "parallelism": f"independent sequence shards x{world}" if world > 1 else "single GPU",
                   "step": "sdm_forward_m0: M0 broadcast (side stream, overlapping the addressing) + addressing + recurrence",
                   "l2": f"inputs larger than L2: {B * H * N * dv * cfg.elem_bytes / 1e9:.2f} GB memory state"},
        "e2e": {"value": tokens_step / (ms_e2e * 1e-3), "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": kernels_per_step * args.steps,
        "roofline": {"bound": "hbm", "kernel": "k_hazard + k_recur_tw (the recurrence phase)", "achieved": achieved, "peak": peaks["hbm_gbs"],
                     "unit": "GB/s", "frac": achieved / peaks["hbm_gbs"], "frac_of_8tbs": achieved / 8000.0,
                     "traffic": RECUR_DRAM_BYTES_PER_TOKEN_HEAD * B * H * T if cfg.name == "layer_1p4b" else None,
                     "traffic_source": "ncu dram__bytes_read.sum + dram__bytes_write.sum of k_hazard + k_recur_tw, "
                                       "one launch on this workload (B=8)",
                     "peak_source": peaks["source"], "bytes_per_launch": rec_bytes, "ms_per_launch": rec_ms},
        "phase_ms": ph,
        "lazy_m0": lazy,
        "around_the_path": around,
        "step_hbm": {"algorithmic_bytes": step_bytes, "gbs": step_bytes / (ms_step * 1e-3) / 1e9,
                     "frac_of_measured": step_bytes / (ms_step * 1e-3) / 1e9 / peaks["hbm_gbs"],
                     "frac_of_8tbs": step_bytes / (ms_step * 1e-3) / 1e9 / 8000.0},
        "clocks": clocks,
    }
    if rank == 0 and world == 1 and not args.no_legs:
        # the other workloads (scan workloads and decode), each in its own process once this
        # process has released its device memory
        del dev, mem, y, ws, idx_w, w_w, idx_r, w_r, bufs, ys
        torch.cuda.synchronize()
        torch.cuda.empty_cache()
        line["workloads"] = legs_in_subprocesses(
            [("small_bf16", max(args.steps, 10)), ("long_ctx", 3), ("decode", 1000), ("next_rows", 2)], args.warmup)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="layer_1p4b", choices=sorted(synth.CONFIGS))
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-legs", action="store_true", help="skip the other workloads' legs")
    ap.add_argument("--leg", default=None, help=argparse.SUPPRESS)   # internal: one workload leg
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.leg:
        run_leg(args)
        return
    cfg = synth.get_config(args.config)
    if cfg.is_decode:
        raise SystemExit("the decode workload is timed by the decode leg of the default run")
    if args.impl == "reference":
        run_reference(args, cfg)
    else:
        run_ours(args, cfg)


if __name__ == "__main__":
    main()
