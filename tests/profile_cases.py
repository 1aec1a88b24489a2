"""Single-case GPU runs for profiler captures (ncu) of the hot path, on device-drawn inputs of a
workload's shapes and distributions.  Each case sets up its inputs, runs the captured call
`--reps` times on one stream, prints one JSON line with the CUDA-event time per call and exits
non-zero if the device status word is set.

    python -m tests.profile_cases recur layer_1p4b --B 8 --reps 2     # hazard pass + recurrence
    python -m tests.profile_cases address layer_1p4b --B 2 --reps 2   # scores, selection, finalize
    python -m tests.profile_cases step layer_1p4b --reps 2            # sdm_forward_m0
    python -m tests.profile_cases decode --H 16 --reps 20             # sdm_decode_step, T = 1

The setup launches (input generation, the addressing and broadcast in front of `recur`) and the
`--warmup` calls come before the timed ones; `ncu -k regex:<kernel> -s <n> -c <n>` picks the
captured launches out.
"""
from __future__ import annotations

import argparse
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main(argv=None) -> int:
    ap = argparse.ArgumentParser(description=__doc__.splitlines()[0])
    ap.add_argument("case", choices=("recur", "address", "step", "decode"))
    ap.add_argument("config", nargs="?", default="layer_1p4b")
    ap.add_argument("--B", type=int, default=0, help="batch (0: the workload's own)")
    ap.add_argument("--T", type=int, default=0, help="tokens (0: the workload's own)")
    ap.add_argument("--H", type=int, default=0, help="heads (0: the workload's own)")
    ap.add_argument("--N", type=int, default=0, help="memory slots (0: the workload's own)")
    ap.add_argument("--reps", type=int, default=2)
    ap.add_argument("--warmup", type=int, default=2, help="untimed calls before the timed ones")
    args = ap.parse_args(argv)

    import torch
    import bench
    import synth
    import paper_2607_07386_gb300 as sdm
    from synth.torch_io import torch_dtype

    cfg = synth.get_config("decode" if args.case == "decode" else args.config)
    if args.B:
        cfg = cfg.with_(B=args.B)
    if args.T and args.case != "decode":
        cfg = cfg.with_(T=args.T)
    if args.H:
        cfg = cfg.with_(H=args.H)
    if args.N:
        cfg = cfg.with_(N=args.N)
    torch.cuda.set_device(0)
    st = torch.cuda.Stream()
    B, H, T, N, dv = cfg.B, cfg.H, cfg.T, cfg.N, cfg.d_v
    dt = torch_dtype(cfg.dtype)
    with torch.cuda.stream(st):
        if args.case == "decode":
            dev = bench.device_inputs(cfg.with_(T=args.reps), seed=cfg.seed)
            T = 1
        else:
            dev = bench.device_inputs(cfg, seed=cfg.seed)
        shape = sdm.SdmShape.make(B, H, T, cfg.d_k, dv, N, cfg.k_write, cfg.k_read, cfg.dtype)
        mem = torch.empty((B, H, N, dv), dtype=dt, device="cuda") if args.case != "address" else None
        y = torch.empty((B, H, T, dv), dtype=dt, device="cuda")
        ws = torch.empty(sdm.workspace_bytes(shape), dtype=torch.uint8, device="cuda")
        lists = {n: torch.empty((B, H, T, k), dtype=tt, device="cuda")
                 for n, k, tt in (("idx_w", cfg.k_write, torch.int32), ("w_w", cfg.k_write, torch.float32),
                                  ("idx_r", cfg.k_read, torch.int32), ("w_r", cfg.k_read, torch.float32))}

        def address():
            sdm.address(shape, dev["P_q"], dev["P_k"], dev["q"], dev["k"], lists["idx_w"], lists["w_w"],
                        lists["idx_r"], lists["w_r"], ws, stream=st)

        def recur():
            sdm.recur(shape, lists["idx_w"], lists["w_w"], lists["idx_r"], lists["w_r"], dev["v"], dev["alpha"],
                      dev["beta"], mem, y, ws, stream=st)

        def step():
            sdm.forward_m0(shape, dev["M0"], dev["P_q"], dev["P_k"], dev["q"], dev["k"], dev["v"], dev["alpha"],
                           dev["beta"], mem, y, ws, stream=st)

        per = None
        if args.case == "decode":
            per = [{n: dev[n][:, :, i].contiguous() for n in ("q", "k", "v", "alpha", "beta")} for i in range(args.reps)]
            yd = y.view(B, H, dv)

        def decode(i):
            x = per[i]
            sdm.decode_step(shape, dev["P_q"], dev["P_k"], x["q"], x["k"], x["v"], x["alpha"], x["beta"], mem, yd, ws,
                            stream=st)

        def call(i):
            if args.case == "recur":
                recur()
            elif args.case == "address":
                address()
            elif args.case == "step":
                step()
            else:
                decode(i % len(per))

        if args.case in ("recur", "decode"):
            sdm.init_memory(shape, dev["M0"], mem, st)
        if args.case == "recur":
            address()
        for i in range(args.warmup):
            call(i)
        st.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(st)
        for i in range(args.reps):
            call(i)
        e1.record(st)
        st.synchronize()
        status = sdm.device_status(st)
    ms = e0.elapsed_time(e1) / args.reps
    print(json.dumps({"case": args.case, "workload": cfg.name, "B": B, "H": H, "T": T, "reps": args.reps,
                      "ms_per_call": round(ms, 4), "status": status}), flush=True)
    return 0 if status == 0 else 1


if __name__ == "__main__":
    sys.exit(main())
