"""The multi-rank (N > 1) path of the benchmark, on CPU with gloo.

The path shards by sequence: rank r owns global sequences [r*B, (r+1)*B).  Their (b, h) chains are
independent, so the shards need no data-path collective.  The only collective is the max of the
per-rank step times.  These tests check that:

- the shards partition the global batch;
- two gloo ranks, each running the float64 oracle on its own shard, reproduce the one-process
  result for the global batch;
- the max-over-ranks reduction and the whole-job weak-scaling value come out right.
"""
import json
import multiprocessing as mp
import os
import socket

import numpy as np
import pytest

import synth

torch = pytest.importorskip("torch")


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_rank_shards_partition_the_global_batch():
    import bench
    cfg = synth.TINY_FP32.with_(B=2, T=32)
    world = 3
    glob = synth.full_inputs(cfg.with_(B=cfg.B * world))
    for r in range(world):
        part = synth.full_inputs(cfg, b0=bench.shard_b0(r, cfg.B))
        for name in ("q", "k", "v", "alpha", "beta"):
            assert np.array_equal(part[name], glob[name][r * cfg.B:(r + 1) * cfg.B]), (r, name)
        assert np.array_equal(part["M0"], glob["M0"])          # parameters are shared, not sharded


def _rank_main(rank: int, world: int, port: int, out_dir: str):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    import torch.distributed as dist
    import bench
    from oracle.reference_run import oracle_slice
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        cfg = synth.TINY_FP32.with_(B=1, T=48)
        b0 = bench.shard_b0(rank, cfg.B)
        # the global sequence b0 + b of the batch, computed on this rank alone
        gcfg = cfg.with_(B=cfg.B * world)
        ys = {b0 + b: oracle_slice(gcfg, b0 + b, 0)["y"] for b in range(cfg.B)}
        step_ms = 10.0 + 5.0 * rank                             # a stand-in per-rank step time
        ms_max = bench.reduce_max(step_ms, dist)
        gathered = [None] * world
        dist.all_gather_object(gathered, {int(k): v.tolist() for k, v in ys.items()})
        if rank == 0:
            line = {"ms_max": ms_max, "value": bench.weak_scaling_value(cfg.B, cfg.T, world, ms_max),
                    "y": {k: v for part in gathered for k, v in part.items()}}
            with open(os.path.join(out_dir, "rank0.json"), "w") as f:
                json.dump(line, f)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_shard_without_exchange_and_reduce_the_max(tmp_path):
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, str(tmp_path))) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
    for p in procs:
        if p.is_alive():
            p.kill()
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    line = json.load(open(tmp_path / "rank0.json"))
    assert line["ms_max"] == 15.0
    cfg = synth.TINY_FP32.with_(B=1, T=48)
    assert line["value"] == pytest.approx(cfg.B * cfg.T * world / 15e-3)
    # every global sequence appears once, and equals the one-process oracle of the global batch
    from oracle.reference_run import oracle_slice
    gcfg = cfg.with_(B=world)
    assert sorted(int(k) for k in line["y"]) == list(range(world))
    for b in range(world):
        assert np.array_equal(np.array(line["y"][str(b)]), oracle_slice(gcfg, b, 0)["y"]), b


def test_reduce_max_is_the_identity_on_one_rank():
    import bench
    assert bench.reduce_max(3.5) == 3.5
    assert bench.weak_scaling_value(8, 4096, 1, 10.0) == pytest.approx(8 * 4096 / 0.01)
