"""The N > 1 path of bench.py on CPU: two gloo ranks on 127.0.0.1.

The hot path does not shard across GPUs in this build (replicas only): each
rank runs the whole layer on its own batch and the ranks exchange nothing but
a barrier and the max-over-ranks reduction of the timed region. These tests
run that logic as two processes with the gloo backend: the barrier holds both
ranks, the reduction returns the slowest rank's time on every rank, the
whole-job throughput counts both ranks' work over that time, and the CPU
reference arm does its work and prints on rank 0 only.
"""
import json
import multiprocessing as mp
import os
import socket
import sys
import time
import types

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, ws, port, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(ws),
                      LOCAL_RANK=str(rank))
    sys.path.insert(0, ROOT)
    import importlib.util

    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    import torch.distributed as dist

    args = types.SimpleNamespace(impl="reference", steps=1, warmup=0, K=64)
    got_ws, got_rank, _ = bench.dist_setup(args, backend="gloo")
    res = {"ws": got_ws, "rank": got_rank}
    # barrier: rank 1 arrives late; rank 0 must wait for it
    t0 = time.time()
    if rank == 1:
        time.sleep(0.5)
    bench.barrier(got_ws)
    res["waited"] = time.time() - t0
    # max over ranks of a per-rank time
    ms = 10.0 + 5.0 * rank
    res["ms_max"] = bench.max_over_ranks(ms, got_ws)
    res["rate"] = bench.job_rate(2048 * 3, got_ws, res["ms_max"])
    # the reference arm works and prints on rank 0 only
    if rank != 0:
        res["reference"] = bench.reference(args, got_ws, got_rank)
    dist.destroy_process_group()
    with open(os.path.join(out_dir, f"rank{rank}.json"), "w") as f:
        json.dump(res, f)


def test_two_gloo_ranks_barrier_max_and_job_rate(tmp_path):
    ws, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_rank_main, args=(r, ws, port, str(tmp_path))) for r in range(ws)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0, f"rank process exited with {p.exitcode}"
    res = [json.load(open(tmp_path / f"rank{r}.json")) for r in range(ws)]
    for r, x in enumerate(res):
        assert x["ws"] == 2 and x["rank"] == r
        assert x["ms_max"] == 15.0  # the slowest rank's time on every rank
        assert x["rate"] == pytest.approx(2 * 2048 * 3 / 0.015)
    assert res[0]["waited"] >= 0.4  # rank 0 was held at the barrier until rank 1 came
    assert res[1]["reference"] is None


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import importlib.util

    spec = importlib.util.spec_from_file_location("bench_mod1", os.path.join(ROOT, "bench.py"))
    bench = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(bench)
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.job_rate(1000, 1, 500.0) == pytest.approx(2000.0)
    bench.barrier(1)
