"""The multi-GPU path is N independent replicas (no data-path exchange):
bench.py gives every rank its own seeded workload, times each rank, and
reports the units of all ranks over the slowest rank's time.  These tests run
that logic as two gloo processes on the CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2501_06807_gb300 import synth


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        w = bench.replica_workload(synth.C5, rank)
        ms = 10.0 + 5.0 * rank                      # rank 1 is the slower one
        t = bench.max_over_ranks(ms, dist)
        v = bench.job_value(1000, world, t)
        seeds = [None] * world
        dist.all_gather_object(seeds, w.seed)
        out[rank] = (t, v, tuple(seeds))
    finally:
        dist.destroy_process_group()


def test_two_replicas_aggregate_over_gloo():
    world = 2
    out = mp.get_context("spawn").Manager().dict()  # no fork of a threaded process
    mp.spawn(_worker, args=(world, _free_port(), out), nprocs=world, join=True)
    for r in range(world):
        t, v, seeds = out[r]
        assert t == 15.0                             # max over ranks
        assert v == pytest.approx(1000 * 2 / 0.015)  # all ranks' units / slowest time
        assert len(set(seeds)) == world              # independent inputs per replica
    assert out[0][2][0] == synth.C5.seed


def test_single_rank_helpers():
    assert bench.max_over_ranks(3.5, None) == 3.5
    assert bench.replica_workload(synth.C3, 0) is synth.C3
    assert bench.job_value(500, 1, 2.0) == pytest.approx(250_000)


def test_reference_arm_rank_nonzero_does_no_work(monkeypatch):
    called = []
    monkeypatch.setattr(bench, "oracle_sample", lambda *a, **k: called.append(1))

    class A:
        workload, warmup, steps = synth.C1.name, 1, 1
    assert bench.run_reference(A, 1, 2) is None
    assert not called


def test_reference_arm_prints_one_contract_line():
    """`bench.py --impl reference` (the oracle on the host cores) prints one
    JSON line with the keys the run driver reads, on the same metric, unit
    and workload config as the CUDA arm."""
    import json
    import subprocess
    import sys
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", synth.C1.name,
                        "--steps", "1", "--warmup", "0"], capture_output=True, text=True, timeout=600,
                       cwd=os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference"
    assert d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert (d["n_gpus"], d["steps"], d["warmup"]) == (1, 1, 0)
    assert d["config"] == bench.workload_config(synth.C1, synth.C1.decode_steps, "cpu")
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
