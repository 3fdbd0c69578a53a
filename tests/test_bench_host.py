"""Host logic of bench.py on the CPU.  Ranks: two gloo ranks (one process each, launched as
torchrun would, rendezvous on 127.0.0.1); every rank replays its own replica of the workload
(weak scaling, no collective on the data path), the job's time is the slowest rank's, and the
rate counts every rank's tokens.  Roofline: the decode kernel's algorithmic bytes per launch,
checked against a count by hand.  Oracle baseline: the process pool's size and the step's
schedule of units over it."""
import os
import socket
import subprocess
import sys

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, local, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        out[rank] = bench.max_over_ranks(local[rank], torch, dist, "cpu")
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_slowest_rank_sets_the_time_gloo_world_2():
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    with ctx.Manager() as manager:
        out = manager.dict()
        mp.start_processes(_rank, args=(2, _free_port(), [183.0, 191.5], out), nprocs=2, join=True,
                           start_method="spawn")
        got = dict(out)
    assert got == {0: 191.5, 1: 191.5}


def test_single_process_time_is_local():
    import torch
    import torch.distributed as dist
    assert bench.max_over_ranks(12.5, torch, dist, "cpu") == 12.5


def test_whole_job_rate_counts_every_rank():
    # 256 tokens per rank and step, 2 ranks, 5 steps in 0.5 s
    assert bench.whole_job_rate(2, 256 * 5, 0.5) == pytest.approx(5120.0)
    assert bench.whole_job_rate(1, 256 * 5, 0.5) == pytest.approx(2560.0)


def test_reference_arm_prints_on_rank_0_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1"],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""


def test_decode_bytes_per_launch_by_hand():
    """One launch of the 100k workload at token t: 8 KV heads x (25,000 + t + 1) rows of
    K_c, V_c (256 bytes each, bf16 d = 128), a 4-byte bias per position (shared by the KV
    heads; per KV head in the per-head mode), plus q and out (32 heads x 256 bytes each) and the
    appended k and v (8 heads x 256 bytes each)."""
    import synth
    wl = synth.WORKLOADS["long_100k"]
    T = 256
    per_token = [(25000 + t + 1) * (8 * 512 + 4) + 2 * 32 * 256 + 2 * 8 * 256 for t in range(T)]
    assert bench.decode_bytes_per_launch(wl, [100000], T) == pytest.approx(sum(per_token) / T)
    assert bench.decode_bytes_per_launch(wl, [100000], T) == pytest.approx(103047330.0)
    per_head = [8 * (25000 + t + 1) * 516 + 2 * 32 * 256 + 2 * 8 * 256 for t in range(T)]
    assert bench.decode_bytes_per_launch(wl, [100000], T, per_head=True) == pytest.approx(sum(per_head) / T)


def test_oracle_pool_sized_by_the_steps_units(monkeypatch):
    """One worker per (sequence, layer) unit of the step, at most one per core; the cores left
    over go to the workers as BLAS threads."""
    import synth
    monkeypatch.setattr(os, "cpu_count", lambda: 16)
    wl = synth.WORKLOADS["long_100k"]                      # 32 layers x 1 sequence
    p = bench._OraclePool.for_step(wl)
    assert (p.P, p.blas_threads) == (16, 1)
    p = bench._OraclePool.for_step(synth.WORKLOADS["llama_layer"])   # one unit
    assert (p.P, p.blas_threads) == (1, 16)
    p = bench._OraclePool.for_step(wl.with_(layers=5))
    assert (p.P, p.blas_threads) == (5, 3)


def test_step_rate_schedules_units_in_rounds():
    """B x L units on P workers take ceil(B L / P) rounds of the mean unit (compression +
    decode_steps tokens); the rate is the step's tokens over that time."""
    import synth
    wl = synth.WORKLOADS["long_100k"]                      # 32 units, 256 tokens a step
    res = [{"compress_s": 8.0, "decode_s_per_token": 0.1}, {"compress_s": 10.0, "decode_s_per_token": 0.1}]
    rate, rounds = bench._step_rate(wl, res, 16)
    assert rounds == 2
    assert rate == pytest.approx(256 / (2 * (9.0 + 256 * 0.1)))
    rate, rounds = bench._step_rate(wl, res, 12)
    assert rounds == 3
    assert rate == pytest.approx(256 / (3 * (9.0 + 256 * 0.1)))
