"""Multi-process (gloo, world size 2, CPU) tests of the N > 1 paths.

* replicas: each rank builds its own sequences; the job time is the max over
  ranks and the rate counts the units of every rank (bench.py helpers);
* the vocabulary-parallel exchange step (designed, not built on the GPU):
  per-shard (max, sum exp, top-k) partials all-gathered and merged equal the
  unsharded log-softmax and top-k of the oracle.
"""
import datetime
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from oracle.shard import merge_partials, shard_partials
from workloads import Config, make_sequences


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run(rank, world, port, fn, out_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    # a rank that fails ends the others' next collective within a minute
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=datetime.timedelta(seconds=60))
    try:
        fn(rank, world, out_dir)
    finally:
        dist.barrier()
        dist.destroy_process_group()


def spawn(fn, tmp_path, world=2):
    oracle.build()  # once, before the ranks start
    mp.spawn(_run, args=(world, free_port(), fn, str(tmp_path)), nprocs=world, join=True)


def _replicas(rank, world, out_dir):
    import bench
    cfg = Config("rep", 2, 300, 64, 3, 4, 4, 8, "bf16", 0.0, 5)
    Dlog, h0 = make_sequences(cfg, rank=rank)
    np.save(os.path.join(out_dir, f"h0_{rank}.npy"), h0)
    local_ms = 3.0 + rank  # pretend rank 1 is the slowest
    ms = bench.allreduce_max(local_ms, world)
    assert ms == 3.0 + world - 1
    rate = bench.whole_job_rate(cfg.expansions_per_round(), world, ms / 1e3)
    assert abs(rate - cfg.expansions_per_round() * world / (ms / 1e3)) < 1e-9


def test_replicas_gloo(tmp_path):
    spawn(_replicas, tmp_path)
    h0a = np.load(tmp_path / "h0_0.npy")
    h0b = np.load(tmp_path / "h0_1.npy")
    assert not np.array_equal(h0a, h0b)  # each replica works on its own sequences
    cfg = Config("rep", 2, 300, 64, 3, 4, 4, 8, "bf16", 0.0, 5)
    np.testing.assert_array_equal(make_sequences(cfg, rank=0)[1], h0a)


def _vocab_shards(rank, world, out_dir):
    cfg = Config("vp", 1, 1003, 32, 2, 4, 7, 8, "f32", 0.7, 6)
    g = np.random.Generator(np.random.PCG64(11))
    E = (g.standard_normal((cfg.V, cfg.d)) * 0.5).astype(np.float32)
    dlog = (g.standard_normal(cfg.V) * 2).astype(np.float32)
    dlog[[5, 900]] = -np.inf
    h = g.standard_normal(cfg.d)
    z = oracle.child_logits(cfg, E, dlog, h)
    v0 = rank * cfg.V // world
    v1 = (rank + 1) * cfg.V // world
    m, s, vals, toks = shard_partials(z[v0:v1], v0, cfg.k)
    # one exchange: 2 + 2k values per node from every rank
    msg = torch.tensor(np.concatenate([[m, s], vals, toks.astype(np.float64)]), dtype=torch.float64)
    got = [torch.empty_like(msg) for _ in range(world)]
    dist.all_gather(got, msg)
    parts = [(float(t[0]), float(t[1]), t[2:2 + cfg.k].numpy(), t[2 + cfg.k:].numpy().astype(np.int64))
             for t in got]
    lse, lq, tk = merge_partials(parts, cfg.k)
    ref_lq, ref_lse = oracle.log_softmax(z)
    ref_tk = oracle.topk(ref_lq, cfg.k)
    assert abs(lse - ref_lse) < 1e-12
    np.testing.assert_array_equal(tk, ref_tk)
    np.testing.assert_allclose(lq, ref_lq[ref_tk], atol=1e-12)


@pytest.mark.parametrize("world", [2, 3])
def test_vocab_parallel_merge_gloo(tmp_path, world):
    """world = 3 splits the 1003 tokens unevenly (334 / 334 / 335)."""
    spawn(_vocab_shards, tmp_path, world=world)


def test_reference_arm_under_torchrun_prints_one_line():
    """`bench.py --impl reference` launched with two ranks: rank 0 alone runs
    the oracle and prints one JSON line; the other rank exits 0 without work."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(free_port()), os.path.join(root, "bench.py"),
           "--impl", "reference", "--config", "toy", "--gpus", "2", "--steps", "1", "--warmup", "3",
           "--cpu-seconds", "2"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=root)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    j = json.loads(lines[0])
    assert j["impl"] == "reference" and j["n_gpus"] == 2 and j["value"] > 0
    assert j["cpu_baseline"]["kind"] == "oracle" and j["cpu_baseline"]["value"] == j["value"]
    assert j["e2e"]["h2d_bytes_per_step"] == 0 and j["e2e"]["d2h_bytes_per_step"] == 0


def test_bench_gpus_flag_spawns_the_ranks_itself():
    """`bench.py --gpus 2` without a launcher starts two ranks itself (the
    reference arm: rank 0 prints the one line)."""
    import json
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = {k: v for k, v in os.environ.items() if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")}
    cmd = [sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--config", "toy", "--gpus", "2",
           "--steps", "1", "--warmup", "3", "--cpu-seconds", "2"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=300, cwd=root, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1 and json.loads(lines[0])["n_gpus"] == 2


def test_bench_refuses_a_world_size_other_than_gpus():
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    env = dict(os.environ, WORLD_SIZE="2", RANK="0", LOCAL_RANK="0")
    cmd = [sys.executable, os.path.join(root, "bench.py"), "--impl", "reference", "--config", "toy", "--gpus", "4"]
    r = subprocess.run(cmd, capture_output=True, text=True, timeout=120, cwd=root, env=env)
    assert r.returncode != 0 and "WORLD_SIZE" in r.stderr
