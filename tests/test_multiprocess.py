"""The multi-process paths, on CPU with the gloo backend.

The commit path needs no data exchange between GPUs: `bench.py --gpus N` runs N independent
replicas, and the processes only meet at the barriers around the timed region and in the
maximum of their times.  These tests run that coordination with two gloo ranks, and the
reference arm (the oracle on the host cores) under torchrun with two ranks: rank 0 alone
prints the result line, and the other rank exits cleanly.
"""
import json
import os
import socket
import subprocess
import sys
from pathlib import Path

import pytest

ROOT = Path(__file__).resolve().parents[1]


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out_dir: str):
    import torch.distributed as dist
    sys.path.insert(0, str(ROOT))
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    bench.barrier(dist)
    value = bench.max_over_ranks(dist, float(10 * rank + 1))
    bench.barrier(dist)
    Path(out_dir, f"rank{rank}.txt").write_text(repr(value))
    dist.destroy_process_group()


def test_barrier_and_max_over_two_gloo_ranks(tmp_path):
    torch = pytest.importorskip("torch")
    mp = torch.multiprocessing.get_context("spawn")
    port = _free_port()
    procs = [mp.Process(target=_rank_main, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    assert [float((tmp_path / f"rank{r}.txt").read_text()) for r in range(2)] == [11.0, 11.0]


def test_reference_arm_under_torchrun_with_two_ranks():
    pytest.importorskip("torch")
    env = dict(os.environ, MASTER_ADDR="127.0.0.1", OMP_NUM_THREADS="1")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py",
           "--impl", "reference", "--gpus", "2", "--steps", "2", "--warmup", "1"]
    r = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["n_gpus"] == 2 and line["steps"] == 2
    assert line["value"] > 0 and line["cpu_baseline"]["kind"] == "oracle"


def _shard_rank_main(rank: int, world: int, port: int, out_dir: str):
    """One rank of a parameter-sharded run: it takes its shard of P from the library's
    partition and commits its slice of every gradient, with the oracle standing in for its
    GPU; the shards meet only at the end, to be compared with one process over all P."""
    import numpy as np
    import torch
    import torch.distributed as dist
    sys.path.insert(0, str(ROOT))
    import oracle
    from paper_1805_08469_gb300 import gem
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    P, n, T = 10_007, 5, 120
    rng = np.random.default_rng(5)
    theta0 = (0.05 * rng.standard_normal(P)).astype(np.float32)
    grads = (0.1 * rng.standard_normal((T, P))).astype(np.float32)
    order, _ = oracle.schedule_uniform(9, n, T)
    b, e = gem.gem_shard_range(P, world, rank)
    th = theta0[b:e].copy()
    m = np.zeros((n, e - b), np.float32)
    s = np.tile(th, (n, 1))
    oracle.gem_run(th, m, s, np.ascontiguousarray(grads[:, b:e]), order, eta=0.01, mu=0.9, eps=1e-8)
    # gather the shards (padded to the largest) on every rank
    width = max(gem.gem_shard_range(P, world, r)[1] - gem.gem_shard_range(P, world, r)[0]
                for r in range(world))
    mine = torch.zeros((1 + 2 * n, width))
    mine[0, :e - b] = torch.from_numpy(th)
    mine[1:1 + n, :e - b] = torch.from_numpy(m)
    mine[1 + n:, :e - b] = torch.from_numpy(s)
    parts = [torch.zeros_like(mine) for _ in range(world)]
    dist.all_gather(parts, mine)
    if rank == 0:
        th_f, m_f, s_f = theta0.copy(), np.zeros((n, P), np.float32), np.tile(theta0, (n, 1))
        oracle.gem_run(th_f, m_f, s_f, grads, order, eta=0.01, mu=0.9, eps=1e-8)
        got = np.concatenate([parts[r].numpy()[:, :gem.gem_shard_range(P, world, r)[1]
                                              - gem.gem_shard_range(P, world, r)[0]]
                              for r in range(world)], axis=1)
        ok = (np.array_equal(got[0], th_f) and np.array_equal(got[1:1 + n], m_f)
              and np.array_equal(got[1 + n:], s_f))
        Path(out_dir, "shards.txt").write_text("equal" if ok else "differ")
    dist.destroy_process_group()


def test_parameter_shards_over_two_gloo_ranks(tmp_path):
    """Two ranks each commit their contiguous shard of P (from gem_shard_range) with no
    exchange during the run; their gathered theta, m and s equal one process over all P bit
    for bit.  The oracle is each rank's compute here (there is one GPU in this setting); the
    CUDA path on shards is checked against one handle in tests/test_gpu_shards.py."""
    torch = pytest.importorskip("torch")
    mp = torch.multiprocessing.get_context("spawn")
    port = _free_port()
    procs = [mp.Process(target=_shard_rank_main, args=(r, 2, port, str(tmp_path))) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    assert (tmp_path / "shards.txt").read_text() == "equal"
