"""Replicas on N > 1 ranks (host logic only, gloo on CPU, world size 2).

The verify step does not shard: `bench.py --gpus N` runs N independent
replicas and reports every rank's tokens over the slowest rank's time.  These
tests run that aggregation and the reference arm's rank split as two gloo
processes; nothing here touches a GPU.
"""
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rate_worker(rank, world, port, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    sys.path.insert(0, ROOT)
    import bench
    # Rank r processed 100 * (r + 1) tokens in 2 + r seconds.
    rate, t = bench._job_rate(100 * (rank + 1), 2.0 + rank, world, torch.device("cpu"))
    out.put((rank, rate, t))
    torch.distributed.destroy_process_group()


def test_job_rate_is_all_tokens_over_slowest_rank():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rate_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(out.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for _, rate, t in res:
        assert t == pytest.approx(3.0)             # the slowest rank's time
        assert rate == pytest.approx(300 / 3.0)    # both ranks' tokens
    assert res[0][1:] == res[1][1:]                # every rank reports the same numbers


def test_job_rate_single_rank():
    sys.path.insert(0, ROOT)
    import bench
    assert bench._job_rate(50, 2.0, 1, torch.device("cpu")) == (25.0, 2.0)


def test_reference_arm_runs_on_rank_zero_only():
    # A rank other than 0 leaves at once, prints nothing and exits 0.
    env = dict(os.environ, WORLD_SIZE="2", RANK="1", LOCAL_RANK="1", MASTER_ADDR="127.0.0.1")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                        "--steps", "1", "--warmup", "0"], cwd=ROOT, env=env, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""
