"""The benchmark's N > 1 path on CPU: two gloo ranks run the host logic that
bench.py runs between NCCL ranks (max-over-ranks timing, whole-job value,
per-rank input seeds, rank-0-only reference arm)."""
import json
import os
import socket
import subprocess
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank: int, world: int, port: int, out_dir: str):
    import torch
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    from paper_2608_03228_gb300 import synth
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # the slowest rank's time decides; every rank sees it
        ms = bench.max_over_ranks(10.0 + 3.0 * rank, dist, "cpu")
        value = bench.job_value(1000.0, world, ms)
        # replicas draw different inputs (seed offset = rank), reproducibly
        w = synth.WORKLOADS["tiny_f32_t512"]
        q = synth.make_torch(w, "cpu", seed_offset=rank)["Q"]
        q2 = synth.make_torch(w, "cpu", seed_offset=rank)["Q"]
        same = bool(torch.equal(q, q2))
        sums = [torch.zeros(1, dtype=torch.float64) for _ in range(world)]
        dist.all_gather(sums, q.double().sum().reshape(1))
        with open(os.path.join(out_dir, f"r{rank}.json"), "w") as f:
            json.dump({"ms": ms, "value": value, "same": same, "sums": [float(s) for s in sums]}, f)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    procs = [ctx.Process(target=_worker, args=(r, world, port, str(tmp_path))) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
        assert p.exitcode == 0
    res = [json.load(open(tmp_path / f"r{r}.json")) for r in range(world)]
    for r in res:
        assert r["ms"] == pytest.approx(13.0)                       # max over ranks
        assert r["value"] == pytest.approx(1000.0 * 2 / 0.013)      # units of both ranks in the slowest time
        assert r["same"]
    assert res[0]["sums"] == res[1]["sums"]
    assert res[0]["sums"][0] != res[0]["sums"][1]                   # each replica has its own inputs


def test_reference_arm_prints_on_rank_zero_only():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                          "tiny_f32_t512", "--steps", "1", "--warmup", "0"], env=env, capture_output=True,
                         text=True, timeout=600)
    assert out.returncode == 0, out.stderr
    assert out.stdout.strip() == ""


def test_reference_arm_line_on_rank_zero():
    env = dict(os.environ, RANK="0", WORLD_SIZE="1", LOCAL_RANK="0")
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload",
                          "tiny_f32_t512", "--steps", "1", "--warmup", "0"], env=env, capture_output=True,
                         text=True, timeout=600)
    assert out.returncode == 0, out.stderr
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["value"] > 0
    assert line["cpu_baseline"]["kind"] == "oracle"
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
