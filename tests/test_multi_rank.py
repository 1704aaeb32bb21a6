"""The bench's multi-process path on CPU: replicas on every rank (weak
scaling), the job's time the slowest rank's (max over ranks through
torch.distributed, here with gloo and two ranks), throughput counted over
all ranks, and a reference arm that only rank 0 runs."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, values, out):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        m = bench.max_over_ranks(values[rank], world)
        out[rank] = (m, bench.job_throughput(m, world))
    finally:
        dist.destroy_process_group()


def test_max_over_ranks_and_throughput_with_two_gloo_ranks():
    world, port = 2, _free_port()
    values = [0.51, 0.53]  # ms per step on each rank
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_rank_main, args=(world, port, values, out), nprocs=world, join=True)
        got = dict(out)
    for rank in range(world):
        m, thr = got[rank]
        assert m == pytest.approx(0.53)                  # the slowest rank's time
        assert thr == pytest.approx(2 * 1e3 / 0.53)      # both ranks' steps in that time


def test_max_over_ranks_single_process_is_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(0.7, 1) == 0.7
    assert bench.job_throughput(0.5, 1) == pytest.approx(2000.0)


def _run_bench(env_extra, *args):
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="", **env_extra)
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], capture_output=True, text=True,
                          env=env, timeout=600, cwd=ROOT)


def test_reference_arm_only_rank_zero_works():
    r = _run_bench(dict(RANK="1", WORLD_SIZE="2"), "--impl", "reference", "--workload", "c1", "--steps", "1",
                   "--warmup", "3")
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_reference_arm_prints_one_line():
    r = _run_bench(dict(RANK="0", WORLD_SIZE="1"), "--impl", "reference", "--workload", "c1", "--steps", "1",
                   "--warmup", "3")
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["unit"] == "steps/s" and d["value"] > 0
    assert d["cpu_baseline"]["kind"] == "oracle" and d["e2e"]["h2d_bytes_per_step"] == 0
