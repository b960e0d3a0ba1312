"""The multi-GPU launch of the benchmark, on CPU ranks: the path runs as independent
replicas (each rank quantizes and multiplies its own batch), so the only cross-rank steps
are the barrier and the max-over-ranks timing reduction.  Both run here as world-size-2
`gloo` process groups; the reference arm's rank > 0 exits without work."""
import json
import multiprocessing as mp
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, values, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        m = bench.max_over_ranks(values[rank], "cpu")
        out.put((rank, m))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def _run_ranks(world, values):
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, values, out))
             for r in range(world)]
    for p in procs:
        p.start()
    got = sorted(out.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return got


def test_step_time_is_the_max_over_two_gloo_ranks():
    # the slower replica decides the job's time
    got = _run_ranks(2, [12.5, 31.25])
    assert got == [(0, 31.25), (1, 31.25)]


def test_single_process_keeps_its_own_time():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(7.0, "cpu") == 7.0


def test_job_throughput_counts_every_replica():
    sys.path.insert(0, ROOT)
    import bench
    ops = 3 * 2 * 12544 * 256 * 2304
    one = bench.job_throughput(ops, 1, 10, 1.15)
    two = bench.job_throughput(ops, 2, 10, 1.15)
    assert two == pytest.approx(2 * one)
    assert one == pytest.approx(ops * 10 / 1.15e-3 / 1e12)


def test_reference_arm_rank_one_exits_quietly():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1",
               MASTER_ADDR="127.0.0.1", MASTER_PORT=str(_free_port()))
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True,
                       text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    assert r.stdout.strip() == ""


def test_reference_arm_rank_zero_prints_one_json_line():
    env = dict(os.environ)
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        env.pop(k, None)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "0"], env=env, capture_output=True,
                       text=True, timeout=600, cwd=ROOT)
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["value"] > 0 and d["n_gpus"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
