"""The N > 1 replica path on CPU (gloo, world size 2).

The hot path does not shard: every rank runs the whole step on its own GPU
and the ranks meet only to agree on the job's time (maximum over ranks).
These tests run that host logic with the gloo backend, the replicas' host
half (fit + integer allocation through librq) on every rank, and the
reference arm launched by torchrun (rank 0 alone prints the line).
"""
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


def _init(rank, world, port):
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    return dist


def _timing_worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import bench
    dist = _init(rank, world, port)
    try:
        ms = bench.max_over_ranks(10.0 + 5.0 * rank, world, "cpu")
        gbs = bench.job_gbs(world, 3e9, ms)
        q.put((rank, ms, gbs))
    finally:
        dist.destroy_process_group()


def _alloc_worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    import torch
    from paper_2605_06675_gb300 import rq
    dist = _init(rank, world, port)
    try:
        rng = np.random.default_rng(7)                  # the same calibration on every replica
        n = 64
        mse = rng.uniform(0.5, 20, n)[:, None] * rng.uniform(3.5, 6.0, n)[:, None] ** (
            -np.arange(1, 9)[None, :])
        w = np.exp(rng.normal(0, 0.74, n))
        a, b, _ = rq.rq_fit_distortion(mse, 2, 6, 0.96, np.arange(n) % 2)
        bits, _ = rq.rq_alloc(w, a, b, 2.5, (1 << 2) | (1 << 3) | (1 << 4))
        t = torch.tensor(np.asarray(bits, dtype=np.int64))
        got = [torch.empty_like(t) for _ in range(world)]
        dist.all_gather(got, t)
        q.put((rank, [g.tolist() for g in got]))
    finally:
        dist.destroy_process_group()


def _run(worker, world=2):
    import torch.multiprocessing as mp
    ctx = mp.get_context("spawn")
    q = ctx.SimpleQueue()
    port = _free_port()
    procs = [ctx.Process(target=worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
    codes = [p.exitcode for p in procs]
    for p in procs:
        if p.is_alive():
            p.kill()
    assert codes == [0] * world, codes
    return sorted(q.get() for _ in range(world))


def test_job_time_is_the_slowest_rank():
    res = _run(_timing_worker)
    assert [r[1] for r in res] == [15.0, 15.0]
    # 2 ranks x 3 GB in 15 ms
    assert all(abs(r[2] - 400.0) < 1e-9 for r in res)


def test_replicas_allocate_identically():
    from paper_2605_06675_gb300 import build
    if not os.path.exists(build.LIB):
        build.build()
    res = _run(_alloc_worker)
    a, b = res[0][1], res[1][1]
    assert a == b and a[0] == a[1]
    assert abs(np.mean(a[0]) - 2.5) < 1e-9


def test_reference_arm_under_torchrun_prints_one_line():
    env = dict(os.environ)
    env["CUDA_VISIBLE_DEVICES"] = ""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()),
           os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
           "--workload", "tiny_1L_S1024_fp16", "--steps", "1", "--warmup", "0"]
    r = subprocess.run(cmd, capture_output=True, text=True, env=env, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"
