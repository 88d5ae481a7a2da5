"""The benchmark's multi-rank path on CPU: two gloo ranks go through the
same set-up, barrier, max-over-ranks timing and whole-job rate that
`bench.py --gpus N` uses under torchrun (independent replicas, no data-path
collective), and the reference arm prints from rank 0 only."""
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


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      LOCAL_RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist
    w, r, local = bench.dist_setup(world)
    try:
        bench.barrier(w)
        # rank r "took" 100 (r + 1) ms for 10 steps
        ms = 100.0 * (r + 1)
        q.put((r, w, local, dist.get_backend(), bench.max_over_ranks(ms, w),
               bench.job_rate(10, ms, w)))
        bench.barrier(w)
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_time_like_the_bench():
    world, port = 2, _free_port()
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    procs = [ctx.Process(target=_worker, args=(r, world, port, q)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
    assert all(p.exitcode == 0 for p in procs), [p.exitcode for p in procs]
    got = sorted(q.get(timeout=5) for _ in range(world))
    for r, (rank, w, local, backend, ms_max, rate) in enumerate(got):
        assert (rank, w, local, backend) == (r, world, r, "gloo")
        # the slowest rank sets the time; the rate counts both ranks' steps
        assert ms_max == 200.0
        assert rate == pytest.approx(10 * world / 0.2)


def test_world_size_must_match_gpus():
    sys.path.insert(0, ROOT)
    import bench
    env = dict(os.environ)
    os.environ.pop("WORLD_SIZE", None)
    try:
        with pytest.raises(SystemExit):
            bench.dist_setup(2)
        assert bench.dist_setup(1) == (1, 0, 0)
        assert bench.job_rate(20, 400.0, 1) == pytest.approx(50.0)
    finally:
        os.environ.clear()
        os.environ.update(env)


def test_reference_arm_prints_from_rank_zero_only():
    """torchrun with two gloo ranks: rank 0 times the oracle and prints one
    JSON line, rank 1 exits 0 without work."""
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--gpus", "2",
           "--impl", "reference", "--steps", "1", "--warmup", "0"]
    out = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600)
    assert out.returncode == 0, out.stderr[-2000:]
    lines = [ln for ln in out.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, out.stdout
    j = json.loads(lines[0])
    assert j["impl"] == "reference" and j["n_gpus"] == 2 and j["value"] > 0
    assert j["cpu_baseline"]["kind"] == "oracle"
    assert j["e2e"]["h2d_bytes_per_step"] == 0
