"""The multi-process path of bench.py on CPU: world size 2 over gloo.

With N GPUs the benchmark runs N independent replicas of the layer (the path
has no exchange step on one GPU's worth of experts), so the only cross-rank
logic is the timing aggregation: a barrier around the timed region, the
slowest rank's time (max) and the total tokens (sum).  The reference arm
runs on rank 0 only; other ranks exit without work or output.
"""
import json
import os
import socket
import subprocess
import sys
import time

import pytest
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import torch
    import bench
    r, w, _ = bench.dist_env()
    bench.init_dist(w, "gloo")
    bench.barrier(w)
    mx = bench.reduce_max(10.0 + 5.0 * r, w)
    sm = bench.reduce_sum(32.0 * (r + 1), w)
    bench.barrier(w)
    q.put((r, mx, sm))
    torch.distributed.destroy_process_group()


def test_timing_aggregation_over_two_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get(timeout=5) for _ in range(2))
    for r, mx, sm in res:
        assert mx == 15.0          # the slowest rank's time
        assert sm == 32.0 + 64.0   # tokens of all ranks


def test_single_rank_reductions_are_identity():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.reduce_max(3.5, 1) == 3.5
    assert bench.reduce_sum(7.0, 1) == 7.0


@pytest.mark.parametrize("rank", [0, 1])
def test_reference_arm_runs_on_rank_zero_only(rank):
    env = dict(os.environ, RANK=str(rank), WORLD_SIZE="2", LOCAL_RANK=str(rank),
               MASTER_ADDR="127.0.0.1", MASTER_PORT=str(_free_port()))
    t0 = time.perf_counter()
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", "tiny", "--steps", "3", "--warmup", "3"],
                       env=env, capture_output=True, text=True, timeout=300, cwd=ROOT)
    wall_s = time.perf_counter() - t0
    assert r.returncode == 0, r.stderr
    lines = [l for l in r.stdout.splitlines() if l.strip()]
    if rank == 0:
        d = json.loads(lines[-1])
        assert d["impl"] == "reference" and d["value"] > 0 and d["n_gpus"] == 2
        assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
        assert d["e2e"]["h2d_bytes_per_step"] == 0
        # Whole layer steps, measured: the K timed steps fit inside the run, and
        # the rate is the batch over the measured mean step time.
        assert "full layer steps" in d["cpu_baseline"]["sample"]
        assert d["steps"] == 3 and d["ms_per_step"] * d["steps"] * 1e-3 < wall_s
        assert abs(d["value"] - 32 / (d["ms_per_step"] * 1e-3)) < 1e-6 * d["value"]
        # The same config object as the GPU arm's line.
        sys.path.insert(0, ROOT)
        import bench
        from paper_2602_07265_gb300 import workloads as W
        assert d["config"] == json.loads(json.dumps(bench.workload_config(W.TINY, 0, 2)))
    else:
        assert lines == []
