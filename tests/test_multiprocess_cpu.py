"""The multi-rank bench logic on CPU: two gloo ranks (one per process, as torchrun launches them).

bench.py runs one independent replica per GPU; its only cross-rank logic is the barrier-bracketed
timing, reduced to the slowest rank, and the whole-job throughput.  The reference arm runs on
rank 0 alone.  Those pieces run here over gloo on 127.0.0.1."""
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


def _rank(rank, world, port, out):
    import torch.distributed as dist

    sys.path.insert(0, ROOT)
    import bench

    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                      MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, wsz, lr = bench.dist_env()
        assert (r, wsz, lr) == (rank, world, rank)
        dist.barrier()
        slowest = bench.max_over_ranks(0.5 + rank, world)  # rank 1 is the slow one
        out.put((rank, slowest, bench.job_throughput(16, 100, slowest, world)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_report_the_slowest_time_and_job_throughput():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    got = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [g[1] for g in got] == [1.5, 1.5]                      # both ranks see the max
    assert got[0][2] == pytest.approx(2 * 16 * 100 / 1.5)          # all ranks' tokens / slowest time


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench

    assert bench.max_over_ranks(0.25, 1) == 0.25
    assert bench.job_throughput(16, 10, 2.0, 1) == 80.0


def test_reference_arm_runs_on_rank_0_only():
    # a rank other than 0 exits at once without work and prints nothing
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "0"], env=env, capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert res.returncode == 0, res.stderr
    assert res.stdout.strip() == ""


def test_reference_arm_prints_the_contract_line():
    # rank 0 alone (no torchrun): the fp64 oracle timed on the host cores, one JSON line with the same
    # metric, unit and config as the CUDA arm, the cpu_baseline describing this run, and an e2e of its own
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--steps", "1",
                          "--warmup", "0"], capture_output=True, text=True, timeout=600, cwd=ROOT,
                         env={k: v for k, v in os.environ.items() if k not in ("RANK", "WORLD_SIZE", "LOCAL_RANK")})
    assert res.returncode == 0, res.stderr
    lines = [ln for ln in res.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    import bench

    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == "tokens/s"
    assert d["higher_is_better"] is True and d["n_gpus"] == 1 and d["steps"] == 1 and d["value"] > 0
    assert d["config"] == bench.headline_config(1) and d["config"]["workload"].startswith("long_context")
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
