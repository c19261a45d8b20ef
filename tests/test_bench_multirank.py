"""The multi-process side of bench.py on CPU (gloo, world size 2): one replica per rank, the step
time taken as the maximum over ranks, the whole-job value summing every rank's work (weak
scaling), and the reference arm printing one line from rank 0 only.  No GPU is used."""

import json
import multiprocessing as mp
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, times, out):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank)})
    sys.path.insert(0, ROOT)
    import torch
    import torch.distributed as dist

    import bench

    w, r, local = bench.dist_init()
    assert (w, r, local) == (world, rank, rank)
    bench.barrier(w)
    ms = bench.max_over_ranks(w, times[rank], torch.device("cpu"))
    value = bench.job_value(w, bench.OPS_STEP, 10, ms)
    out.put((rank, ms, value))
    dist.destroy_process_group()


def test_max_over_ranks_and_weak_scaling_value():
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    port = _free_port()
    times = [3.0, 5.0]  # rank 1 is the slower one
    procs = [ctx.Process(target=_rank_main, args=(r, 2, port, times, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    got = sorted(out.get(timeout=10) for _ in range(2))
    for rank, ms, value in got:
        assert ms == 5.0  # every rank reports the slowest rank's time
        assert value == pytest.approx(2 * 164.3e9 * 10 / 5e-3 / 1e12, rel=1e-3)


def test_reference_arm_under_torchrun_prints_once_from_rank_zero():
    port = _free_port()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port), "bench.py", "--impl", "reference",
           "--gpus", "2", "--steps", "1", "--warmup", "1"]
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["steps"] == 1
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_clock_record_prefers_samples_inside_the_timed_region():
    sys.path.insert(0, ROOT)
    import bench

    rows = [(1900.0, 2070.0, 900.0, ["sw_power_cap"], False)] * 5 + [(2070.0, 2070.0, 800.0, [], True)] * 3
    c = bench.ClockSampler.summarize(rows, "test")
    assert c["sm_mhz"] == 2070.0 and c["samples_in_timed_region"] == 3 and c["reasons"] == []
    assert c["window"] == "the timed region"
    # fewer than three samples inside: the bracketing window, with its reasons
    c = bench.ClockSampler.summarize(rows[:6], "test")
    assert c["sm_mhz"] == 1900.0 and c["reasons"] == ["sw_power_cap"] and c["samples"] == 6
    assert bench.ClockSampler.summarize([], "test") is None
