"""The N > 1 path of bench.py runs N independent replicas (weak scaling, no
data-path collective): each rank times its own steps, the ranks meet at a
barrier on both sides of the timed region, the time is the maximum over
ranks, and the value counts the tokens of all ranks.  Two gloo ranks on the
CPU run bench.py's own rendezvous, barrier and max-over-ranks code; the
reference arm leaves all of its work to rank 0."""
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

RANK_SCRIPT = r"""
import os, sys
sys.path.insert(0, os.getcwd())
import bench
dist, rank, world, local = bench.dist_setup(2)
bench.barrier(dist)
m = bench.max_over_ranks(dist, 10.0 + 5.0 * rank)
bench.barrier(dist)
print("RESULT", rank, world, m, flush=True)
dist.destroy_process_group()
"""

REFERENCE_SCRIPT = r"""
import os, sys, argparse
sys.path.insert(0, os.getcwd())
import bench
if int(os.environ["RANK"]) == 1:
    class Refuse:
        def __init__(self, *a, **k):
            raise RuntimeError("rank 1 must not run the oracle")
    bench.OracleSample = Refuse
    bench.run_reference(argparse.Namespace(gpus=2, workload="tiny", steps=1, warmup=3))
    print("RANK1_DONE", flush=True)
else:
    dist, rank, world, local = bench.dist_setup(2)
    print("RANK0_JOINED", flush=True)
"""


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _run_two(script: str):
    port = _free_port()
    procs = []
    for rank in range(2):
        env = dict(os.environ, MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE="2",
                   LOCAL_RANK=str(rank), CUDA_VISIBLE_DEVICES="")
        procs.append(subprocess.Popen([sys.executable, "-c", script], cwd=ROOT, env=env, stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True))
    outs = []
    try:
        for p in procs:
            out, err = p.communicate(timeout=120)
            assert p.returncode == 0, err[-2000:]
            outs.append(out)
    finally:
        for p in procs:
            if p.poll() is None:
                p.kill()
    return outs


def test_two_gloo_ranks_meet_and_take_the_max_time():
    outs = _run_two(RANK_SCRIPT)
    res = sorted(tuple(line.split()[1:]) for out in outs for line in out.splitlines() if line.startswith("RESULT"))
    assert [(int(r), int(w), float(m)) for r, w, m in res] == [(0, 2, 15.0), (1, 2, 15.0)]


def test_reference_arm_runs_on_rank_zero_only():
    outs = _run_two(REFERENCE_SCRIPT)
    assert "RANK0_JOINED" in outs[0] and "RANK1_DONE" in outs[1]


def test_job_value_counts_every_rank_over_the_slowest_time():
    sys.path.insert(0, ROOT)
    import bench
    # 2 ranks x 10 steps x 8192 tokens in 600 ms (the slower rank)
    assert bench.job_value(2, 10, 8192, 600.0) == pytest.approx(2 * 10 * 8192 / 0.6)
    assert bench.job_value(1, 10, 8192, 600.0) == pytest.approx(10 * 8192 / 0.6)
