"""The multi-GPU path of bench.py is replicas only: each rank runs the whole
workload on its own GPU, the job's time is the slowest rank's (an all-reduce
of the timings) and its value is the sum over the replicas.  Here that host
logic runs as two gloo ranks on the CPU, and a non-zero rank of the oracle
reference arm exits without output."""
import json
import os
import socket
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

RANK_CODE = """
import json, os, sys
sys.path.insert(0, {root!r})
import torch.distributed as dist
import bench
dist.init_process_group("gloo", init_method="env://")
ws, rank, _ = bench._dist()
ms = bench.max_over_ranks(10.0 + 5.0 * rank, ws, "cpu")
# per timed window, the slower rank's duration
win = bench.window_max_over_ranks([1.0 + rank, 3.0 - rank, 2.0], ws, "cpu")
print(json.dumps({{"rank": rank, "ms": ms, "tbs": bench.job_tbs(ws, 1000000, 20, ms),
                  "win": win}}))
dist.destroy_process_group()
"""


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_take_the_slowest_time_and_sum_the_replicas():
    port = _free_port()
    procs = []
    for rank in range(2):
        env = dict(os.environ, RANK=str(rank), LOCAL_RANK=str(rank), WORLD_SIZE="2",
                   MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
        procs.append(subprocess.Popen([sys.executable, "-c", RANK_CODE.format(root=ROOT)],
                                      env=env, stdout=subprocess.PIPE, stderr=subprocess.PIPE,
                                      text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=180)
        assert p.returncode == 0, err[-2000:]
        outs.append(json.loads(out.strip().splitlines()[-1]))
    for o in outs:
        assert o["ms"] == 15.0  # the slower rank's 15 ms, on every rank
        assert o["win"] == [2.0, 3.0, 2.0]
        # two replicas of 1 MB per step, 20 steps in 15 ms
        assert abs(o["tbs"] - 2 * 1e6 * 20 / 15e-3 / 1e12) < 1e-12


def test_reference_arm_rank_one_exits_without_output():
    env = dict(os.environ, RANK="1", LOCAL_RANK="1", WORLD_SIZE="2")
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--steps", "1", "--warmup", "3"], env=env, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks(12.5, 1) == 12.5
    assert bench.window_max_over_ranks([1.0, 2.0], 1) == [1.0, 2.0]
    assert bench.job_tbs(1, 142208000, 10, 0.5) == 142208000 * 10 / 0.5e-3 / 1e12
