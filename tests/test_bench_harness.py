"""bench.py's multi-rank harness and reference arm on the CPU (gloo, world size 2)."""
import json
import os
import socket
import subprocess
import sys

import pytest
import torch
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, ws, port, q):
    os.environ.update({"MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port), "RANK": str(rank),
                       "WORLD_SIZE": str(ws), "LOCAL_RANK": str(rank)})
    bench.init_dist("gloo")
    import time
    calls = []

    def step():
        calls.append(1)
        time.sleep(0.01 * (rank + 1))   # rank 1 is the slow replica

    secs = bench.timed_loop(step, K=5, W=3, ws=ws, device="cpu", use_cuda=False)
    q.put((rank, secs, len(calls)))
    torch.distributed.destroy_process_group()


def test_timed_loop_takes_max_over_ranks():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    res = sorted(q.get() for _ in range(2))
    assert res[0][2] == res[1][2] == 8                 # 3 warm-up + 5 timed on every rank
    assert abs(res[0][1] - res[1][1]) < 1e-9           # both ranks report the same (max) time
    assert res[0][1] >= 5 * 0.02                       # the slow rank bounds it


def test_reference_arm_line():
    out = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                          "--steps", "2", "--warmup", "3", "--workload", "ddp128", "--steps-override",
                          "2000"],
                         capture_output=True, text=True, timeout=600, cwd=ROOT)
    assert out.returncode == 0, out.stderr
    line = json.loads(out.stdout.strip().splitlines()[-1])
    assert line["impl"] == "reference" and line["unit"] == "records/s" and line["value"] > 0
    # whole 1000-step windows, one per host thread: the two windows of 2000 steps
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["cores"] == min(os.cpu_count(), 2)
    assert line["config"]["W"] == 1000 and line["config"]["T"] == 2000
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["value"] == line["value"]
    assert line["higher_is_better"] is True and line["steps"] == 2


def test_reference_arm_other_ranks_exit_quietly(monkeypatch):
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")
    args = bench.argparse.Namespace(workload="tiny", seed=0, steps_override=None,
                                    warmup=3, steps=1)
    assert bench.run_reference(args) is None
