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


def test_fractions_carry_the_nominal_rate_beside_the_measured_copy():
    """Every record with GB/s and `frac` also gets `frac_nominal` (GB/s over the
    nominal 8000 GB/s), in nested records and lists; other fields are left alone."""
    line = {"roofline": {"achieved": 5780.0, "frac": 0.8537},
            "lag_pass": {"gbs": 2816.0, "frac": 0.416},
            "configs": [{"frontier": {"gbs": 6400.0, "frac": 0.945}, "aggregate": {"gbs": 4000.0, "frac": 0.59}}],
            "e2e": {"h2d_gbs": 150.0, "frac_of_link": 1.0}}
    out = bench.add_nominal(line, 6770.5, "measured")
    assert out["roofline"]["frac_nominal"] == round(5780.0 / 8000.0, 4)
    assert out["lag_pass"]["frac_nominal"] == round(2816.0 / 8000.0, 4)
    assert out["configs"][0]["frontier"]["frac_nominal"] == 0.8
    assert out["configs"][0]["aggregate"]["frac_nominal"] == 0.5
    assert "frac_nominal" not in out["e2e"]
    rec = bench.peaks_record(6770.5, "measured")
    assert "6770.5" in rec["frac"] and "8000" in rec["frac_nominal"]
