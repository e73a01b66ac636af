"""The N > 1 path of bench.py on CPU: two processes launched like torchrun (RANK, WORLD_SIZE,
LOCAL_RANK, MASTER_ADDR = 127.0.0.1, MASTER_PORT in the environment) over gloo.  The mixer
shards over the batch with no exchange (replicas only), so what there is to test is the host
logic: the rank environment, the MAX over ranks of the timed region, the whole-job value and the
reference arm, which only rank 0 runs."""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
WORKER = os.path.join(ROOT, "tests", "_multirank_worker.py")


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_gloo_ranks_agree_on_the_slowest_time_and_the_job_value():
    port = free_port()
    procs = []
    for rank in range(2):
        env = dict(os.environ, RANK=str(rank), WORLD_SIZE="2", LOCAL_RANK=str(rank), MASTER_ADDR="127.0.0.1",
                   MASTER_PORT=str(port), CUDA_VISIBLE_DEVICES="")
        procs.append(subprocess.Popen([sys.executable, WORKER], env=env, stdout=subprocess.PIPE,
                                      stderr=subprocess.PIPE, text=True))
    outs = []
    for p in procs:
        out, err = p.communicate(timeout=300)
        assert p.returncode == 0, err[-2000:]
        outs.append(json.loads(out.strip().splitlines()[-1]))
    outs.sort(key=lambda d: d["rank"])
    assert [d["rank"] for d in outs] == [0, 1] and all(d["world"] == 2 for d in outs)
    assert [d["local"] for d in outs] == [0, 1]
    for d in outs:
        assert d["elapsed"] == 15.0                      # the slower rank's 15 ms
        assert d["value"] == pytest.approx(2 * 65536 * 100 / 0.015)


def test_single_process_defaults_and_reference_arm_on_other_ranks(monkeypatch, capsys):
    sys.path.insert(0, ROOT)
    import bench
    from paper_2607_25234_gb300 import inputs
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench.dist_env() == (1, 0, 0)
    assert bench.max_over_ranks(3.5, 1, None) == 3.5
    # under torchrun only rank 0 times the oracle and prints; the others return without work
    monkeypatch.setenv("WORLD_SIZE", "2")
    monkeypatch.setenv("RANK", "1")

    class Args:
        steps, warmup, gpus = 1, 1, 2
    assert bench.reference_arm(Args(), inputs.WORKLOADS["tiny_1x256x64_f32"]) is None
    assert capsys.readouterr().out == ""
