"""Multi-GPU is replicas only: under torchrun every rank runs its own copy of
the workload, the step time is the slowest rank's, and the job's throughput
counts every rank's tokens.  These checks run that host logic as two gloo
ranks on the CPU; nothing here touches a GPU."""
import json
import os
import socket
import subprocess
import sys

import pytest

pytest.importorskip("torch")

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_two_replicas_report_the_slowest_rank_and_all_tokens(tmp_path):
    tokens = 924672
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node=2",
           "--master-addr=127.0.0.1", f"--master-port={_free_port()}",
           os.path.join(ROOT, "tests", "replica_worker.py"), str(tokens), str(tmp_path)]
    env = dict(os.environ, OMP_NUM_THREADS="1")
    res = subprocess.run(cmd, capture_output=True, text=True, timeout=300, env=env, cwd=ROOT)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = []
    for r in range(2):
        with open(tmp_path / f"rank{r}.json") as f:
            lines.append(json.load(f))
    assert sorted(d["rank"] for d in lines) == [0, 1]
    slowest = max(d["local_ms"] for d in lines)
    for d in lines:
        assert d["world"] == 2
        assert d["ms"] == slowest
        assert d["value"] == pytest.approx(2 * tokens / (slowest * 1e-3), rel=1e-12)


def test_reference_arm_runs_on_rank_zero_only():
    """A rank other than 0 of the reference arm exits 0 without output."""
    env = dict(os.environ, RANK="1", WORLD_SIZE="2", LOCAL_RANK="1")
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2",
                          "--steps", "1", "--warmup", "0"],
                         capture_output=True, text=True, timeout=300, env=env, cwd=ROOT)
    assert res.returncode == 0, res.stderr[-2000:]
    assert res.stdout.strip() == ""
