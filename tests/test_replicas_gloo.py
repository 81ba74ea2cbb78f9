"""bench.py's host logic, on the CPU.  Multi-GPU is replicas only: under
torchrun every rank runs its own copy of the workload, the step time is the
slowest rank's, and the job's throughput counts every rank's tokens; these
checks run that logic as two gloo ranks.  The reference arm (the oracle on
the host cores) is checked for its one contract line.  Nothing here touches
a GPU."""
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


def test_reference_arm_prints_one_contract_line():
    """The reference arm (the oracle on the host cores) prints one JSON line
    with the keys the bench contract names, on the small 2k-token workload."""
    res = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--config", "0",
                          "--steps", "2", "--warmup", "1"],
                         capture_output=True, text=True, timeout=300, cwd=ROOT,
                         env=dict(os.environ, RANK="0", WORLD_SIZE="1"))
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [x for x in res.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["value"] > 0 and d["higher_is_better"] is True
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["config"]["workload"] == "qwen0.5b-1L-2k"
