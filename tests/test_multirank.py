"""The N > 1 path on CPU: world size 2, gloo, launched like the multi-GPU bench.

The verification step shards by sequence with no collective on the data path
(replicas), so what multi-GPU adds is host logic: each rank draws its own
batch, the job's step time is the slowest rank's, and only rank 0 prints the
JSON line (for the oracle arm, only rank 0 runs at all)."""
import json
import os
import socket
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _torchrun(args, timeout):
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), *args]
    env = {**os.environ, "CUDA_VISIBLE_DEVICES": "", "OMP_NUM_THREADS": "1"}
    return subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=timeout, env=env)


def test_replicas_reduce_to_slowest_and_draw_own_batches(tmp_path):
    r = _torchrun([os.path.join("tests", "multirank_worker.py"), str(tmp_path)], timeout=300)
    assert r.returncode == 0, r.stderr[-3000:]
    ranks = [json.load(open(tmp_path / f"rank{i}.json")) for i in range(2)]
    assert [d["rank"] for d in ranks] == [0, 1] and all(d["world"] == 2 for d in ranks)
    # the job's step time is the slowest rank's (1.5 and 2.5 ms here)
    assert all(d["max"] == 2.5 for d in ranks)
    # same shapes, different inputs: each replica verifies its own batch
    assert ranks[0]["shape"] == ranks[1]["shape"]
    assert ranks[0]["qsums"] == ranks[1]["qsums"]
    assert ranks[0]["qsums"][0] != ranks[0]["qsums"][1]


def test_oracle_arm_two_ranks_prints_one_line():
    r = _torchrun(["bench.py", "--impl", "reference", "--gpus", "2", "--config", "tiny", "--steps", "1",
                   "--warmup", "0"], timeout=300)
    assert r.returncode == 0, r.stderr[-3000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
    assert len(lines) == 1, r.stdout[-2000:]
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["gpu_launches"] == 0
    assert d["value"] > 0 and d["cpu_baseline"]["kind"] == "oracle"
