"""The N > 1 path of bench.py on CPU: two ranks under torch.distributed.run with gloo.

The GPU path is replicas only (one independent step per rank, no data-path collective);
what the ranks share is the barrier around the timed region, the maximum of the ranks'
times and the whole-job rate, checked here, plus the reference arm's rule that rank 0
alone runs and prints."""

import json
import os
import socket
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _torchrun(args, timeout=600, env_extra=None):
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(_free_port())] + args
    env = dict(os.environ, OMP_NUM_THREADS="1", CUDA_VISIBLE_DEVICES="", **(env_extra or {}))
    return subprocess.run(cmd, capture_output=True, text=True, timeout=timeout, cwd=ROOT, env=env)


def test_two_gloo_ranks_agree_on_the_slowest_time_and_the_job_rate(tmp_path):
    out = _torchrun([os.path.join(ROOT, "tests", "dist_worker.py")], env_extra={"OPD_TEST_OUT": str(tmp_path)})
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [json.loads((tmp_path / f"rank{r}.json").read_text()) for r in range(2)]
    assert sorted(d["rank"] for d in lines) == [0, 1]
    for d in lines:
        assert d["world"] == 2
        assert d["max_ms"] == 110.0  # the slower rank's time, on every rank
        assert abs(d["rate"] - 1000 * 5 * 2 / 0.110) < 1e-6  # units of both ranks over that time


def test_reference_arm_under_two_ranks_prints_once_from_rank_zero():
    out = _torchrun([os.path.join(ROOT, "bench.py"), "--impl", "reference", "--gpus", "2", "--workload",
                     "tiny_fp32", "--steps", "2", "--warmup", "3", "--ref-rows", "4"])
    assert out.returncode == 0, out.stderr[-3000:]
    lines = [json.loads(l) for l in out.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = lines[0]
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
