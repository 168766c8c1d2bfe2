"""The bench's reference arm (the fp64 oracle timed on the host cores) keeps
the bench contract on the CPU: one JSON line with the same metric and unit as
the GPU arm, a cpu_baseline describing the run, an e2e block with no copies;
under torchrun with two ranks, rank 0 alone prints and both ranks exit 0."""
import json
import os
import socket
import subprocess
import sys


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _lines(out):
    return [json.loads(x) for x in out.splitlines() if x.strip().startswith("{")]


def _check(line, n_gpus):
    assert line["impl"] == "reference"
    assert line["unit"] == "µs/layer" and line["higher_is_better"] is False
    assert line["n_gpus"] == n_gpus and line["steps"] == 2 and line["warmup"] == 1
    assert line["value"] > 0 and line["dtype"] == "f64" and line["data"] == "synthetic"
    assert line["config"]["workload"].startswith("tiny:")
    cpu = line["cpu_baseline"]
    assert cpu["kind"] == "oracle" and cpu["cores"] >= 1 and cpu["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"],
                           "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_one_process(repo_root):
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--config", "tiny",
                        "--steps", "2", "--warmup", "1"], cwd=repo_root, capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = _lines(r.stdout)
    assert len(lines) == 1
    _check(lines[0], 1)


def test_reference_arm_two_ranks_under_torchrun(repo_root):
    env = dict(os.environ, MASTER_ADDR="127.0.0.1")
    r = subprocess.run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1",
                        "--nproc-per-node", "2", "--master-addr", "127.0.0.1",
                        "--master-port", str(_free_port()), "bench.py", "--impl", "reference",
                        "--gpus", "2", "--config", "tiny", "--steps", "2", "--warmup", "1"],
                       cwd=repo_root, capture_output=True, text=True, timeout=300, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = _lines(r.stdout)
    assert len(lines) == 1
    _check(lines[0], 2)
