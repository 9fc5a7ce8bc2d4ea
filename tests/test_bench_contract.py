"""The benchmark's JSON line, through its CPU-only reference arm (the oracle on bounded samples).

One JSON line with the contract's keys; under torchrun with two ranks, rank 0 alone
prints it and both ranks exit 0.
"""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
KEYS = {"metric", "impl", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better",
        "scaling", "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"}


def _run(cmd, env_extra=None):
    env = dict(os.environ, **(env_extra or {}))
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=600, env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    return [json.loads(l) for l in r.stdout.splitlines() if l.startswith("{")]


def _check(line, steps, warmup, n_gpus):
    assert KEYS <= set(line), KEYS - set(line)
    assert line["impl"] == "reference"
    assert (line["steps"], line["warmup"], line["n_gpus"]) == (steps, warmup, n_gpus)
    assert line["value"] > 0 and line["ms_per_step"] > 0 and line["higher_is_better"] is True
    assert line["unit"] == line["cpu_baseline"]["unit"] == line["e2e"]["unit"] == "tokens/s"
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"]["value"] == line["value"]
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["e2e"]["d2h_bytes_per_step"] == 0
    assert line["vs_baseline"] is None and line["data"] == "synthetic"
    assert "workload" in line["config"] and "sample" in line["config"]


@pytest.mark.parametrize("workload", ["lm1p3b", "decode"])
def test_reference_arm_prints_one_contract_line(workload):
    lines = _run([sys.executable, "bench.py", "--impl", "reference", "--workload", workload, "--steps", "3",
                  "--warmup", "3", "--reference-tokens", "128"])
    assert len(lines) == 1
    _check(lines[0], 3, 3, 1)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_reference_arm_under_torchrun_prints_on_rank_zero_only():
    lines = _run([sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
                  "--master-addr", "127.0.0.1", "--master-port", str(_free_port()), "bench.py", "--gpus", "2", "--impl",
                  "reference", "--steps", "3", "--warmup", "3", "--reference-tokens", "128"],
                 {"OMP_NUM_THREADS": "1"})
    assert len(lines) == 1
    _check(lines[0], 3, 3, 2)
