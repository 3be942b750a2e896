"""The reference arm of bench.py (the fp64 oracle on the host cores) prints the benchmark's JSON line on rank 0
and nothing on the other ranks. CPU only, on the 4,096-entry workload."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CMD = [sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference", "--workload", "tiny-4k", "--steps", "2",
       "--warmup", "1"]


def _run(**env):
    run = subprocess.run(CMD, cwd=ROOT, env=dict(os.environ, **env), capture_output=True, text=True, timeout=600)
    assert run.returncode == 0, run.stderr[-2000:]
    return [line for line in run.stdout.splitlines() if line.startswith("{")]


def test_reference_arm_prints_one_complete_line():
    lines = _run()
    assert len(lines) == 1
    line = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
                "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in line, key
    assert line["impl"] == "reference" and line["unit"] == "queries/s" and line["higher_is_better"] is True
    assert line["steps"] == 2 and line["warmup"] == 1 and line["value"] > 0 and line["ms_per_step"] > 0
    assert line["config"]["workload"] == "tiny-4k" and line["config"]["entries"] == 4096
    cb = line["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == line["value"] and cb["cores"] >= 1 and cb["sample"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    # every step looks up the whole 64-query batch: the value follows from the timed steps
    assert abs(line["value"] - 64 / (line["ms_per_step"] / 1e3)) <= 1e-6 * line["value"]


def test_reference_arm_runs_on_rank_zero_only():
    assert _run(RANK="1", LOCAL_RANK="1", WORLD_SIZE="2") == []


def test_gpus_flag_starts_one_rank_per_gpu():
    """Without torchrun, --gpus N starts the N ranks itself (torch.distributed.run on this node): every rank sees
    WORLD_SIZE = N, and only rank 0 prints, with n_gpus = N."""
    env = {k: v for k, v in os.environ.items()
           if k not in ("RANK", "LOCAL_RANK", "WORLD_SIZE", "MASTER_ADDR", "MASTER_PORT")}
    run = subprocess.run(CMD + ["--gpus", "2"], cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert run.returncode == 0, run.stderr[-2000:]
    lines = [line for line in run.stdout.splitlines() if line.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["n_gpus"] == 2 and line["impl"] == "reference" and line["value"] > 0
