"""bench.py's reference arm and the JSON line it prints (CPU only: the reference arm times the
oracle on the host cores, on the same workload and metric as the GPU arm)."""
import json
import os
import re
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
ARGS = ["--impl", "reference", "--workload", "tiny", "--steps", "1", "--warmup", "0"]


def _run(args, env=None):
    r = subprocess.run([sys.executable, "bench.py"] + args, cwd=ROOT, capture_output=True, text=True, timeout=900,
                       env=env)
    assert r.returncode == 0, r.stderr[-2000:]
    return [l for l in r.stdout.splitlines() if l.startswith("{")]


def test_reference_arm_prints_one_line_with_the_contract_keys():
    lines = _run(ARGS)
    assert len(lines) == 1
    d = json.loads(lines[0])
    for key in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
                "vs_baseline", "dtype", "data", "config", "cpu_baseline", "e2e"):
        assert key in d, key
    assert d["impl"] == "reference" and d["unit"] == "ms" and d["higher_is_better"] is False
    assert d["steps"] == 1 and d["warmup"] == 0 and d["n_gpus"] == 1
    assert d["value"] > 0 and d["cpu_baseline"]["value"] == d["value"] == d["e2e"]["value"] == d["ms_per_step"]
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["unit"] == "ms" and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"]["unit"] == "ms" and d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
    assert d["config"]["workload"].startswith("tiny")
    # the sample never exceeds the rows the method recomputes
    k, nq = d["config"]["k"], d["config"]["n_query"]
    m = re.search(r"on (\d+) of (\d+) recomputed rows", cb["sample"])
    assert m and int(m.group(2)) == k + nq
    assert 1 <= int(m.group(1)) <= k + nq


def test_reference_arm_other_ranks_print_nothing():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2")
    assert _run(ARGS, env=env) == []
