"""The bench's host side on CPU: the reference arm (the oracle timed on the host's cores) prints
one JSON line of the contract, the CPU baseline reports every core and one thread, and the value
search sizes a step by its token budget."""
import json
import os
import subprocess
import sys

import bench
from paper_2409_17836_gb300 import configs, inputs as I

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def test_reference_arm_json_line():
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny", "--steps", "2",
                        "--warmup", "1", "--ref-positions", "8"], cwd=ROOT, capture_output=True, text=True,
                       timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip()]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["steps"] == 2 and d["warmup"] == 1 and d["value"] > 0
    assert d["unit"] == "MB/s" and d["higher_is_better"] is True and d["config"]["workload"] == "tiny"
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["cores"] >= 1 and cb["value"] == d["value"] and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": "MB/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_print_nothing():
    env = dict(os.environ, RANK="1", WORLD_SIZE="2")
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "tiny", "--steps", "1",
                        "--warmup", "0"], cwd=ROOT, capture_output=True, text=True, timeout=300, env=env)
    assert r.returncode == 0 and r.stdout.strip() == ""


def test_cpu_baseline_all_cores_and_one_thread():
    cfg, vals = configs.TINY, I.tiny_gradient(0)
    cb = bench.cpu_baseline(cfg, vals, 9.0, 4, 0.2)
    assert cb["kind"] == "oracle" and cb["unit"] == "MB/s" and cb["value"] > 0
    assert cb["cores"] == max(1, len(os.sched_getaffinity(0)))
    st = cb["single_thread"]
    assert st["cores"] == 1 and st["value"] > 0 and "tokens of window 0" in st["sample"]


def test_values_for_tokens():
    # 9 tokens per value, budget 100 tokens -> 11 values; monotone counts with a fixed part
    assert bench.values_for_tokens(lambda n: 9 * n, 1000, 100) == 11
    assert bench.values_for_tokens(lambda n: 9 * n, 5, 100) == 5
    assert bench.values_for_tokens(lambda n: 2 * n + (n + 2) // 3, 10 ** 6, 2 * 3001 + 1001) == 3001
