"""bench.py's reference arm on the CPU: it times the oracle and prints one
JSON line with the main arm's metric and config keys; under several ranks
only rank 0 prints."""

import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run(rank, world):
    env = dict(os.environ, RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    r = subprocess.run([sys.executable, "bench.py", "--impl", "reference", "--workload", "c1",
                        "--steps", "1", "--warmup", "3"], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stderr[-2000:]
    return r.stdout.strip()


def test_reference_line():
    sys.path.insert(0, ROOT)
    import bench
    line = json.loads(_run(0, 1))
    assert line["impl"] == "reference" and line["metric"] == bench.METRIC
    assert line["unit"] == bench.UNIT and line["higher_is_better"] is True
    assert line["value"] > 0 and line["steps"] == 1 and line["warmup"] == 3
    assert line["cpu_baseline"]["kind"] == "oracle" and line["cpu_baseline"]["value"] == line["value"]
    assert line["e2e"] == {"value": line["value"], "unit": line["unit"], "h2d_bytes_per_step": 0,
                           "d2h_bytes_per_step": 0}
    wl = bench.WORKLOADS["c1"]
    # the main arm builds its config with the same call and note, so the two
    # arms' configs are equal key for key (tau: the planner's, bit-exact with
    # the library's calibration)
    cfg = bench.workload_config(wl, wl.batch, wl.steps, line["config"]["tau"], 1, bench.L2_NOTE)
    assert line["config"] == cfg


def test_reference_other_ranks_print_nothing():
    assert _run(1, 2) == ""
