"""Host-side checks of bench.py's reference arm (the oracle timed on the host cores): the
JSON line it prints carries the contract's keys, and under a multi-rank launch only rank
0 prints. No GPU is used."""
import json
import os
import subprocess
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def run_bench(args, env_extra=None):
    env = dict(os.environ)
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        env.pop(k, None)
    env.update(env_extra or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py")] + args, cwd=ROOT, env=env,
                          capture_output=True, text=True, timeout=600)


def test_reference_arm_prints_the_contract_line():
    r = run_bench(["--impl", "reference", "--config", "1", "--steps", "1", "--warmup", "3"])
    assert r.returncode == 0, r.stderr[-2000:]
    d = json.loads(r.stdout.strip().splitlines()[-1])
    for k in ("metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step", "higher_is_better", "scaling",
              "vs_baseline", "dtype", "data", "config", "e2e", "cpu_baseline"):
        assert k in d, k
    assert d["impl"] == "reference" and d["n_gpus"] == 1 and d["steps"] == 1 and d["warmup"] == 3
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["higher_is_better"] is True
    assert d["e2e"] == {"value": d["value"], "unit": d["unit"], "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert "workload" in d["config"]


def test_reference_arm_other_ranks_exit_quietly():
    r = run_bench(["--impl", "reference", "--config", "1", "--steps", "1", "--warmup", "3", "--gpus", "2"],
                  {"RANK": "1", "WORLD_SIZE": "2", "LOCAL_RANK": "1"})
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""


def test_warmup_below_three_is_refused():
    r = run_bench(["--impl", "reference", "--config", "1", "--steps", "1", "--warmup", "1"])
    assert r.returncode != 0
    assert "warmup" in r.stderr


def test_cpu_baseline_times_all_cores_and_one():
    """The GPU arm's cpu_baseline: the oracle on every host core, and on one core over a
    sample sized from the all-core rate (a bounded run)."""
    import importlib.util
    import types
    spec = importlib.util.spec_from_file_location("bench_mod", os.path.join(ROOT, "bench.py"))
    b = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(b)
    args = types.SimpleNamespace(config=1, lanes=0, programs=1, dtype="f64", cpu_lanes=0)
    progs, _ = b.workload_for(args, b.SEED)
    cb = b.cpu_baseline(args, progs)
    assert cb["kind"] == "oracle" and cb["unit"] == b.UNIT and cb["cores"] >= 1 and cb["value"] > 0
    one = cb["single_core"]
    assert one["cores"] == 1 and one["value"] > 0 and one["unit"] == b.UNIT and one["sample"]
