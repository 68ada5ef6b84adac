"""The recorded DRAM traffic (profiles/traffic.json) applies to the launches it was
captured on: while the record's source digest matches the library's sources, the
planner must still emit, for every measured workload, the plans recorded with it."""
import json
import os
import shutil
import subprocess

import pytest

import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_03574_gb300", "csrc")


def sources_digest():
    import hashlib
    h = hashlib.sha256()
    for name in sorted(os.listdir(CSRC)):
        path = os.path.join(CSRC, name)
        if os.path.isfile(path):
            h.update(name.encode())
            with open(path, "rb") as f:
                h.update(f.read())
    return h.hexdigest()


def measured_plans_hash(tmp_path):
    cxx = shutil.which("g++")
    if not cxx:
        pytest.skip("no C++ compiler")
    exe = str(tmp_path / "planhash")
    srcs = [os.path.join(ROOT, "tests", "planhash.cpp")] + [os.path.join(CSRC, f) for f in
                                                             ("plan.cpp", "tape.cpp", "trace_scheme.cpp",
                                                              "trace_bytecode.cpp")]
    subprocess.run([cxx, "-O2", "-std=c++17", "-I", CSRC, *srcs, "-o", exe], check=True)
    env = {k: v for k, v in os.environ.items() if not k.startswith("NDVM_")}
    scheme = [w.program for w in W.random_exprs(200, B=2)] + [W.config(c, B=2).program for c in (1, 4, 5, 6)]
    files = []
    for i, text in enumerate(scheme + [W.config(3, B=2).program]):
        p = tmp_path / f"prog_{i:03d}.txt"
        p.write_text(text)
        files.append(str(p))
    a = subprocess.run([exe, "0", *files[:-1]], capture_output=True, text=True, env=env, check=True).stdout.strip()
    b = subprocess.run([exe, "1", files[-1]], capture_output=True, text=True, env=env, check=True).stdout.strip()
    return f"{a}:{b}"


def test_recorded_traffic_matches_the_plans_it_was_taken_on(tmp_path):
    with open(os.path.join(ROOT, "profiles", "traffic.json")) as f:
        rec = json.load(f)
    if rec.get("sources_sha256") != sources_digest():
        pytest.skip("the record does not claim the current sources (the bench then reports no traffic)")
    assert rec.get("plans_fnv1a64") == measured_plans_hash(tmp_path), \
        "the measured workloads' plans changed: capture the traffic again"
