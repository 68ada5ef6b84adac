"""The planner under AddressSanitizer and UndefinedBehaviorSanitizer.

tests/plansim.cpp links the planner (plan.cpp), the tape and both front ends; built with
-fsanitize=address,undefined it plans and executes gradient plans (plain and paired
streams) and value-only plans of scalar, data-axis, control-flow, bytecode and matrix
programs, and every run must end without a sanitizer report.  (The value-only plans once
read one element past a renumbering table: a plan without a reverse sweep starts that
sweep one past its last instruction.)
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

import workloads as W
from conftest import hazard_workloads, matrix_program

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_03574_gb300", "csrc")


@pytest.fixture(scope="module")
def plansim_asan(tmp_path_factory):
    cxx = shutil.which("g++")
    if not cxx:
        pytest.skip("no C++ compiler")
    exe = str(tmp_path_factory.mktemp("plansim_asan") / "plansim")
    srcs = [os.path.join(ROOT, "tests", "plansim.cpp")] + [os.path.join(CSRC, f) for f in
                                                            ("plan.cpp", "tape.cpp", "trace_scheme.cpp",
                                                             "trace_bytecode.cpp")]
    r = subprocess.run([cxx, "-O1", "-g", "-std=c++17", "-fsanitize=address,undefined", "-fno-sanitize-recover=all",
                        "-I", CSRC, *srcs, "-o", exe], capture_output=True, text=True)
    if r.returncode != 0:
        pytest.skip("sanitizers unavailable: " + r.stderr[-200:])
    return exe


def programs():
    ws = hazard_workloads() + [W.config(1)]
    ws += W.random_exprs(3, B=4, n_points=16, seed=7)
    ws += W.control_fuzz(6, B=4, seed=5)
    ws += W.second_client(B=4)
    ws += [W.logistic(B=2), W.kalman_cv4(B=2, T=5), W.kalman_rand8(B=2, T=3),
           W.kalman_highd(B=1, D=12, m=4, T=2)]
    for i in range(12):
        rng = np.random.default_rng(500 + i)
        ws.append(W.Workload(f"matrix_{i}", matrix_program(np.random.default_rng(2000 + i)), 0,
                             rng.normal(0.0, 0.5, (2, 4)), np.zeros(0), np.zeros(4)))
    return ws


def test_planner_is_clean_under_sanitizers(plansim_asan):
    env = {k: v for k, v in os.environ.items() if not k.startswith("NDVM_")}
    env["ASAN_OPTIONS"] = "detect_leaks=0"
    failures = []
    for w in programs():
        B = min(w.B, 2)
        for stream in (0, 1, 2):  # gradient plan, its paired stream, the value-only plan
            head = f"{w.frontend} {B} {w.P} {w.obs.size} {stream}\n"
            body = (" ".join(repr(float(x)) for x in w.params[:B].ravel()) + "\n" +
                    " ".join(repr(float(x)) for x in w.obs) + "\n")
            r = subprocess.run([plansim_asan], input=head + body + w.program, capture_output=True, text=True,
                               env=env, timeout=300)
            if r.returncode not in (0, 3) or "runtime error" in r.stderr or "Sanitizer" in r.stderr:
                failures.append((w.name, stream, r.returncode, r.stderr[:300]))
    assert not failures, failures
