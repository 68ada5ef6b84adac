"""The planner's stream rewrites checked without a GPU.

tests/plansim.cpp executes the replay plans on the CPU with the device interpreter's
instruction semantics (scalar, data-axis and matrix tapes, one thread per lane). For every program: the simulated replay matches the oracle under the
parity rule, the paired stream gives the same values as the unpaired one, and the
plans built with every rewrite switched off give the same values as the default plans
(copies coalesced, seeds hoisted, observation loads merged, dependent and saving pairs,
trimmed fetch windows, shared per-point values, prefetch). Zeros compare equal
whatever their sign (slot sharing may keep a zero adjoint's sign).
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

import workloads as W
from conftest import hazard_workloads, matrix_program, oracle_ref, rel_check

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2607_03574_gb300", "csrc")
OFF = {"NDVM_COALESCE": "0", "NDVM_HOIST": "0", "NDVM_MERGELOADS": "0", "NDVM_DEPPAIR": "0", "NDVM_SAVEPAIR": "0",
       "NDVM_FETCHTRIM": "0", "NDVM_DERIVE": "0", "NDVM_PREFETCH": "0"}


@pytest.fixture(scope="module")
def plansim(tmp_path_factory):
    cxx = shutil.which("g++")
    if not cxx:
        pytest.skip("no C++ compiler")
    exe = str(tmp_path_factory.mktemp("plansim") / "plansim")
    srcs = [os.path.join(ROOT, "tests", "plansim.cpp")] + [os.path.join(CSRC, f) for f in
                                                            ("plan.cpp", "tape.cpp", "trace_scheme.cpp",
                                                             "trace_bytecode.cpp")]
    subprocess.run([cxx, "-O2", "-std=c++17", "-I", CSRC, *srcs, "-o", exe], check=True)
    return exe


def simulate(exe, w, stream=0, env_extra=None):
    """(loss[B], grad[B, P]) of the simulated replay, or None for a tape with matrix
    instructions."""
    env = {k: v for k, v in os.environ.items() if not k.startswith("NDVM_")}
    env.update(env_extra or {})
    head = f"{w.frontend} {w.B} {w.P} {w.obs.size} {stream}\n"
    body = " ".join(repr(float(x)) for x in w.params.ravel()) + "\n" + " ".join(repr(float(x)) for x in w.obs) + "\n"
    r = subprocess.run([exe], input=head + body + w.program, capture_output=True, text=True, env=env, timeout=300)
    if r.returncode == 3:
        return None
    assert r.returncode == 0, r.stderr
    rows = np.array([[float.fromhex(t) for t in line.split()] for line in r.stdout.strip().splitlines()])
    return rows[:, 0], rows[:, 1:]


def programs():
    ws = hazard_workloads() + [W.config(1)]
    ws += W.random_exprs(6, B=48, n_points=32, seed=99)
    ws += W.control_fuzz(24, B=24)
    ws += W.second_client(B=24)
    ws.append(W.logistic(B=12))
    ws.append(W.kalman_cv4(B=6, T=12))
    ws.append(W.kalman_rand8(B=4, T=6))
    ws.append(W.kalman_highd(B=2, D=12, m=3, T=3))
    return ws


CASES = programs()


@pytest.mark.parametrize("k", range(len(CASES)))
def test_simulated_plans_match_the_oracle_and_each_other(plansim, oracle_mod, k):
    w = CASES[k]
    base = simulate(plansim, w, 0)
    if base is None:
        pytest.skip("matrix instructions are not simulated")
    ol, og, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs, frontend=w.frontend)
    ok, rep = rel_check(base[0], base[1], ol, og, 1e-12, sp)
    assert ok, (w.name, rep)
    value = simulate(plansim, w, 2)
    assert np.array_equal(value[0], base[0]), w.name  # the value-only plan gives the same loss bits
    for stream, env in ((1, None), (0, OFF), (1, OFF)):
        other = simulate(plansim, w, stream, env)
        assert np.array_equal(other[0], base[0]), (w.name, stream, env)
        assert np.array_equal(other[1], base[1]), (w.name, stream, env)


MATRIX_CASES = [matrix_program(np.random.default_rng(1000 + i)) for i in range(60)]


@pytest.mark.parametrize("k", range(len(MATRIX_CASES)))
def test_simulated_matrix_programs(plansim, oracle_mod, k):
    """Seeded matrix programs (the adjoint slots of sums, transposes and products meet
    in many ways): the simulated replay matches the oracle, with and without the
    rewrites, on the plain and the paired stream. (A determinant of a singular matrix
    gives a NaN gradient through A^-T on both sides; NaNs compare equal here.)"""
    rng = np.random.default_rng(k)
    w = W.Workload(f"matrix_{k}", MATRIX_CASES[k], 0, rng.normal(0.0, 0.5, (6, 4)), np.zeros(0), np.zeros(4))
    base = simulate(plansim, w, 0)
    ol, og, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs)
    ok, rep = rel_check(base[0], base[1], ol, og, 1e-12, sp)
    assert ok, (w.program, rep)
    for stream, env in ((1, None), (0, OFF), (1, OFF)):
        other = simulate(plansim, w, stream, env)
        assert np.array_equal(other[0], base[0], equal_nan=True), (w.program, stream, env)
        assert np.array_equal(other[1], base[1], equal_nan=True), (w.program, stream, env)
