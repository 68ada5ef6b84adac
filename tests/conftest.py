import os
import sys

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def pytest_configure(config):
    config.addinivalue_line("markers", "gpu: needs a CUDA GPU (GB300); runs the replay kernels through the C ABI")
    config.addinivalue_line("markers", "slow: long-running; selected only when NDVM_SLOW=1")


def pytest_collection_modifyitems(config, items):
    if os.environ.get("NDVM_SLOW") == "1":
        return
    skip = pytest.mark.skip(reason="slow test (set NDVM_SLOW=1)")
    for it in items:
        if "slow" in it.keywords:
            it.add_marker(skip)


@pytest.fixture(scope="session")
def oracle_mod():
    import oracle
    oracle.build()
    return oracle


@pytest.fixture(scope="session")
def ndvm():
    import paper_2607_03574_gb300 as nd
    nd.load()
    return nd


@pytest.fixture(scope="session")
def cuda():
    import torch
    if not torch.cuda.is_available():
        pytest.fail("GPU test selected but no CUDA device is visible")
    return torch.device("cuda:0")


# A lane's bound is relaxed only where the oracle's own two derivative engines disagree
# by more than tol / SPREAD_FACTOR; there it is SPREAD_FACTOR times their disagreement.
SPREAD_FACTOR = 8.0


def oracle_ref(oracle_mod, program, params, obs, frontend=0, f32=False, nthreads=8):
    """The oracle's (loss, grad, spread) for every lane.

    spread[b] = max_k |g_bk(reverse mode) - g_bk(dual numbers)| / max_j |g_bj(reverse)|:
    the disagreement of the oracle's two independent derivative engines (the pointer-graph
    reverse sweep and forward-mode dual numbers sum the same chain-rule terms in different
    orders), a measured rounding spread of that lane's gradient.  It is about 1e-16..1e-14
    on well-conditioned lanes (every Kalman lane included); it is large only where a
    gradient is a near-total cancellation, where no two evaluation orders agree to 1e-12."""
    loss, grad = oracle_mod.run(program, params, obs, frontend=frontend, nthreads=nthreads, f32=f32)
    _, dual = oracle_mod.run(program, params, obs, frontend=frontend, nthreads=nthreads, f32=f32,
                             mode=oracle_mod.MODE_DUAL)
    if grad.size == 0:
        return loss, grad, np.zeros(len(loss))
    with np.errstate(invalid="ignore", divide="ignore"):
        s = np.maximum(np.max(np.abs(grad), axis=1), 1e-300)
        spread = np.max(np.abs(grad - dual), axis=1) / s
    spread[~np.isfinite(spread)] = 0.0
    return loss, grad, spread


def rel_check(gpu_loss, gpu_grad, ora_loss, ora_grad, tol, spread=None):
    """Comparison rule for one batch of lanes.

    Loss: |gpu - ora| <= tol * |ora|.  Gradient component k of lane b:
    |gpu_bk - ora_bk| <= tol_b * max_j |ora_bj| -- the scale is the lane's largest oracle
    gradient component, nothing else, so a sign-flipped or a 1e-9-perturbed gradient
    fails.  tol_b = max(tol, SPREAD_FACTOR * spread_b) with spread_b the lane's measured
    rounding spread (oracle_ref); tol_b = tol when no spread is given.  The report counts
    the lanes whose bound was relaxed.  A lane whose oracle loss is non-finite must be
    non-finite in the same class (NaN vs +-inf) on the GPU and is excluded from the
    relative checks.  Returns (ok, report).
    """
    gpu_loss = np.asarray(gpu_loss, dtype=np.float64)
    ora_loss = np.asarray(ora_loss, dtype=np.float64)
    fin = np.isfinite(ora_loss)
    bad = []
    if (~fin).any():
        for b in np.nonzero(~fin)[0]:
            same = (np.isnan(ora_loss[b]) and np.isnan(gpu_loss[b])) or (ora_loss[b] == gpu_loss[b])
            if not same:
                bad.append(f"lane {b}: non-finite class {ora_loss[b]} vs {gpu_loss[b]}")
    el = np.abs(gpu_loss[fin] - ora_loss[fin]) / np.maximum(np.abs(ora_loss[fin]), 1e-300)
    worst_l = float(el.max()) if el.size else 0.0
    if worst_l > tol:
        b = np.nonzero(fin)[0][int(np.argmax(el))]
        bad.append(f"loss lane {b}: gpu {gpu_loss[b]!r} oracle {ora_loss[b]!r} rel {worst_l:.3e}")
    worst_g, relaxed, max_spread = 0.0, 0, 0.0
    if gpu_grad is not None and ora_grad is not None and ora_grad.size:
        g = np.asarray(gpu_grad, dtype=np.float64)[fin]
        o = np.asarray(ora_grad, dtype=np.float64)[fin]
        gfin = np.isfinite(o).all(axis=1)
        s = np.maximum(np.max(np.abs(o[gfin]), axis=1, keepdims=True), 1e-300)
        lane_tol = np.full((int(gfin.sum()), 1), float(tol))
        if spread is not None:
            sp = np.asarray(spread, dtype=np.float64)[fin][gfin].reshape(-1, 1)
            lane_tol = np.maximum(lane_tol, SPREAD_FACTOR * sp)
            relaxed = int((lane_tol > tol).sum())
            max_spread = float(sp.max()) if sp.size else 0.0
        eg = np.abs(g[gfin] - o[gfin]) / s
        worst_g = float(eg.max()) if eg.size else 0.0
        over = eg / lane_tol
        if over.size and over.max() > 1.0:
            i, k = np.unravel_index(int(np.argmax(over)), over.shape)
            bad.append(f"grad lane {i} comp {k}: gpu {g[gfin][i, k]!r} oracle {o[gfin][i, k]!r} "
                       f"rel {eg[i, k]:.3e} bound {lane_tol[i, 0]:.3e}")
        nf = ~gfin
        if nf.any() and not np.array_equal(np.isnan(g[nf]), np.isnan(o[nf])):
            bad.append("non-finite gradient class mismatch")
    return (not bad), {"worst_loss": worst_l, "worst_grad": worst_g, "nonfinite_lanes": int((~fin).sum()),
                       "relaxed_lanes": relaxed, "max_spread": max_spread, "problems": bad}


# hand-derived fixtures under tests/golden (each cites the rule it exercises and shows
# its derivation)
GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden")


def golden_cases():
    return sorted(f for f in os.listdir(GOLDEN) if f.endswith(".json"))


def load_golden(name):
    import json
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def golden_close(got, want, tol):
    """Exact equality when tol == 0, else |got - want| <= tol * |want| element by element."""
    got, want = np.asarray(got, dtype=np.float64), np.asarray(want, dtype=np.float64)
    if tol == 0:
        return np.array_equal(got, want)
    return bool(np.all(np.abs(got - want) <= tol * np.maximum(np.abs(want), 1e-300)))


# Programs where an input's adjoint and the output adjoint it copies could share slots
# while a product's or a transpose's rule reads the one and writes the other: the
# slots must stay apart there (the rule reads elements it has already written).
HAZARDS = {
    "transpose_sum": "(model (params a b c) (let* ((B (matrix 2 2 a b c a)) (A (transpose B)) (Z (m+ A B))) "
                     "(trace (matmul Z Z))))",
    "matmul_sum": "(model (params a b c) (let* ((B (matrix 2 2 a b c a)) (C (matrix 2 2 1.5 0.5 -0.25 2.0)) "
                  "(A (matmul B C)) (Z (m+ A B))) (trace (matmul Z Z))))",
    "scalar_sum": "(model (params a b c) (let* ((x (* a b)) (z (+ x a c))) (* z z)))",
}


def hazard_workloads():
    import workloads as _W
    rng = np.random.default_rng(5)
    return [_W.Workload(name, text, 0, rng.normal(size=(8, 3)), np.zeros(0), np.zeros(3))
            for name, text in HAZARDS.items()]


def matrix_program(rng, n_params=4):
    """A seeded program over small matrices: let*-bound intermediates that later terms
    reuse (sums of a matrix and its own transposes, products, scalings), reduced by
    trace, element reference, determinant and log-determinant of well-conditioned
    matrices. Text only."""
    n = int(rng.integers(2, 4))
    p = [f"p{i}" for i in range(n_params)]

    def leaf():
        return "(matrix {n} {n} {els})".format(n=n, els=" ".join(
            str(rng.choice(p)) if rng.random() < 0.6 else repr(round(float(rng.normal()), 3)) for _ in range(n * n)))

    binds, names = [], []
    for i in range(int(rng.integers(3, 6))):
        pool = names or [leaf()]
        a = str(rng.choice(pool)) if names else leaf()
        b = str(rng.choice(names)) if names and rng.random() < 0.7 else leaf()
        kind = rng.integers(0, 8)
        expr = {0: f"(m+ {a} {b})", 1: f"(m- {a} {b})", 2: f"(matmul {a} {b})", 3: f"(transpose {a})",
                4: f"(mscale {rng.choice(p)} {a})", 5: f"(m+ {a} (transpose {a}))",
                6: f"(m+ (transpose {a}) {a})", 7: f"(m+ (matmul {a} {b}) {a})"}[int(kind)]
        names.append(f"M{i}")
        binds.append(f"(M{i} {expr})")
    terms = []
    for m in names[-3:]:
        spd = f"(m+ (matmul {m} (transpose {m})) (identity {n}))"
        terms += [f"(trace {m})", f"(mref {m} 0 {n - 1})", f"(logdet {spd})", f"(trace (inv {spd}))",
                  f"(* 0.1 (det {m}))"]
    body = " ".join(str(t) for t in rng.choice(terms, size=4, replace=False))
    return f"(model (params {' '.join(p)}) (let* ({' '.join(binds)}) (+ {body})))"
