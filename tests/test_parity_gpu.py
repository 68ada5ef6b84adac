"""GPU parity: the CUDA replay (through the C ABI) against the oracle, lane by lane.

Tolerance (fp64): 1e-12 relative, with the rule in conftest.rel_check -- loss relative
to |oracle loss|, each gradient component relative to the largest |component| of that
lane's oracle gradient.  Inputs are the seeded workloads of ``workloads`` at small
sizes (every lane checked, ragged lane counts) and at the benchmark's full sizes
(lanes sampled and recomputed by the oracle one by one).
"""
import numpy as np
import pytest

import workloads as W
from conftest import golden_cases, golden_close, hazard_workloads, load_golden, oracle_ref, rel_check

pytestmark = pytest.mark.gpu

TOL64 = 1e-12


def gpu_run(nd, w, dtype="f64", ws_bytes=None, lanes=None):
    import torch
    tdt = torch.float64 if dtype == "f64" else torch.float32
    tape = nd.trace_build(w.program, w.frontend)
    params = w.params if lanes is None else w.params[:lanes]
    p = torch.tensor(params, dtype=tdt, device="cuda")
    o = torch.tensor(w.obs, dtype=tdt, device="cuda")
    loss, grad = nd.value_and_grad(tape, p, o, ws_bytes=ws_bytes)
    fl = nd.forward(tape, p, o)
    torch.cuda.synchronize()
    nd.check_device(tape)
    return loss.double().cpu().numpy(), grad.double().cpu().numpy(), fl.double().cpu().numpy()


def oracle_run(oracle_mod, w, idx=None, nthreads=8, f32=False):
    """(loss, grad, spread) of the oracle for all lanes or the lanes idx (conftest.oracle_ref)."""
    params = w.params if idx is None else w.params[idx]
    return oracle_ref(oracle_mod, w.program, params, w.obs, frontend=w.frontend, nthreads=nthreads, f32=f32)


def check(gl, gg, ol, og, sp, tol=TOL64):
    ok, rep = rel_check(gl, gg, ol, og, tol, sp)
    assert ok, rep
    return rep


def test_exp_decay_full(ndvm, oracle_mod, cuda):
    w = W.exp_decay()                      # B = 64 lanes, 50 points
    gl, gg, fl = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)
    np.testing.assert_array_equal(fl, gl)  # value-only plan gives the same bits


@pytest.mark.parametrize("B", [1, 37, 300])
def test_exp_decay_ragged(ndvm, oracle_mod, cuda, B):
    w = W.exp_decay(B=B, n_points=23, seed=7)
    gl, gg, _ = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)


def test_random_exprs_small(ndvm, oracle_mod, cuda):
    ws = W.random_exprs(n_programs=40, B=37, n_points=256, seed=1234)
    worst = 0.0
    for w in ws:
        gl, gg, fl = gpu_run(ndvm, w)
        ol, og, sp = oracle_run(oracle_mod, w)
        rep = check(gl, gg, ol, og, sp)
        worst = max(worst, rep["worst_loss"], rep["worst_grad"])
        np.testing.assert_array_equal(fl, gl)
    print("worst relative error", worst)


def test_random_exprs_full_size_sampled(ndvm, oracle_mod, cuda):
    """Full benchmark size (B = 4096 lanes, 256 points); 64 sampled lanes per program."""
    ws = W.random_exprs(n_programs=8, B=4096, n_points=256, seed=1234)
    rng = np.random.default_rng(0)
    for w in ws:
        gl, gg, _ = gpu_run(ndvm, w)
        idx = np.sort(rng.choice(w.B, 64, replace=False))
        ol, og, sp = oracle_run(oracle_mod, w, idx)
        check(gl[idx], gg[idx], ol, og, sp)


def test_logistic_bytecode(ndvm, oracle_mod, cuda):
    w = W.logistic(B=200)
    gl, gg, fl = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)
    np.testing.assert_array_equal(fl, gl)


def test_logistic_full_size_sampled(ndvm, oracle_mod, cuda):
    w = W.logistic()                       # B = 16384
    gl, gg, _ = gpu_run(ndvm, w)
    idx = np.sort(np.random.default_rng(1).choice(w.B, 96, replace=False))
    ol, og, sp = oracle_run(oracle_mod, w, idx)
    check(gl[idx], gg[idx], ol, og, sp)


def test_logistic_workspace_chunks(ndvm, oracle_mod, cuda):
    """A workspace smaller than B lanes runs the lanes in several launches."""
    w = W.logistic(B=1000)
    tape = ndvm.trace_build(w.program, w.frontend)
    per_lane = tape.workspace_bytes(1)
    gl, gg, _ = gpu_run(ndvm, w, ws_bytes=per_lane * 300)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)


def test_kalman_cv4(ndvm, oracle_mod, cuda):
    w = W.kalman_cv4(B=70, T=200)
    gl, gg, fl = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)
    np.testing.assert_array_equal(fl, gl)


def test_kalman_cv4_full_size_sampled(ndvm, oracle_mod, cuda):
    w = W.kalman_cv4()                     # B = 8192, T = 200
    gl, gg, _ = gpu_run(ndvm, w)
    idx = np.sort(np.random.default_rng(2).choice(w.B, 64, replace=False))
    ol, og, sp = oracle_run(oracle_mod, w, idx)
    check(gl[idx], gg[idx], ol, og, sp)


def test_kalman_rand8_short(ndvm, oracle_mod, cuda):
    w = W.kalman_rand8(B=40, T=60)
    gl, gg, fl = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)
    np.testing.assert_array_equal(fl, gl)


def test_kalman_rand8_full_T_sampled(ndvm, oracle_mod, cuda):
    """T = 1000 steps at the full-size launch shape, on the first 1024 of the 65536 lanes."""
    w = W.kalman_rand8()
    gl, gg, _ = gpu_run(ndvm, w, lanes=1024)
    idx = np.sort(np.random.default_rng(3).choice(1024, 24, replace=False))
    ol, og, sp = oracle_run(oracle_mod, w, idx)
    check(gl[idx], gg[idx], ol, og, sp)


def test_lane_decomposition(ndvm, cuda):
    """A batched run equals single-lane runs, bit for bit (section 6's lane decomposition)."""
    for w in (W.exp_decay(B=9), W.logistic(B=9), W.kalman_cv4(B=9, T=30), W.random_exprs(2, B=9, n_points=40)[1]):
        gl, gg, _ = gpu_run(ndvm, w)
        for b in range(w.B):
            one = W.Workload(w.name, w.program, w.frontend, w.params[b:b + 1], w.obs, w.truth)
            l1, g1, _ = gpu_run(ndvm, one)
            np.testing.assert_array_equal(l1[0], gl[b])
            np.testing.assert_array_equal(g1[0], gg[b])


def test_identical_lanes_identical_outputs(ndvm, cuda):
    w = W.kalman_cv4(B=5, T=40)
    w.params[:] = w.params[0]
    gl, gg, _ = gpu_run(ndvm, w)
    assert np.all(gl == gl[0]) and np.all(gg == gg[0])


def test_repeat_runs_bit_identical(ndvm, cuda):
    w = W.random_exprs(3, B=500, n_points=256)[2]
    a = gpu_run(ndvm, w)
    b = gpu_run(ndvm, w)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


SELECT_PROG = """
(model (params a b)
  (let* ((x (* a 2.0))
         (y (if (< x 1.0) (* x b) (exp (- x b))))
         (z (if (> b 0.0) (log (- 0.0 b)) (* b b))))
    (+ y z (sqrt (- a 0.5)) (abs b))))
"""


def test_select_clamps_and_gating(ndvm, oracle_mod, cuda):
    """Per-lane branches (lane masks) and the 1e-8 clamps of log/sqrt at their edges."""
    rng = np.random.default_rng(5)
    a = np.concatenate([rng.uniform(-1, 2, 60), [0.5, 0.5 + 1e-9, 0.5 + 2e-8, 0.49, 0.0]])
    b = np.concatenate([rng.uniform(-2, 2, 60), [0.0, -1e-9, 1.0, -0.5, 0.0]])
    w = W.Workload("select", SELECT_PROG, 0, np.stack([a, b], 1), np.zeros(0), np.zeros(2))
    gl, gg, _ = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)


def test_empty_batch_and_zero_points(ndvm, cuda):
    import torch
    t = ndvm.trace_build(W.exp_decay(B=1).program)
    p = torch.zeros((0, 3), dtype=torch.float64, device="cuda")
    o = torch.zeros(100, dtype=torch.float64, device="cuda")
    loss, grad = ndvm.value_and_grad(t, p, o)
    assert loss.numel() == 0 and grad.shape == (0, 3)
    prog = "(model (params a) (+ (data-sum 0 2 (* a (dobs 0))) (* a a)))"
    t2 = ndvm.trace_build(prog)
    p2 = torch.tensor([[3.0], [-2.0]], dtype=torch.float64, device="cuda")
    l2, g2 = ndvm.value_and_grad(t2, p2, None)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(l2.cpu().numpy(), [9.0, 4.0])
    np.testing.assert_array_equal(g2.cpu().numpy(), [[6.0], [-4.0]])


def test_host_entry_point_matches_device(ndvm, cuda):
    w = W.logistic(B=77)
    tape = ndvm.trace_build(w.program, w.frontend)
    hl, hg = ndvm.value_and_grad_host(tape, w.params, w.obs)
    gl, gg, _ = gpu_run(ndvm, w)
    np.testing.assert_array_equal(hl, gl)
    np.testing.assert_array_equal(hg, gg)


def test_logistic_fp32_variant(ndvm, oracle_mod, cuda):
    """fp32 replay against the oracle in binary32 arithmetic, 1e-5 relative."""
    w = W.logistic(B=300)
    w.params = w.params.astype(np.float32).astype(np.float64)
    gl, gg, fl = gpu_run(ndvm, w, dtype="f32")
    ol, og, sp = oracle_run(oracle_mod, w, f32=True)
    check(gl, gg, ol, og, sp, tol=1e-5)
    np.testing.assert_array_equal(fl, gl)


def test_exp_decay_fp32_variant(ndvm, oracle_mod, cuda):
    w = W.exp_decay(B=64)
    w.params = w.params.astype(np.float32).astype(np.float64)
    gl, gg, _ = gpu_run(ndvm, w, dtype="f32")
    ol, og, sp = oracle_run(oracle_mod, w, f32=True)
    check(gl, gg, ol, og, sp, tol=1e-5)


ARITH_PROG = """
(model (params a b c)
  (- (* (+ a b) (- c a)) (* (- 0.0 b) (+ c 0.5)) (* a -0.0) (- c)))
"""


def test_fused_forward_is_bit_exact(ndvm, oracle_mod, cuda):
    """add, sub, mul and neg run in the fused multiply-add form; the rewrite is exact,
    so a program made only of them gives the oracle's loss bit for bit -- signed zeros,
    infinities, NaNs and subnormals included."""
    rng = np.random.default_rng(11)
    special = [0.0, -0.0, np.inf, -np.inf, np.nan, 5e-324, -2.5e-310, 1e308, -1e308, 1.0]
    cols = [np.concatenate([rng.normal(size=40), rng.choice(special, 24)]) for _ in range(3)]
    w = W.Workload("arith", ARITH_PROG, 0, np.stack(cols, 1), np.zeros(0), np.zeros(3))
    gl, _, fl = gpu_run(ndvm, w)
    ol, _, _ = oracle_run(oracle_mod, w)
    same = (gl.view(np.int64) == ol.view(np.int64)) | (np.isnan(gl) & np.isnan(ol))
    assert same.all(), np.nonzero(~same)
    same_fwd = (fl.view(np.int64) == gl.view(np.int64)) | (np.isnan(fl) & np.isnan(gl))
    assert same_fwd.all(), np.nonzero(~same_fwd)


SKIP_PROG = """
(model (params a b)
  (+ (if (< a 0.0) (* a (exp b)) (* a a))
     (log (* (- 0.0 a) (exp b)))))
"""


def test_zero_adjoints_skip_infinite_factors(ndvm, oracle_mod, cuda):
    """An adjoint that is exactly zero contributes nothing even when the other factor
    is infinite: the untaken branch's product and the product under a clamped log
    (zero gradient) leave the gradient finite where the oracle's is finite."""
    a = np.array([0.5, 2.0, -1.0, 3.0, 0.0, -0.0, 1e-3])
    b = np.array([800.0, 1e3, 1.0, 30.0, 800.0, 2.0, 40.0])
    w = W.Workload("skip", SKIP_PROG, 0, np.stack([a, b], 1), np.zeros(0), np.zeros(2))
    gl, gg, _ = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    assert np.isfinite(ol).all() and np.isfinite(og).all()  # the pin: every lane stays finite
    check(gl, gg, ol, og, sp)


def test_async_host_entry_point_overlaps_tapes(ndvm, cuda):
    """Asynchronous host-buffer calls on different tapes and streams give the
    synchronous call's results once the streams are synchronized."""
    import torch
    ws = [W.logistic(B=50), W.exp_decay(B=40), W.kalman_cv4(B=30, T=12)]
    tapes = [ndvm.trace_build(w.program, w.frontend) for w in ws]
    streams = [torch.cuda.Stream() for _ in ws]
    pin = lambda a: torch.tensor(a).pin_memory().numpy()
    hp, ho = [pin(w.params) for w in ws], [pin(w.obs) for w in ws]
    hl = [torch.empty(w.B, dtype=torch.float64).pin_memory().numpy() for w in ws]
    hg = [torch.empty(w.params.shape, dtype=torch.float64).pin_memory().numpy() for w in ws]
    for k in range(len(ws)):
        ndvm.value_and_grad_host_async(tapes[k], hp[k], ho[k], hl[k], hg[k], stream=streams[k])
    for s in streams:
        s.synchronize()
    for k, w in enumerate(ws):
        sl, sg = ndvm.value_and_grad_host(tapes[k], w.params, w.obs)
        np.testing.assert_array_equal(hl[k], sl)
        np.testing.assert_array_equal(hg[k], sg)


@pytest.mark.parametrize("k", range(4), ids=["W1", "W2", "W3", "W4"])
def test_second_client_bytecode_workloads(ndvm, oracle_mod, cuda, k):
    """The bytecode VM's W1-W4 (scalar expression, counted loop, data-independent
    branch, summed matrix-vector product) over 256 lanes against the oracle."""
    w = W.second_client(B=256)[k]
    gl, gg, fl = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)
    np.testing.assert_array_equal(fl, gl)


STRUCTURAL_PROGRAMS = {
    "recursion": "(define (pw x n) (if (= n 0) 1.0 (* x (pw x (- n 1))))) (model (params a b) (+ (pw a 5) (pw b 2)))",
    "closure": "(define (scale k) (lambda (x) (* k x))) (model (params a b) (let ((f (scale a))) (+ (f b) (f 2.0))))",
    "lists": "(define (sum l) (if (null? l) 0.0 (+ (car l) (sum (cdr l))))) "
             "(define (mp f l) (if (null? l) (quote ()) (cons (f (car l)) (mp f (cdr l))))) "
             "(model (params a b) (sum (mp (lambda (x) (* x (sin x))) (list a b (* a b) 3.0))))",
    "compose": "(define (compose f g) (lambda (x) (f (g x)))) (model (params a b) ((compose exp sin) (* a b)))",
    "mutual": "(define (ev n x) (if (= n 0) x (od (- n 1) (* 1.5 x)))) "
              "(define (od n x) (if (= n 0) x (ev (- n 1) (+ x (tanh x))))) (model (params a b) (ev 7 (* a b)))",
}


@pytest.mark.parametrize("name", sorted(STRUCTURAL_PROGRAMS))
def test_structural_surface_programs(ndvm, oracle_mod, cuda, name):
    """Recursion, closures, lists and higher-order functions are structural (they record
    no tape nodes); the realized numeric trace replays to the oracle's values."""
    rng = np.random.default_rng(3)
    w = W.Workload(name, STRUCTURAL_PROGRAMS[name], 0, rng.uniform(-1.5, 1.5, (100, 2)), np.zeros(0), np.zeros(2))
    gl, gg, _ = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)


def test_degenerate_programs(ndvm, oracle_mod, cuda):
    """A parameter that the trace never reaches has an exactly zero gradient; a program
    without parameters has a loss and no gradient columns; a constant program gives the
    constant on every lane."""
    import torch
    w = W.Workload("unused", "(model (params a b c) (* (sin a) (exp c)))", 0,
                   np.random.default_rng(1).normal(size=(37, 3)), np.zeros(0), np.zeros(3))
    gl, gg, _ = gpu_run(ndvm, w)
    ol, og, sp = oracle_run(oracle_mod, w)
    check(gl, gg, ol, og, sp)
    np.testing.assert_array_equal(gg[:, 1], 0.0)
    t0 = ndvm.trace_build("(model (params) (* 2.0 (+ 1.5 (obs 0))))")
    p0 = torch.zeros((5, 0), dtype=torch.float64, device="cuda")
    o0 = torch.tensor([0.25], dtype=torch.float64, device="cuda")
    l0, g0 = ndvm.value_and_grad(t0, p0, o0)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(l0.cpu().numpy(), np.full(5, 3.5))
    assert g0.shape == (5, 0)
    tc = ndvm.trace_build("(model (params a) 4.25)")
    lc, gc = ndvm.value_and_grad(tc, torch.ones((3, 1), dtype=torch.float64, device="cuda"), None)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(lc.cpu().numpy(), np.full(3, 4.25))
    np.testing.assert_array_equal(gc.cpu().numpy(), 0.0)


def test_million_lanes_sampled(ndvm, oracle_mod, cuda):
    """2^20 lanes in one call (8192 blocks): sampled lanes against the oracle."""
    rng = np.random.default_rng(8)
    base = W.exp_decay(B=1)
    w = W.Workload("big", base.program, 0, 1.0 + 0.3 * rng.standard_normal((1 << 20, 3)), base.obs, base.truth)
    gl, gg, _ = gpu_run(ndvm, w)
    idx = np.array([0, 1, 12345, 524287, 524288, (1 << 20) - 1])
    ol, og, sp = oracle_run(oracle_mod, w, idx)
    check(gl[idx], gg[idx], ol, og, sp)


TWO_REGION_PROG = """
(model (params a b)
  (+ (* 0.25 (data-sum 24 3 0 (let ((s (sin (* 2.0 (dobs 0)))) (c (exp (/ (dobs 1) 4.0))))
                                (let ((r (- (* a s) (* b c) (dobs 2)))) (* r r)))))
     (data-sum 10 2 72 (let ((q (log (+ 1.0 (* (dobs 1) (dobs 1))))))
                         (* (+ a q) (- b (cos (dobs 0))))))
     (data-sum 5 1 92 (* (dobs 0) (dobs 0)))))
"""


def test_shared_point_values_match_per_lane_values(ndvm, oracle_mod, cuda, monkeypatch):
    """Values that depend on the data point but on no parameter are computed once per call
    (three regions: shared values feeding parameter terms, a product of two shared values,
    and a region that is shared as a whole). The replay with them equals, bit for bit,
    the replay that recomputes them on every lane, and the oracle at 1e-12."""
    import torch
    rng = np.random.default_rng(21)
    obs = rng.normal(size=97)
    params = rng.normal(size=(70, 2))
    w = W.Workload("regions", TWO_REGION_PROG, 0, params, obs, np.zeros(2))
    shared = ndvm.trace_build(w.program)
    monkeypatch.setenv("NDVM_DERIVE", "0")
    per_lane = ndvm.trace_build(w.program)
    monkeypatch.delenv("NDVM_DERIVE")
    assert shared.cost()["work_shared"] > 0 and per_lane.cost()["work_shared"] == 0
    assert shared.workspace_bytes(70) > 0
    p = torch.tensor(params, device="cuda")
    o = torch.tensor(obs, device="cuda")
    l1, g1 = ndvm.value_and_grad(shared, p, o)
    l2, g2 = ndvm.value_and_grad(per_lane, p, o)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(l1.cpu().numpy(), l2.cpu().numpy())
    np.testing.assert_array_equal(g1.cpu().numpy(), g2.cpu().numpy())
    ol, og, sp = oracle_run(oracle_mod, w)
    check(l1.cpu().numpy(), g1.cpu().numpy(), ol, og, sp)


@pytest.mark.parametrize("cfg,B", [(3, 16384), (4, 8192), (6, 256)])
def test_paired_chains_and_trimmed_fetches_are_exact(ndvm, oracle_mod, cuda, monkeypatch, cfg, B):
    """Three stream rewrites change no arithmetic: sharing a slot between an adjoint and
    its first contribution when that is a plain copy (equal values; only a zero's sign
    may differ, and zeros compare equal), pairing fused updates that save their result,
    pairing a fused update with the next one
    that reads its result (two contributions to one adjoint, a step of a recurrence), and
    leaving out the fetch records of reverse-sweep windows that fetch nothing (waits then
    count only the groups that were committed). The replay with them equals the replay
    without them (copies kept, independent pairs without saves only, a commit and a wait in
    every window),
    at the launch shape the bench uses, and the oracle at 1e-12 on sampled lanes."""
    import torch
    w = W.config(cfg, B=B)
    monkeypatch.setenv("NDVM_DEPPAIR", "0")
    monkeypatch.setenv("NDVM_SAVEPAIR", "0")
    monkeypatch.setenv("NDVM_FETCHTRIM", "0")
    monkeypatch.setenv("NDVM_COALESCE", "0")
    plain = ndvm.trace_build(w.program, w.frontend)
    monkeypatch.delenv("NDVM_DEPPAIR")
    monkeypatch.delenv("NDVM_SAVEPAIR")
    monkeypatch.delenv("NDVM_FETCHTRIM")
    monkeypatch.delenv("NDVM_COALESCE")
    tape = ndvm.trace_build(w.program, w.frontend)
    p = torch.tensor(w.params, device="cuda")
    o = torch.tensor(w.obs, device="cuda")
    l1, g1 = ndvm.value_and_grad(tape, p, o)
    l2, g2 = ndvm.value_and_grad(plain, p, o)
    torch.cuda.synchronize()
    ndvm.check_device(tape)
    ndvm.check_device(plain)
    np.testing.assert_array_equal(l1.cpu().numpy(), l2.cpu().numpy())
    np.testing.assert_array_equal(g1.cpu().numpy(), g2.cpu().numpy())
    idx = np.array([0, 1, B // 2, B - 1])
    ol, og, sp = oracle_run(oracle_mod, w, idx)
    check(l1.cpu().numpy()[idx], g1.cpu().numpy()[idx], ol, og, sp)


def _region_workloads():
    rng = np.random.default_rng(33)
    ws = [W.config(1)]
    ws += W.random_exprs(6, B=512, seed=77)
    ws.append(W.Workload("regions", TWO_REGION_PROG, 0, rng.normal(size=(300, 2)), rng.normal(size=97), np.zeros(2)))
    return ws


@pytest.mark.parametrize("k", range(8))
def test_point_loads_and_hoisted_seed_are_exact(ndvm, oracle_mod, cuda, monkeypatch, k):
    """Rewrites of data-axis loops change no arithmetic: the current point's observations
    load at the start of the loop body as asynchronous copies, up to four per record; the
    reverse sweep's seed d(body)/d(body) = 1 is set once before the loop when nothing in
    the body writes its slot; an adjoint whose first contribution is a plain copy shares
    the copied slot. The replay with them equals the replay without them (a zero's sign
    may differ; zeros compare equal), and the oracle at 1e-12 on sampled lanes."""
    import torch
    w = _region_workloads()[k]
    monkeypatch.setenv("NDVM_MERGELOADS", "0")
    monkeypatch.setenv("NDVM_HOIST", "0")
    monkeypatch.setenv("NDVM_COALESCE", "0")
    plain = ndvm.trace_build(w.program, w.frontend)
    monkeypatch.delenv("NDVM_MERGELOADS")
    monkeypatch.delenv("NDVM_HOIST")
    monkeypatch.delenv("NDVM_COALESCE")
    tape = ndvm.trace_build(w.program, w.frontend)
    p = torch.tensor(w.params, device="cuda")
    o = torch.tensor(w.obs, device="cuda")
    l1, g1 = ndvm.value_and_grad(tape, p, o)
    l2, g2 = ndvm.value_and_grad(plain, p, o)
    f1 = ndvm.forward(tape, p, o)
    torch.cuda.synchronize()
    ndvm.check_device(tape)
    ndvm.check_device(plain)
    np.testing.assert_array_equal(l1.cpu().numpy(), l2.cpu().numpy())
    np.testing.assert_array_equal(g1.cpu().numpy(), g2.cpu().numpy())
    np.testing.assert_array_equal(f1.cpu().numpy(), l1.cpu().numpy())
    B = len(w.params)
    idx = np.array([0, 1, B // 2, B - 1])
    ol, og, sp = oracle_run(oracle_mod, w, idx)
    check(l1.cpu().numpy()[idx], g1.cpu().numpy()[idx], ol, og, sp)


@pytest.mark.parametrize("name", golden_cases())
def test_golden_fixtures_gpu(ndvm, cuda, name):
    """The replay reproduces the hand-derived values of tests/golden: exactly where every
    intermediate is exact in binary64 (the fused updates round once, which changes
    nothing there), else within 1e-12 (the library's own logarithm is faithful, not
    correctly rounded). Both the gradient plan and the value-only plan."""
    import torch
    g = load_golden(name)
    fe = ndvm.FE_BYTECODE if g["frontend"] == "bytecode" else ndvm.FE_SCHEME
    tape = ndvm.trace_build(g["program"], fe)
    p = torch.tensor(g["params"], dtype=torch.float64, device="cuda")
    o = torch.tensor(g["obs"] if g["obs"] else [0.0], dtype=torch.float64, device="cuda")
    loss, grad = ndvm.value_and_grad(tape, p, o)
    fl = ndvm.forward(tape, p, o)
    torch.cuda.synchronize()
    ndvm.check_device(tape)
    tol = 0 if g["tol"] == 0 else 1e-12
    assert golden_close(loss.cpu().numpy(), g["loss"], tol), (name, loss)
    assert golden_close(fl.cpu().numpy(), g["loss"], tol), (name, fl)
    assert golden_close(grad.cpu().numpy(), g["grad"], tol), (name, grad)


def test_shared_adjoint_slots_stay_apart_where_a_rule_reads_after_writing(ndvm, oracle_mod, cuda, monkeypatch):
    """Z = A + B with A = B^T (or A = B C): the sum's rule copies Z's adjoint to both A and
    B, and the transpose's (product's) rule then reads A's adjoint while it writes B's.
    Sharing one slot there would let the rule read elements it has already written, so
    the planner keeps those adjoints apart: the replay equals the one without slot
    sharing and the oracle."""
    import torch
    for w in hazard_workloads():
        tape = ndvm.trace_build(w.program)
        monkeypatch.setenv("NDVM_COALESCE", "0")
        plain = ndvm.trace_build(w.program)
        monkeypatch.delenv("NDVM_COALESCE")
        p = torch.tensor(w.params, device="cuda")
        o = torch.zeros(1, dtype=torch.float64, device="cuda")
        l1, g1 = ndvm.value_and_grad(tape, p, o)
        l2, g2 = ndvm.value_and_grad(plain, p, o)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(l1.cpu().numpy(), l2.cpu().numpy())
        np.testing.assert_array_equal(g1.cpu().numpy(), g2.cpu().numpy())
        ol, og, sp = oracle_run(oracle_mod, w)
        check(l1.cpu().numpy(), g1.cpu().numpy(), ol, og, sp)
