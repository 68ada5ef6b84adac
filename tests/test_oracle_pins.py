"""Pins of the oracle to things other than itself (no GPU).

Each test checks the oracle's loss and gradient against an independent fact:
closed-form gradients, the dense-Gaussian form of a Kalman likelihood, a
forward-sensitivity recursion, central finite differences, and invariants.  The
reverse mode and the dual-number mode of the oracle are also checked against each
other on every workload.
"""
import math


import numpy as np
import pytest

import workloads as W
from conftest import golden_cases, golden_close, load_golden

REV, DUAL, VAL = 0 + 1, 2, 0


def run(oracle_mod, prog, params, obs=(), frontend=0, mode=1):
    return oracle_mod.run(prog, np.atleast_2d(np.asarray(params, dtype=float)), np.asarray(obs, dtype=float),
                          frontend=frontend, mode=mode)


def assert_rel(a, b, tol, scale=None):
    a, b = np.asarray(a, float), np.asarray(b, float)
    s = np.maximum(np.abs(b), 1e-300) if scale is None else scale
    err = np.max(np.abs(a - b) / s)
    assert err <= tol, (err, a, b)


# ---------------------------------------------------------------- closed forms
LINREG = """
(model (params a b)
  (/ (data-sum {n} 2 (let ((r (- (+ (* a (dobs 0)) b) (dobs 1)))) (* r r))) {nf}))
"""


def test_linear_regression_closed_form(oracle_mod):
    rng = np.random.default_rng(11)
    n = 40
    x = rng.uniform(-3, 3, n)
    y = 0.7 * x - 1.2 + rng.normal(0, 0.3, n)
    obs = np.stack([x, y], 1).reshape(-1)
    th = rng.normal(0, 1, (6, 2))
    loss, grad = run(oracle_mod, LINREG.format(n=n, nf=f"{n}.0"), th, obs)
    for b in range(6):
        r = th[b, 0] * x + th[b, 1] - y
        assert_rel(loss[b], np.mean(r * r), 1e-13)
        assert_rel(grad[b], [2 * np.mean(r * x), 2 * np.mean(r)], 1e-12, scale=np.max(np.abs(grad[b])))


def test_exp_decay_closed_form(oracle_mod):
    w = W.exp_decay(B=16)
    loss, grad = run(oracle_mod, w.program, w.params, w.obs)
    t, y = w.obs[0::2], w.obs[1::2]
    for b in range(w.B):
        a, k, c = w.params[b]
        e = np.exp(-k * t)
        r = a * e + c - y
        assert_rel(loss[b], np.mean(r * r), 1e-13)
        g = [2 * np.mean(r * e), -2 * np.mean(r * a * t * e), 2 * np.mean(r)]
        assert_rel(grad[b], g, 1e-12, scale=np.max(np.abs(g)))


# ---------------------------------------------- Kalman: dense Gaussian identity
SCALAR_KALMAN = """
(define (nll q r y0 T)
  (let loop ((t 0) (x 0.0) (P {p0}) (acc 0.0))
    (if (= t T) acc
        (let* ((Pp (+ P q)) (S (+ Pp r)) (v (- (obs t) x)) (K (/ Pp S)))
          (loop (+ t 1) (+ x (* K v)) (* (- 1.0 K) Pp)
                (+ acc (* 0.5 (+ (log S) (/ (* v v) S) 1.8378770664093453))))))))
(model (params lq lr) (nll (exp lq) (exp lr) 0 {T}))
"""


def dense_gaussian_nll(y, Sig, dSig):
    """NLL of y ~ N(0, Sig) and its gradient given dSig/dtheta_k (list)."""
    L = np.linalg.cholesky(Sig)
    alpha = np.linalg.solve(Sig, y)
    nll = 0.5 * (2 * np.sum(np.log(np.diag(L))) + y @ alpha + len(y) * math.log(2 * math.pi))
    Si = np.linalg.inv(Sig)
    g = [0.5 * np.trace(Si @ D) - 0.5 * alpha @ D @ alpha for D in dSig]
    return nll, np.array(g)


def test_scalar_random_walk_kalman_is_dense_gaussian(oracle_mod):
    rng = np.random.default_rng(3)
    T, p0 = 30, 2.5
    y = np.cumsum(rng.normal(0, 0.5, T)) + rng.normal(0, 0.4, T)
    th = np.array([[math.log(0.25), math.log(0.16)], [math.log(1.3), math.log(0.02)], [0.1, -0.3]])
    loss, grad = run(oracle_mod, SCALAR_KALMAN.format(p0=repr(p0), T=T), th, y)
    i = np.arange(1, T + 1)
    Lm = np.minimum.outer(i, i).astype(float)
    for b in range(len(th)):
        q, r = np.exp(th[b])
        Sig = p0 + q * Lm + r * np.eye(T)
        nll, g = dense_gaussian_nll(y, Sig, [q * Lm, r * np.eye(T)])
        assert_rel(loss[b], nll, 1e-11)
        assert_rel(grad[b], g, 1e-10, scale=np.max(np.abs(g)))


def lgssm_dense_cov(F, H, Q, R, P0, T):
    """Covariance of the stacked observations of x_t = F x_{t-1} + w_t, y_t = H x_t + v_t, x_0 ~ N(0, P0)."""
    n, m = F.shape[0], H.shape[0]
    cov = [None] * (T + 1)
    cov[0] = P0
    for t in range(1, T + 1):
        cov[t] = F @ cov[t - 1] @ F.T + Q
    Sig = np.zeros((m * T, m * T))
    for t in range(1, T + 1):
        for s in range(1, t + 1):
            Ft = np.linalg.matrix_power(F, t - s)
            C = H @ Ft @ cov[s] @ H.T
            Sig[(t - 1) * m:t * m, (s - 1) * m:s * m] = C
            Sig[(s - 1) * m:s * m, (t - 1) * m:t * m] = C.T
        Sig[(t - 1) * m:t * m, (t - 1) * m:t * m] += R
    return Sig


def test_kalman_cv4_is_dense_gaussian(oracle_mod):
    T = 6
    w = W.kalman_cv4(B=5, T=T)
    loss, grad = run(oracle_mod, w.program, w.params, w.obs[: 2 * T])
    F = np.array([[1, 0, 1, 0], [0, 1, 0, 1], [0, 0, 1, 0], [0, 0, 0, 1]], float)
    H = np.eye(2, 4)
    P0 = 10 * np.eye(4)

    def sig(v):
        qx, qy, rx, ry = v
        Q = np.array([[qx / 3, 0, qx / 2, 0], [0, qy / 3, 0, qy / 2], [qx / 2, 0, qx, 0], [0, qy / 2, 0, qy]])
        return lgssm_dense_cov(F, H, Q, np.diag([rx, ry]), P0, T)

    base = sig(np.zeros(4))
    A = [sig(np.eye(4)[k]) - base for k in range(4)]   # Sigma is affine in the variances
    y = w.obs[: 2 * T]
    for b in range(w.B):
        v = np.exp(2 * w.params[b])
        Sig = base + sum(v[k] * A[k] for k in range(4))
        nll, g = dense_gaussian_nll(y, Sig, [2 * v[k] * A[k] for k in range(4)])
        assert_rel(loss[b], nll, 1e-11)
        assert_rel(grad[b], g, 1e-9, scale=np.max(np.abs(g)))


def test_kalman_rand8_is_dense_gaussian(oracle_mod):
    T = 4
    w = W.kalman_rand8(B=3, T=T)
    F = w.meta["F"]
    n, m = 8, 3
    H = np.zeros((m, n))
    H[:, :m] = np.eye(m)
    y = w.obs[: m * T]
    loss, grad = run(oracle_mod, w.program, w.params, y)

    def sig(v):
        return lgssm_dense_cov(F, H, np.diag(v[:n]), np.diag(v[n:n + m]), v[-1] * np.eye(n), T)

    base = sig(np.zeros(n + m + 1))
    A = [sig(np.eye(n + m + 1)[k]) - base for k in range(n + m + 1)]
    for b in range(w.B):
        v = np.exp(2 * w.params[b])
        Sig = base + sum(v[k] * A[k] for k in range(n + m + 1))
        nll, g = dense_gaussian_nll(y, Sig, [2 * v[k] * A[k] for k in range(n + m + 1)])
        assert_rel(loss[b], nll, 1e-10)
        assert_rel(grad[b], g, 1e-8, scale=np.max(np.abs(g)))


@pytest.mark.parametrize("m", [4, 6, 8])
def test_kalman_highd_is_dense_gaussian(oracle_mod, m):
    """The population Kalman likelihood with an m x m innovation covariance (m = 4..8,
    the elimination branch of the oracle's determinant, log-determinant and inverse)
    equals the dense Gaussian NLL of the stacked observations, and its gradient the
    trace formula (Appendix C's logdet and inv adjoints, prediction-error decomposition)."""
    T, D = 3, 12
    w = W.kalman_highd(B=3, D=D, m=m, T=T)
    F = w.meta["F"]
    H = np.zeros((m, D))
    H[:, :m] = np.eye(m)
    y = w.obs[: m * T]
    loss, grad = run(oracle_mod, w.program, w.params, y)

    def sig(v):
        return lgssm_dense_cov(F, H, v[0] * np.eye(D), v[1] * np.eye(m), v[2] * np.eye(D), T)

    base = sig(np.zeros(3))
    A = [sig(np.eye(3)[k]) - base for k in range(3)]
    for b in range(w.B):
        v = np.exp(2 * w.params[b])
        Sig = base + sum(v[k] * A[k] for k in range(3))
        nll, g = dense_gaussian_nll(y, Sig, [2 * v[k] * A[k] for k in range(3)])
        assert_rel(loss[b], nll, 1e-11)
        assert_rel(grad[b], g, 1e-9, scale=np.max(np.abs(g)))


@pytest.mark.parametrize("n", [4, 5, 6, 8])
def test_det_logdet_by_elimination_against_lapack(oracle_mod, n):
    """det and logdet of non-symmetric n x n matrices (n >= 4: the oracle eliminates with
    partial pivoting) against LAPACK's LU determinant. The matrices are row permutations
    of diagonally dominant ones, so every column's pivot lies below the diagonal and the
    elimination swaps rows; an odd permutation makes det negative. Gradients follow
    Appendix C: d det/dA = det(A) A^-T, d logdet/dA = A^-T."""
    rng = np.random.default_rng(100 + n)
    names = " ".join(f"p{k}" for k in range(n * n))
    DET = f"(model (params {names}) (det (matrix {n} {n} {names})))"
    LOGDET = f"(model (params {names}) (logdet (matrix {n} {n} {names})))"
    for trial in range(3):
        base = rng.normal(0, 0.6, (n, n)) + np.diag(rng.uniform(2.0, 4.0, n) * rng.choice([-1.0, 1.0], n))
        perm = np.roll(np.arange(n), 1 + trial)          # a cyclic shift: every pivot is off the diagonal
        A = base[perm]
        assert not np.array_equal(perm, np.arange(n))
        l, g = run(oracle_mod, DET, A.reshape(1, -1))
        d = np.linalg.det(A)
        assert_rel(l[0], d, 1e-12)
        np.testing.assert_allclose(g[0].reshape(n, n), d * np.linalg.inv(A).T, rtol=1e-11,
                                   atol=1e-12 * abs(d) * np.max(np.abs(np.linalg.inv(A))))
        Ap = A if d > 0 else A[np.r_[1, 0, 2:n]]         # one more swap makes det positive
        sgn, ld = np.linalg.slogdet(Ap)
        assert sgn > 0
        l2, g2 = run(oracle_mod, LOGDET, Ap.reshape(1, -1))
        assert abs(l2[0] - ld) <= 1e-13 * max(1.0, abs(ld))
        np.testing.assert_allclose(g2[0].reshape(n, n), np.linalg.inv(Ap).T, rtol=1e-11,
                                   atol=1e-12 * np.max(np.abs(np.linalg.inv(Ap))))
    # the sign of an odd permutation of a positive-determinant matrix
    M = np.eye(n) * 3.0 + rng.normal(0, 0.3, (n, n))
    odd = M[np.r_[1, 0, 2:n]]
    l, _ = run(oracle_mod, DET, odd.reshape(1, -1))
    assert np.sign(l[0]) == np.sign(np.linalg.det(odd)) == -np.sign(np.linalg.det(M))


# --------------------------------------------------- logistic: tangent-linear recursion
def test_logistic_forward_sensitivity(oracle_mod):
    w = W.logistic(B=6)
    loss, grad = run(oracle_mod, w.program, w.params, w.obs, frontend=1)
    dt = 0.01
    for b in range(w.B):
        r, K = w.params[b]
        x, s = 0.1, np.zeros(2)
        se, gacc = 0.0, np.zeros(2)
        k = 0
        for n in range(1000):
            f_x = r * (1 - 2 * x / K)
            f_th = np.array([x * (1 - x / K), r * x * x / (K * K)])
            s = s + dt * (f_x * s + f_th)
            x = x + dt * (r * x * (1 - x / K))
            if (n + 1) % 10 == 0:
                res = x - w.obs[k]
                se += res * res
                gacc += 2 * res * s
                k += 1
        assert_rel(loss[b], se / 100, 1e-12)
        assert_rel(grad[b], gacc / 100, 1e-11, scale=np.max(np.abs(gacc / 100)))


# ---------------------------------------------------------- finite differences
def central_fd(oracle_mod, prog, th, obs, frontend=0):
    th = np.asarray(th, float)
    P = th.size
    rows = []
    hs = 1e-5 * np.maximum(1.0, np.abs(th))
    for k in range(P):
        for sgn in (1, -1):
            t = th.copy()
            t[k] += sgn * hs[k]
            rows.append(t)
    lv, _ = run(oracle_mod, prog, np.array(rows), obs, frontend=frontend, mode=0)
    return (lv[0::2] - lv[1::2]) / (2 * hs)


@pytest.mark.parametrize("i", range(12))
def test_random_programs_match_finite_differences(oracle_mod, i):
    w = W.random_exprs(n_programs=12, B=2, n_points=24, seed=99)[i]
    loss, grad = run(oracle_mod, w.program, w.params, w.obs)
    for b in range(w.B):
        fd = central_fd(oracle_mod, w.program, w.params[b], w.obs)
        assert_rel(grad[b], fd, 2e-6, scale=max(np.max(np.abs(grad[b])), 1e-3))


def test_kalman_matches_finite_differences(oracle_mod):
    w = W.kalman_cv4(B=2, T=25)
    _, grad = run(oracle_mod, w.program, w.params, w.obs)
    for b in range(w.B):
        fd = central_fd(oracle_mod, w.program, w.params[b], w.obs)
        assert_rel(grad[b], fd, 1e-6, scale=np.max(np.abs(grad[b])))


# -------------------------------------------------- matrix primitives (App. C)
MATPROG = """
(model (params a b c d e f g h i)
  (let* ((A (matrix 3 3 a b c d e f g h i))
         (S (m+ (matmul A (transpose A)) (identity 3)))
         (B2 (submatrix A 0 2 1 2)))
    (+ (det A) (logdet S) (trace (matmul (inv S) A)) (mref (inv B2) 0 1)
       (* 0.5 (dot (matmul A (matrix 3 1 1.0 -2.0 0.5)) (matrix 3 1 0.3 0.2 0.1)))
       (trace (mscale a A)))))
"""


def test_matrix_primitives_closed_form_and_fd(oracle_mod):
    rng = np.random.default_rng(17)
    th = rng.normal(0, 1, (4, 9)) + 2 * np.eye(3).reshape(-1)
    loss, grad = run(oracle_mod, MATPROG, th)
    loss_d, grad_d = run(oracle_mod, MATPROG, th, mode=2)
    for b in range(4):
        A = th[b].reshape(3, 3)
        S = A @ A.T + np.eye(3)
        B2 = A[0:2, 1:3]
        v = 0.5 * ((A @ np.array([1.0, -2.0, 0.5])) @ np.array([0.3, 0.2, 0.1]))
        ref = (np.linalg.det(A) + np.log(np.linalg.det(S)) + np.trace(np.linalg.inv(S) @ A)
               + np.linalg.inv(B2)[0, 1] + v + np.trace(A[0, 0] * A))
        assert_rel(loss[b], ref, 1e-12)
        fd = central_fd(oracle_mod, MATPROG, th[b], ())
        assert_rel(grad[b], fd, 1e-7, scale=np.max(np.abs(grad[b])))
        assert_rel(grad[b], grad_d[b], 1e-13, scale=np.max(np.abs(grad[b])))
    # det: d det A / dA = det(A) A^-T (Appendix C); pin on a non-symmetric matrix
    DET = "(model (params a b c d e f g h i) (det (matrix 3 3 a b c d e f g h i)))"
    A = np.array([[2.0, -1.0, 0.5], [0.3, 1.7, -0.2], [1.1, 0.4, 3.0]])
    _, gd = run(oracle_mod, DET, A.reshape(1, 9))
    np.testing.assert_allclose(gd[0].reshape(3, 3), np.linalg.det(A) * np.linalg.inv(A).T, rtol=1e-13, atol=1e-13)
    # inv of a 5x5 (Gauss-Jordan path): d/dA sum(W * inv(A)) = -A^-T W A^-T
    n = 5
    A5 = np.eye(n) * 3 + rng.normal(0, 0.5, (n, n))
    Wm = rng.normal(0, 1, (n, n))
    names = " ".join(f"p{k}" for k in range(n * n))
    wel = " ".join(repr(float(x)) for x in Wm.reshape(-1))
    INV5 = (f"(model (params {names}) (trace (matmul (matrix {n} {n} {wel}) "
            f"(transpose (inv (matrix {n} {n} {names}))))))")
    l5, g5 = run(oracle_mod, INV5, A5.reshape(1, -1))
    Ai = np.linalg.inv(A5)
    assert_rel(l5[0], np.sum(Wm * Ai), 1e-12)
    np.testing.assert_allclose(g5[0].reshape(n, n), -Ai.T @ Wm @ Ai.T, rtol=1e-11, atol=1e-12)


# --------------------------------------------- primitive rules and edge cases
def test_clamps_abs_and_pow_int(oracle_mod):
    # log/sqrt: forward on max(x, 1e-8), zero gradient unless x > 1e-8 (Appendix C)
    LOGP = "(model (params x) (log x))"
    SQRTP = "(model (params x) (sqrt x))"
    xs = np.array([[1e-8], [5e-9], [-1.0], [2e-8], [3.0]])
    l, g = run(oracle_mod, LOGP, xs)
    np.testing.assert_array_equal(l[:3], np.log(1e-8))
    np.testing.assert_array_equal(g[:3, 0], 0.0)
    np.testing.assert_allclose(g[3:, 0], 1 / xs[3:, 0], rtol=1e-15)
    l, g = run(oracle_mod, SQRTP, xs)
    np.testing.assert_array_equal(l[:3], math.sqrt(1e-8))
    np.testing.assert_array_equal(g[:3, 0], 0.0)
    np.testing.assert_allclose(g[3:, 0], 0.5 / np.sqrt(xs[3:, 0]), rtol=1e-15)
    # abs'(0) = 0
    l, g = run(oracle_mod, "(model (params x) (abs x))", [[0.0], [-2.0], [3.0]])
    np.testing.assert_array_equal(g[:, 0], [0.0, -1.0, 1.0])
    # integer power by repeated multiplication; derivative n a^(n-1), finite at 0
    l, g = run(oracle_mod, "(model (params x) (pow x 3))", [[0.0], [-1.5], [2.0]])
    np.testing.assert_array_equal(l, [0.0, -3.375, 8.0])
    np.testing.assert_array_equal(g[:, 0], [0.0, 6.75, 12.0])
    l, g = run(oracle_mod, "(model (params x) (pow x 0))", [[0.0], [5.0]])
    np.testing.assert_array_equal(l, [1.0, 1.0])
    np.testing.assert_array_equal(g[:, 0], [0.0, 0.0])
    # general pow (Appendix C): a^e, d/da = e z / a, d/de = z ln a
    l, g = run(oracle_mod, "(model (params a e) (pow a e))", [[2.0, 1.5]])
    z = 2.0 ** 1.5
    np.testing.assert_allclose(g[0], [1.5 * z / 2.0, z * math.log(2.0)], rtol=1e-15)


def test_nary_forms(oracle_mod):
    # Appendix C: sub z = x0 - sum(x_i), div z = x0 / prod(x_i); single-argument - and / negate / invert
    P = "(model (params a b c) (+ (- a b c) (/ a b c) (- a) (/ b) (* a b c)))"
    th = np.array([[1.5, -2.0, 0.7]])
    l, g = run(oracle_mod, P, th)
    a, b, c = th[0]
    assert_rel(l[0], (a - b - c) + a / (b * c) - a + 1 / b + a * b * c, 1e-15)
    ga = 1 + 1 / (b * c) - 1 + b * c
    gb = -1 - a / (b * b * c) - 1 / (b * b) + a * c
    gc = -1 - a / (b * c * c) + a * b
    assert_rel(g[0], [ga, gb, gc], 1e-14, scale=max(abs(ga), abs(gb), abs(gc)))


def test_per_lane_branch_gating(oracle_mod):
    # Property 1: a parameter that appears only in a test gets no gradient; the taken side gets it
    P = "(model (params a t) (if (< t 0.0) (* a a) (* 3.0 a)))"
    l, g = run(oracle_mod, P, [[2.0, -1.0], [2.0, 1.0]])
    np.testing.assert_array_equal(l, [4.0, 6.0])
    np.testing.assert_array_equal(g, [[4.0, 0.0], [3.0, 0.0]])
    # an untaken side that would be infinite never leaks into the gradient
    P2 = "(model (params a) (if (> a 0.0) (log a) (* 2.0 a)))"
    l, g = run(oracle_mod, P2, [[0.5], [-1.0]])
    np.testing.assert_allclose(g[:, 0], [2.0, 2.0])


def test_invariants(oracle_mod):
    # a parameter-free program has zero gradient
    l, g = run(oracle_mod, "(model (params a b) (+ (exp 1.0) (obs 0)))", [[1.0, 2.0], [3.0, 4.0]], [5.0])
    np.testing.assert_array_equal(g, 0.0)
    np.testing.assert_allclose(l, math.e + 5.0)
    # identical lanes give identical outputs; lane order does not matter
    w = W.random_exprs(n_programs=3, B=6, n_points=32, seed=5)[2]
    p = np.repeat(w.params[:1], 4, axis=0)
    l, g = run(oracle_mod, w.program, p, w.obs)
    assert np.all(l == l[0]) and np.all(g == g[0])
    perm = np.array([3, 0, 5, 1, 4, 2])
    l1, g1 = run(oracle_mod, w.program, w.params, w.obs)
    l2, g2 = run(oracle_mod, w.program, w.params[perm], w.obs)
    np.testing.assert_array_equal(l1[perm], l2)
    np.testing.assert_array_equal(g1[perm], g2)


@pytest.mark.parametrize("cfg", [1, 2, 3, 4, 5])
def test_reverse_mode_equals_dual_numbers(oracle_mod, cfg):
    if cfg == 2:
        ws = W.random_exprs(n_programs=10, B=3, n_points=64, seed=2)
    elif cfg == 5:
        ws = [W.kalman_rand8(B=2, T=40)]
    elif cfg == 4:
        ws = [W.kalman_cv4(B=3, T=60)]
    else:
        ws = [W.config(cfg, B=4)]
    for w in ws:
        l1, g1 = run(oracle_mod, w.program, w.params, w.obs, frontend=w.frontend, mode=1)
        l2, g2 = run(oracle_mod, w.program, w.params, w.obs, frontend=w.frontend, mode=2)
        np.testing.assert_array_equal(l1, l2)
        s = np.max(np.abs(g1), axis=1, keepdims=True)
        assert np.max(np.abs(g1 - g2) / s) < 1e-13


@pytest.mark.parametrize("case", ["cv4_T200", "rand8_T1000", "highd_D12"])
def test_parity_rule_rejects_perturbed_gradients(oracle_mod, case):
    """The 1e-12 comparison rule measures each gradient component against the lane's
    largest oracle component, so on the Kalman likelihoods -- whose recursions make the
    terms summed into a component many orders larger than the component -- it still
    rejects a sign-flipped gradient, one perturbed by 1e-9 relative, a dropped component
    and a loss perturbed by 1e-11, while it accepts the oracle's dual-number gradient (a
    second derivative engine with another summation order).  The measured rounding
    spread of every Kalman lane is below 1e-13, so no lane's bound is relaxed."""
    from conftest import oracle_ref, rel_check
    w = {"cv4_T200": lambda: W.kalman_cv4(B=6, T=200), "rand8_T1000": lambda: W.kalman_rand8(B=3),
         "highd_D12": lambda: W.kalman_highd(B=3, D=12, m=4, T=6)}[case]()
    l, g, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs, nthreads=6)
    assert sp.max() < 1e-13, sp
    ld, gd = oracle_mod.run(w.program, w.params, w.obs, nthreads=6, mode=oracle_mod.MODE_DUAL)
    ok, rep = rel_check(ld, gd, l, g, 1e-12, sp)
    assert ok and rep["relaxed_lanes"] == 0, rep
    assert not rel_check(l, -g, l, g, 1e-12, sp)[0]
    rng = np.random.default_rng(0)
    assert not rel_check(l, g * (1 + 1e-9 * rng.choice([-1.0, 1.0], g.shape)), l, g, 1e-12, sp)[0]
    k = int(np.argmax(np.abs(g[0])))
    g1 = g.copy()
    g1[0, k] *= 1 + 1e-9
    assert not rel_check(l, g1, l, g, 1e-12, sp)[0]
    assert not rel_check(l * (1 + 1e-11), g, l, g, 1e-12, sp)[0]
    g2 = g.copy()
    g2[:, 0] = 0.0          # a dropped component
    assert not rel_check(l, g2, l, g, 1e-12, sp)[0]


def test_ill_conditioned_lane_spread(oracle_mod):
    """Lane 12 of random program 27 (200-program set, seed 1234, 37 lanes): its only
    parameter t0 = -0.0041 enters through log|1 + t0^2| and nested g / (1 + g^2) terms,
    whose derivative 1/(1 + g^2) - 2 g^2 / (1 + g^2)^2 cancels near g = 1; the gradient is
    4.5e-12 while its per-point contributions are 140 times larger and cancel too.  The
    oracle's reverse mode and dual numbers disagree there by about 2e-10 of the gradient,
    so no evaluation order can be checked at 1e-12: the rule relaxes this lane to 8 times
    that spread, which still rejects a sign flip or a 1e-8 perturbation.  Such lanes are
    rare: 15 of the 7400 lanes of all 200 programs (12 of them in program 27, whose
    parameter only enters through log|1 + t0^2| with t0 near 0); the test allows 1 %."""
    from conftest import oracle_ref, rel_check
    ws = W.random_exprs(n_programs=200, B=37, n_points=256, seed=1234)
    w = ws[27]
    l, g, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs)
    assert sp[12] > 1e-11 and np.abs(g[12]).max() < 1e-10, (sp[12], g[12])
    ok, rep = rel_check(l, g * (1 + 1e-13), l, g, 1e-12, sp)
    assert ok and rep["relaxed_lanes"] >= 1, rep
    assert not rel_check(l, -g, l, g, 1e-12, sp)[0]
    g1 = g.copy()
    g1[12] *= 1 + 1e-8
    assert not rel_check(l, g1, l, g, 1e-12, sp)[0]
    relaxed = total = 0
    for v in ws:
        _, _, s = oracle_ref(oracle_mod, v.program, v.params, v.obs)
        relaxed += int((8 * s > 1e-12).sum())
        total += len(s)
    assert relaxed <= total // 100, (relaxed, total)


def test_threads_do_not_change_results(oracle_mod):
    w = W.kalman_cv4(B=13, T=30)
    a = oracle_mod.run(w.program, w.params, w.obs, nthreads=1)
    b = oracle_mod.run(w.program, w.params, w.obs, nthreads=5)
    np.testing.assert_array_equal(a[0], b[0])
    np.testing.assert_array_equal(a[1], b[1])


# ------------------------------------------------------ bytecode (section 7)
def test_bytecode_workloads(oracle_mod):
    # W1 scalar expression: exp(a) * sin(b) - log(c) / 2
    W1 = "PARAM 0\nEXP\nPARAM 1\nSIN\nMUL\nPARAM 2\nLOG\nPUSH 2.0\nDIV\nSUB\n"
    th = np.array([[0.3, 1.1, 2.5]])
    l, g = run(oracle_mod, W1, th, frontend=1)
    a, b, c = th[0]
    assert_rel(l[0], math.exp(a) * math.sin(b) - math.log(c) / 2, 1e-15)
    assert_rel(g[0], [math.exp(a) * math.sin(b), math.exp(a) * math.cos(b), -0.5 / c], 1e-15)
    # W2 counted loop: x <- x * a + b, 7 times from x = 1
    W2 = "PUSH 1.0\nSTORE 0\nLOOP 7\nLOAD 0\nPARAM 0\nMUL\nPARAM 1\nADD\nSTORE 0\nEND\nLOAD 0\n"
    th = np.array([[0.9, 0.2]])
    l, g = run(oracle_mod, W2, th, frontend=1)
    x, dxa, dxb = 1.0, 0.0, 0.0
    for _ in range(7):
        dxa, dxb = dxa * 0.9 + x, dxb * 0.9 + 1.0
        x = x * 0.9 + 0.2
    assert_rel(l[0], x, 1e-15)
    assert_rel(g[0], [dxa, dxb], 1e-14)
    # W3 branch (lane mask): a < b ? a*b : a+b
    W3 = "PARAM 0\nPARAM 1\nLT\nPARAM 0\nPARAM 1\nMUL\nPARAM 0\nPARAM 1\nADD\nSEL\n"
    l, g = run(oracle_mod, W3, [[1.0, 3.0], [4.0, 2.0]], frontend=1)
    np.testing.assert_array_equal(l, [3.0, 6.0])
    np.testing.assert_array_equal(g, [[3.0, 1.0], [1.0, 1.0]])
    # W4 dot product and LOOP 0
    W4 = "PARAM 0\nPARAM 1\nPUSH 2.0\nPUSH 3.0\nDOT 2\nLOOP 0\nPUSH 9.0\nEND\n"
    l, g = run(oracle_mod, W4, [[0.5, -1.0]], frontend=1)
    np.testing.assert_array_equal(l, [0.5 * 2 - 3.0])
    np.testing.assert_array_equal(g, [[2.0, 3.0]])


def test_errors_are_reported(oracle_mod):
    with pytest.raises(oracle_mod.OracleError):
        run(oracle_mod, "(model (params a) (+ a", [[1.0]])
    with pytest.raises(oracle_mod.OracleError):
        run(oracle_mod, "(model (params a) (matmul (identity 2) (identity 3)))", [[1.0]])
    with pytest.raises(oracle_mod.OracleError):
        run(oracle_mod, "PARAM 0\nADD\n", [[1.0]], frontend=1)


def test_fp32_mode_is_binary32_arithmetic(oracle_mod):
    # every result rounded to float: identical to numpy float32 arithmetic step by step
    P = "(model (params a b) (- (/ (+ a 0.1) (* b 3.0)) (* a a)))"
    th = np.array([[0.7, 1.3], [-2.5, 0.11]])
    l, g = oracle_mod.run(P, th, np.zeros(0), f32=True)
    f = np.float32
    for b in range(2):
        a, bb = f(th[b, 0]), f(th[b, 1])
        ref = (a + f(0.1)) / (bb * f(3.0)) - a * a
        assert l[b] == float(ref)
    bc = "PARAM 0\nOBS 0\nADD\nPUSH 0.3\nMUL\n"
    l, g = oracle_mod.run(bc, np.array([[0.1]]), np.array([0.2]), frontend=1, f32=True)
    assert l[0] == float((f(0.1) + f(0.2)) * f(0.3))
    assert g[0, 0] == float(f(0.3))


def test_fp32_mode_matrix_primitives_are_binary32(oracle_mod):
    """Matrix primitives in fp32 mode round every product and every partial sum to
    binary32 (IEEE 754 single precision), as the fp32 variant's arithmetic does.  A dot
    product 1 + 2^-24 + 2^-24 accumulated in binary32 stays 1 (each addition is a tie
    rounded to even), whereas accumulating in binary64 and rounding once gives 1 + 2^-23;
    the same for a matrix product, a trace, a matrix sum, and the pivot products of the
    elimination that gives a 4 x 4 determinant."""
    e = 2.0 ** -24
    for prog in ("(model (params a b c) (dot (matrix 3 1 a b c) (matrix 3 1 1.0 1.0 1.0)))",
                 "(model (params a b c) (mref (matmul (matrix 1 3 a b c) (matrix 3 1 1.0 1.0 1.0)) 0 0))",
                 "(model (params a b c) (trace (matrix 3 3 a 0.0 0.0 0.0 b 0.0 0.0 0.0 c)))"):
        l32, _ = oracle_mod.run(prog, np.array([[1.0, e, e]]), np.zeros(0), f32=True)
        l64, _ = oracle_mod.run(prog, np.array([[1.0, e, e]]), np.zeros(0))
        assert l32[0] == 1.0 and l64[0] == 1.0 + 2 * e, prog
    # matrix sum: (1 + 2^-24) is not a binary32 value; the element rounds to 1
    l32, _ = oracle_mod.run("(model (params a b) (mref (m+ (matrix 1 1 a) (matrix 1 1 b)) 0 0))",
                            np.array([[1.0, e]]), np.zeros(0), f32=True)
    assert l32[0] == 1.0
    # 4 x 4 determinant (elimination): every output is a binary32 value, within a few
    # binary32 ulps of LAPACK's binary64 value, and not the binary64 value rounded once
    rng = np.random.default_rng(4)
    names = " ".join(f"p{k}" for k in range(16))
    DET = f"(model (params {names}) (det (matrix 4 4 {names})))"
    diffs = 0
    for _ in range(20):
        A = (rng.normal(0, 1, (4, 4)) + 3 * np.eye(4)).astype(np.float32).astype(np.float64)
        l32, g32 = oracle_mod.run(DET, A.reshape(1, -1), np.zeros(0), f32=True)
        assert float(np.float32(l32[0])) == l32[0]
        assert np.all(g32.astype(np.float32).astype(np.float64) == g32)
        d = np.linalg.det(A)
        assert abs(l32[0] - d) <= 64 * np.finfo(np.float32).eps * abs(d)
        diffs += l32[0] != float(np.float32(d))
    assert diffs > 0


def test_control_fuzz_reverse_equals_dual_numbers_and_fd(oracle_mod):
    """The oracle on the control-flow fuzz surface (let, let*, per-lane if, bounded loops,
    data sums): its reverse mode agrees with its dual-number mode, and with central
    differences where no lane sits near a branch switch."""
    for w in W.control_fuzz(n_programs=12, B=4, seed=77):
        l1, g1 = run(oracle_mod, w.program, w.params, w.obs, mode=1)
        l2, g2 = run(oracle_mod, w.program, w.params, w.obs, mode=2)
        np.testing.assert_array_equal(l1, l2)
        s = np.maximum(np.max(np.abs(g1), axis=1, keepdims=True), 1e-300)
        assert np.max(np.abs(g1 - g2) / s) < 1e-13, w.name
    w = W.control_fuzz(n_programs=1, B=3, seed=5)[0]
    _, g = run(oracle_mod, w.program, w.params, w.obs)
    for k in range(w.params.shape[1]):
        h = 1e-6
        pp, pm = w.params.copy(), w.params.copy()
        pp[:, k] += h
        pm[:, k] -= h
        lp, _ = run(oracle_mod, w.program, pp, w.obs)
        lm, _ = run(oracle_mod, w.program, pm, w.obs)
        np.testing.assert_allclose(g[:, k], (lp - lm) / (2 * h), rtol=1e-5, atol=1e-7)


def test_second_client_workloads(oracle_mod):
    """W1-W4 (bytecode): reverse mode equals dual numbers and central differences; W3's
    side not taken contributes nothing (its parameter enters only through the taken side)."""
    for w in W.second_client(B=3, seed=9):
        l1, g1 = run(oracle_mod, w.program, w.params, w.obs, frontend=w.frontend, mode=1)
        l2, g2 = run(oracle_mod, w.program, w.params, w.obs, frontend=w.frontend, mode=2)
        np.testing.assert_array_equal(l1, l2)
        s = np.max(np.abs(g1), axis=1, keepdims=True)
        assert np.max(np.abs(g1 - g2) / s) < 1e-13, w.name
        for k in range(w.P):
            h = 1e-6 * max(1.0, float(np.abs(w.params[:, k]).max()))
            pp, pm = w.params.copy(), w.params.copy()
            pp[:, k] += h
            pm[:, k] -= h
            lp, _ = run(oracle_mod, w.program, pp, w.obs, frontend=w.frontend)
            lm, _ = run(oracle_mod, w.program, pm, w.obs, frontend=w.frontend)
            np.testing.assert_allclose(g1[:, k], (lp - lm) / (2 * h), rtol=1e-6, atol=1e-8, err_msg=w.name)
    # W3 with the taken side made independent of parameter 1: its gradient is exactly zero
    text = W.bytecode_w3(2).replace("PARAM 1\nADD\nTANH", "PUSH 0.5\nADD\nTANH")
    _, g = run(oracle_mod, text, np.array([[0.3, 2.0], [1.0, 50.0]]), np.array([0.1, 0.2]), frontend=1)
    np.testing.assert_array_equal(g[:, 1], 0.0)


@pytest.mark.parametrize("name", golden_cases())
def test_golden_fixtures(oracle_mod, name):
    """Hand-derived values (each fixture cites the adjoint rule it exercises and shows the
    derivation): the oracle's reverse mode and its dual numbers both reproduce them,
    exactly where every intermediate is exact in binary64, else within the fixture's
    tolerance (a correctly rounded logarithm)."""
    g = load_golden(name)
    fe = oracle_mod.FRONTEND_BYTECODE if g["frontend"] == "bytecode" else oracle_mod.FRONTEND_SCHEME
    params = np.array(g["params"], dtype=np.float64)
    obs = np.array(g["obs"], dtype=np.float64)
    for mode in (oracle_mod.MODE_REVERSE, oracle_mod.MODE_DUAL):
        loss, grad = oracle_mod.run(g["program"], params, obs, frontend=fe, mode=mode)
        assert golden_close(loss, g["loss"], g["tol"]), (name, mode, loss)
        assert golden_close(grad, g["grad"], g["tol"]), (name, mode, grad)


def test_integer_helpers_and_stack_ops(oracle_mod):
    """The oracle's surface for the structural helpers and the bytecode stack moves, at
    values fixed by arithmetic: 7 quotient 2 + 7 remainder 3 + the third of (4 5 6) = 10,
    so L = 10 a; expt a 3 = a^3 with derivative 3 a^2; (p1 - p0)^2 after SWAP, SUB."""
    p = np.array([[2.0], [-0.5]])
    loss, grad = oracle_mod.run("(model (params a) (* a (exact->inexact (+ (quotient 7 2) (remainder 7 3) "
                                "(list-ref (list 4 5 6) 2)))))", p, np.zeros(0))
    np.testing.assert_array_equal(loss, [20.0, -5.0])
    np.testing.assert_array_equal(grad, [[10.0], [10.0]])
    loss, grad = oracle_mod.run("(model (params a) (expt a 3))", p, np.zeros(0))
    np.testing.assert_array_equal(loss, [8.0, -0.125])
    np.testing.assert_array_equal(grad, [[12.0], [0.75]])
    loss, grad = oracle_mod.run("PARAM 0\nPARAM 1\nSWAP\nSUB\nPOWI 2\n", np.array([[1.0, 4.0]]), np.zeros(0),
                                frontend=oracle_mod.FRONTEND_BYTECODE)
    np.testing.assert_array_equal(loss, [9.0])
    np.testing.assert_array_equal(grad, [[-6.0, 6.0]])


def test_matrix_programs_reverse_equals_dual_numbers(oracle_mod):
    """Seeded programs over small matrices (sums, differences, products, transposes,
    scalings, inverses, determinants, log-determinants, traces, element references,
    with reused intermediates): the oracle's reverse mode agrees with its dual numbers
    (two independent derivative engines) under the parity rule."""
    from conftest import matrix_program, rel_check
    for i in range(40):
        prog = matrix_program(np.random.default_rng(7000 + i))
        params = np.random.default_rng(i).normal(0.0, 0.5, (4, 4))
        lr, gr = oracle_mod.run(prog, params, np.zeros(0))
        ld, gd = oracle_mod.run(prog, params, np.zeros(0), mode=oracle_mod.MODE_DUAL)
        ok, rep = rel_check(lr, gr, ld, gd, 1e-12)
        assert ok, (prog, rep)
