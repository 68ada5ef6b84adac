"""Seeded synthetic workloads for the NDVM tape-replay path.

This module only *synthesises inputs*: program texts, observation vectors and
per-lane parameter draws, from numpy's PCG64 generator with fixed seeds.  It holds
none of the method's arithmetic (no tape, no adjoint, no loss reduction), and it is
the only code shared by the product's tests/benchmark and the oracle.  Simulating
the data-generating process (an Euler trajectory, a linear-Gaussian state-space
model, a random expression evaluated at its hidden constants) is part of the input
recipe, done here with plain numpy.

Five workloads, shaped like the paper's (sections 6-7 and Appendix A):

  1 exp-decay      y = a exp(-b t) + c, 50 points, MSE, P=3, B=64
  2 random exprs   200 programs (+ - * / exp log|x| sin pow-int, depth <= 6,
                   1-8 constants), 256 points, MSE, B=4096 lanes per program
  3 logistic       bytecode, explicit Euler dx/dt = r x (1 - x/K), 1000 steps,
                   dt = 0.01, 100 observations, MSE, P=2, B=16384
  4 kalman-4       4-state constant-velocity Kalman NLL, 2-d obs, T=200, P=4, B=8192
  5 kalman-8       8-state random stable Kalman NLL, 3-d obs, T=1000, P=12, B=65536

Every generator takes the sizes as arguments, so tests can build small instances
of the same recipe.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

FRONTEND_SCHEME = 0
FRONTEND_BYTECODE = 1


@dataclass
class Workload:
    name: str
    program: str            # program text (the single source of truth for both paths)
    frontend: int           # 0 Scheme-style, 1 stack bytecode
    params: np.ndarray      # (B, P) float64 lane parameters
    obs: np.ndarray         # (n_obs,) float64 observations shared by all lanes
    truth: np.ndarray       # (P,) hidden parameters used to synthesise obs
    meta: dict = field(default_factory=dict)

    @property
    def B(self) -> int:
        return int(self.params.shape[0])

    @property
    def P(self) -> int:
        return int(self.params.shape[1])


def _fmt(x: float) -> str:
    """Shortest round-tripping decimal for a double, always with a '.' or exponent."""
    s = repr(float(x))
    if "e" not in s and "." not in s and "inf" not in s and "nan" not in s:
        s += ".0"
    return s


# --------------------------------------------------------------------------
# 1. exponential decay
# --------------------------------------------------------------------------
def exp_decay(B: int = 64, n_points: int = 50, seed: int = 1234) -> Workload:
    rng = np.random.default_rng(seed)
    truth = np.array([1.3, 0.8, 0.9])
    t = rng.uniform(0.0, 5.0, n_points)
    y = truth[0] * np.exp(-truth[1] * t) + truth[2] + rng.normal(0.0, 0.05, n_points)
    obs = np.empty(2 * n_points)
    obs[0::2] = t
    obs[1::2] = y
    params = rng.normal(1.0, 0.3, (B, 3))
    program = (
        ";; exponential decay y = a exp(-b t) + c, mean squared error over the data axis\n"
        "(model (params a b c)\n"
        f"  (/ (data-sum {n_points} 2\n"
        "       (let ((r (- (+ (* a (exp (- (* b (dobs 0))))) c) (dobs 1))))\n"
        "         (* r r)))\n"
        f"     {_fmt(float(n_points))}))\n"
    )
    return Workload("exp_decay", program, FRONTEND_SCHEME, params, obs, truth,
                    {"n_points": n_points})


# --------------------------------------------------------------------------
# 2. random expression programs (the paper's typed program generator, section 6)
# --------------------------------------------------------------------------
# Grammar: + - * / exp log|x| sin pow-int over x and constants theta_k.
# Domain guards in the spirit of the paper's generator (section 6): a division by d
# divides by 1 + d*d instead, a log argument a becomes 1 + a*a (inside log|.|), an exp
# argument a becomes a / (1 + a*a), bounded by 1/2.  A program is kept only if every intermediate value
# stays within 1e4 in magnitude at the hidden constants and at sampled lanes.

_BIN = ("+", "-", "*", "/")
_UN = ("exp", "log", "sin", "pow")


class _Gen:
    def __init__(self, rng, max_depth, max_consts):
        self.rng = rng
        self.max_depth = max_depth
        self.max_consts = max_consts
        self.nconst = 0

    def leaf(self):
        # x or a constant
        if self.rng.random() < 0.5 or self.nconst == 0:
            if self.nconst < self.max_consts and self.rng.random() < 0.6:
                k = self.nconst
                self.nconst += 1
                return ("c", k)
            if self.nconst > 0 and self.rng.random() < 0.3:
                return ("c", int(self.rng.integers(0, self.nconst)))
        return ("x",)

    def expr(self, depth):
        p_leaf = 0.15 + 0.85 * (depth / self.max_depth) ** 2
        if depth >= self.max_depth or (depth > 0 and self.rng.random() < p_leaf):
            return self.leaf()
        if self.rng.random() < 0.65:
            op = _BIN[int(self.rng.integers(0, 4))]
            return (op, self.expr(depth + 1), self.expr(depth + 1))
        op = _UN[int(self.rng.integers(0, 4))]
        if op == "pow":
            return ("pow", self.expr(depth + 1), int(self.rng.integers(2, 4)))
        return (op, self.expr(depth + 1))


def _expr_text(e, names=None) -> str:
    """Program text of a generator tree; guarded operands are let-bound once."""
    if names is None:
        names = [0]

    def fresh():
        names[0] += 1
        return f"g{names[0]}"

    k = e[0]
    if k == "x":
        return "x"
    if k == "c":
        return f"t{e[1]}"
    if k in ("+", "-", "*"):
        return f"({k} {_expr_text(e[1], names)} {_expr_text(e[2], names)})"
    if k == "/":
        a = _expr_text(e[1], names)
        d = _expr_text(e[2], names)
        v = fresh()
        return f"(let (({v} {d})) (/ {a} (+ 1.0 (* {v} {v}))))"
    if k == "exp":
        a = _expr_text(e[1], names)
        v = fresh()
        return f"(let (({v} {a})) (exp (/ {v} (+ 1.0 (* {v} {v})))))"
    if k == "log":
        a = _expr_text(e[1], names)
        v = fresh()
        return f"(let (({v} {a})) (log (abs (+ 1.0 (* {v} {v})))))"
    if k == "sin":
        return f"(sin {_expr_text(e[1], names)})"
    if k == "pow":
        return f"(pow {_expr_text(e[1], names)} {e[2]})"
    raise ValueError(k)


def _expr_eval(e, x, th, guard):
    """numpy evaluation of the generator's own tree (data synthesis only)."""
    k = e[0]
    if k == "x":
        v = x
    elif k == "c":
        v = th[..., e[1]][..., None] * np.ones_like(x)
    elif k in _BIN:
        a = _expr_eval(e[1], x, th, guard)
        b = _expr_eval(e[2], x, th, guard)
        if k == "+":
            v = a + b
        elif k == "-":
            v = a - b
        elif k == "*":
            v = a * b
        else:
            v = a / (1.0 + b * b)
    elif k == "exp":
        a = _expr_eval(e[1], x, th, guard)
        v = np.exp(a / (1.0 + a * a))
    elif k == "log":
        a = _expr_eval(e[1], x, th, guard)
        v = np.log(np.abs(1.0 + a * a))
    elif k == "sin":
        v = np.sin(_expr_eval(e[1], x, th, guard))
    elif k == "pow":
        v = _expr_eval(e[1], x, th, guard) ** e[2]
    else:
        raise ValueError(k)
    guard.append(float(np.max(np.abs(v))) if v.size else 0.0)
    return v


def _uses_x(e) -> bool:
    if e[0] == "x":
        return True
    if e[0] == "c":
        return False
    return any(_uses_x(s) for s in e[1:] if isinstance(s, tuple))


def _size(e) -> int:
    if e[0] in ("x", "c"):
        return 1
    return 1 + sum(_size(s) for s in e[1:] if isinstance(s, tuple))


def random_program(rng, n_points: int, max_depth: int = 6, max_consts: int = 8,
                   guard_lanes: int = 32):
    """Draw one accepted random-expression program; returns (text, tree, theta*, x, y)."""
    while True:
        g = _Gen(rng, max_depth, max_consts)
        tree = g.expr(0)
        if g.nconst < 1 or not _uses_x(tree) or _size(tree) < 4:
            continue
        P = g.nconst
        theta = rng.uniform(-2.0, 2.0, P)
        x = rng.uniform(-2.0, 2.0, n_points)
        lanes = theta + rng.normal(0.0, 0.3, (guard_lanes, P))
        with np.errstate(all="ignore"):
            guard = []
            f_star = _expr_eval(tree, x[None, :], theta[None, :], guard)[0]
            _expr_eval(tree, x[None, :], lanes, guard)
        if not all(np.isfinite(guard)) or max(guard) > 1e4:
            continue
        y = f_star + rng.normal(0.0, 0.05, n_points)
        names = " ".join(f"t{k}" for k in range(P))
        body = _expr_text(tree)
        text = (
            ";; random expression program, mean squared error over the data axis\n"
            f"(model (params {names})\n"
            f"  (/ (data-sum {n_points} 2\n"
            f"       (let* ((x (dobs 0)) (r (- {body} (dobs 1))))\n"
            "         (* r r)))\n"
            f"     {_fmt(float(n_points))}))\n"
        )
        return text, tree, theta, x, y


def random_exprs(n_programs: int = 200, B: int = 4096, n_points: int = 256, seed: int = 1234,
                 max_depth: int = 6):
    """List of Workloads (one per program)."""
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n_programs):
        text, tree, theta, x, y = random_program(rng, n_points, max_depth=max_depth)
        obs = np.empty(2 * n_points)
        obs[0::2] = x
        obs[1::2] = y
        params = theta + rng.normal(0.0, 0.3, (B, theta.size))
        out.append(Workload(f"random_expr_{i}", text, FRONTEND_SCHEME, params, obs, theta,
                            {"n_points": n_points, "tree_size": _size(tree)}))
    return out


# --------------------------------------------------------------------------
# 3. logistic growth, stack bytecode (section 7's second client)
# --------------------------------------------------------------------------
# ---------------------------------------------------------------- control-flow fuzz programs
# Seeded Scheme programs over the surface a program search explores (section 6's
# fuzzer: let, let*, per-lane if, bounded named-let loops, data sums), with the same
# domain guards as the random expressions.  Text only: no arithmetic of the method.

class _CtlGen:
    def __init__(self, rng, n_params: int, n_points: int):
        self.rng, self.P, self.N = rng, n_params, n_points
        self.vars = 0

    def fresh(self):
        self.vars += 1
        return f"v{self.vars}"

    def const(self):
        return _fmt(float(np.round(self.rng.uniform(-2, 2), 3)))

    def leaf(self, env):
        r = self.rng.random()
        if env and r < 0.45:
            return env[self.rng.integers(len(env))]
        if r < 0.8:
            return f"p{self.rng.integers(self.P)}"
        return self.const()

    def expr(self, d, env, in_sum=False):
        if d <= 0:
            return "(dobs 0)" if in_sum and self.rng.random() < 0.4 else self.leaf(env)
        k = self.rng.integers(11)
        e = lambda: self.expr(d - 1, env, in_sum)
        if k <= 2:
            op = ["+", "-", "*"][k]
            return f"({op} {e()} {e()})"
        if k == 3:
            a = e()
            return f"(/ {e()} (+ 1.0 (* {a} {a})))"
        if k == 4:
            a = e()
            return f"(exp (/ {a} (+ 1.0 (* {a} {a}))))"
        if k == 5:
            a = e()
            return f"(log (+ 1.0 (* {a} {a})))"
        if k == 6:
            return f"({['sin', 'cos', 'tanh'][self.rng.integers(3)]} {e()})"
        if k == 7:
            cmp = ["<", ">", "<=", ">="][self.rng.integers(4)]
            return f"(if ({cmp} {e()} {e()}) {e()} {e()})"
        if k == 8:
            v = self.fresh()
            return f"(let (({v} {e()})) {self.expr(d - 1, env + [v], in_sum)})"
        if k == 9:
            v1, v2 = self.fresh(), self.fresh()
            b1 = e()
            b2 = self.expr(d - 1, env + [v1], in_sum)
            return f"(let* (({v1} {b1}) ({v2} {b2})) {self.expr(d - 1, env + [v1, v2], in_sum)})"
        # bounded loop: a contraction keeps the accumulator in range
        acc, i = self.fresh(), self.fresh()
        n = int(self.rng.integers(2, 5))
        step = self.expr(d - 1, env + [acc], in_sum)
        return f"(let lp (({i} 0) ({acc} {e()})) (if (= {i} {n}) {acc} (lp (+ {i} 1) (* 0.5 (+ {acc} (tanh {step}))))))"


def control_program(rng, n_params: int = 3, n_points: int = 16, depth: int = 4) -> str:
    g = _CtlGen(rng, n_params, n_points)
    params = " ".join(f"p{k}" for k in range(n_params))
    lane = g.expr(depth, [])
    body = g.expr(depth - 1, [], in_sum=True)
    return (f"(model (params {params})\n  (+ {lane}\n     (* {_fmt(1.0 / n_points)} "
            f"(data-sum {n_points} 1 0 (let ((r (- {body} (dobs 0)))) (* r r))))))")


def control_fuzz(n_programs: int = 40, B: int = 96, n_params: int = 3, n_points: int = 16,
                 seed: int = 1234) -> list:
    """Control-flow fuzz programs: a lane-level term and a squared-residual data sum."""
    rng = np.random.default_rng(seed)
    out = []
    for i in range(n_programs):
        text = control_program(rng, n_params, n_points)
        obs = rng.uniform(-2, 2, n_points)
        params = rng.normal(0.0, 1.0, (B, n_params))
        out.append(Workload(f"control_{i}", text, FRONTEND_SCHEME, params, obs, np.zeros(n_params),
                            {"n_points": n_points}))
    return out


# ---------------------------------------------------------------- second-client workloads
# The four bytecode workloads of section 7's second client, written for this VM:
# W1 a scalar closed-form expression, W2 a counted loop, W3 a data-independent
# conditional (a lane mask whose predicate compares constants, so every lane takes
# the same side), W4 a small summed matrix-vector product.  Each is fitted by
# squared error to seeded observations.

def bytecode_w1(n_obs: int = 8) -> str:
    lines = ["; W1: y = a exp(-b t) + c sin(t), squared error at t = 0.5, 1.0, ...", "PUSH 0.0", "STORE 0"]
    for k in range(n_obs):
        t = _fmt(0.5 * (k + 1))
        lines += ["PARAM 0", f"PUSH -{t}", "PARAM 1", "MUL", "EXP", "MUL", "PARAM 2", f"PUSH {t}", "SIN", "MUL",
                  "ADD", "OBSN", "SUB", "DUP", "MUL", "LOAD 0", "ADD", "STORE 0"]
    return "\n".join(lines + ["LOAD 0"]) + "\n"


def bytecode_w2(steps: int = 40, every: int = 10) -> str:
    lines = ["; W2: x' = a - b x by explicit Euler (dt 0.05), squared error every 10 steps",
             "PUSH 0.0", "STORE 0", "PUSH 0.0", "STORE 1", f"LOOP {steps // every}", f"  LOOP {every}",
             "    LOAD 0", "    PARAM 0", "    PARAM 1", "    LOAD 0", "    MUL", "    SUB", "    PUSH 0.05", "    MUL",
             "    ADD", "    STORE 0", "  END", "  LOAD 0", "  OBSN", "  SUB", "  DUP", "  MUL", "  LOAD 1", "  ADD",
             "  STORE 1", "END", "LOAD 1"]
    return "\n".join(lines) + "\n"


def bytecode_w3(n_obs: int = 6) -> str:
    lines = ["; W3: a branch on a data-independent test (1 < 2): every lane takes the first side",
             "PUSH 0.0", "STORE 0"]
    for k in range(n_obs):
        t = _fmt(0.25 * (k + 1))
        lines += ["PUSH 1.0", "PUSH 2.0", "LT",
                  "PARAM 0", f"PUSH {t}", "MUL", "PARAM 1", "ADD", "TANH",      # taken side
                  "PARAM 1", f"PUSH {t}", "MUL", "EXP",                          # side not taken
                  "SEL", "OBSN", "SUB", "DUP", "MUL", "LOAD 0", "ADD", "STORE 0"]
    return "\n".join(lines + ["LOAD 0"]) + "\n"


def bytecode_w4(n: int = 4, reps: int = 3) -> str:
    lines = [f"; W4: sum of (A x) over {reps} observed vectors x, A = {n}x{n} parameters (row-major)",
             "PUSH 0.0", "STORE 0"]
    for r in range(reps):
        lines += ["PUSH 0.0", "STORE 1"]
        for i in range(n):
            lines += [f"PARAM {i * n + j}" for j in range(n)]
            lines += [f"OBS {r * (n + 1) + j}" for j in range(n)]
            lines += [f"DOT {n}", "LOAD 1", "ADD", "STORE 1"]
        lines += ["LOAD 1", f"OBS {r * (n + 1) + n}", "SUB", "DUP", "MUL", "LOAD 0", "ADD", "STORE 0"]
    return "\n".join(lines + ["LOAD 0"]) + "\n"


def second_client(B: int = 256, seed: int = 1234) -> list:
    """W1-W4 with seeded observations and lanes around the generating parameters."""
    rng = np.random.default_rng(seed)
    out = []
    t1 = 0.5 * np.arange(1, 9)
    th1 = np.array([1.2, 0.7, 0.4])
    obs1 = th1[0] * np.exp(-th1[1] * t1) + th1[2] * np.sin(t1) + rng.normal(0, 0.02, 8)
    out.append(("W1", bytecode_w1(8), th1, obs1))
    th2 = np.array([1.0, 0.8])
    x, obs2 = 0.0, []
    for s in range(40):
        x = x + 0.05 * (th2[0] - th2[1] * x)
        if (s + 1) % 10 == 0:
            obs2.append(x + rng.normal(0, 0.01))
    out.append(("W2", bytecode_w2(40, 10), th2, np.array(obs2)))
    t3 = 0.25 * np.arange(1, 7)
    th3 = np.array([0.9, -0.2])
    out.append(("W3", bytecode_w3(6), th3, np.tanh(th3[0] * t3 + th3[1]) + rng.normal(0, 0.02, 6)))
    th4 = rng.normal(0, 1, 16)
    xs = rng.normal(0, 1, (3, 4))
    obs4 = np.concatenate([np.append(x_, (th4.reshape(4, 4) @ x_).sum() + rng.normal(0, 0.05)) for x_ in xs])
    out.append(("W4", bytecode_w4(4, 3), th4, obs4))
    return [Workload(name, text, FRONTEND_BYTECODE, theta + rng.normal(0, 0.2, (B, theta.size)), obs, theta, {})
            for name, text, theta, obs in out]


def logistic_bytecode(n_obs: int = 100, every: int = 10, dt: float = 0.01, x0: float = 0.1) -> str:
    lines = [
        "; logistic growth dx/dt = r x (1 - x/K), explicit Euler; MSE against observations",
        "PARAM 0", "STORE 0            ; r",
        "PARAM 1", "STORE 1            ; K",
        f"PUSH {_fmt(x0)}", "STORE 2            ; x",
        "PUSH 0.0", "STORE 3            ; squared-error accumulator",
        f"LOOP {n_obs}",
        f"  LOOP {every}",
        "    LOAD 2", "    LOAD 0", "    LOAD 2", "    MUL            ; r x",
        "    PUSH 1.0", "    LOAD 2", "    LOAD 1", "    DIV            ; x / K",
        "    SUB            ; 1 - x/K", "    MUL            ; r x (1 - x/K)",
        f"    PUSH {_fmt(dt)}", "    MUL", "    ADD            ; x + dt f(x)", "    STORE 2",
        "  END",
        "  LOAD 3", "  LOAD 2", "  OBSN", "  SUB", "  DUP", "  MUL", "  ADD", "  STORE 3",
        "END",
        "LOAD 3", f"PUSH {_fmt(float(n_obs))}", "DIV",
    ]
    return "\n".join(lines) + "\n"


def logistic(B: int = 16384, n_obs: int = 100, every: int = 10, seed: int = 1234) -> Workload:
    rng = np.random.default_rng(seed)
    truth = np.array([0.8, 1.0])
    dt, x = 0.01, 0.1
    ys = []
    for _ in range(n_obs):
        for _ in range(every):
            x = x + dt * (truth[0] * x * (1.0 - x / truth[1]))
        ys.append(x)
    obs = np.array(ys) + rng.normal(0.0, 0.01, n_obs)
    params = truth * np.exp(0.25 * rng.normal(0.0, 1.0, (B, 2)))
    return Workload("logistic", logistic_bytecode(n_obs, every, dt), FRONTEND_BYTECODE, params, obs,
                    truth, {"steps": n_obs * every, "n_obs": n_obs})


# --------------------------------------------------------------------------
# 4/5. Kalman filter negative log-likelihood (prediction-error decomposition)
# --------------------------------------------------------------------------
def _matrix_text(M) -> str:
    r, c = M.shape
    el = " ".join(_fmt(v) for v in M.reshape(-1))
    return f"(matrix {r} {c} {el})"


_KALMAN_LOOP = """(define (kalman-nll Q R P0 T)
  (let loop ((t 0) (x (zeros {n} 1)) (P P0) (nll 0.0))
    (if (= t T)
        nll
        (let* ((xp (matmul F x))
               (Pp (m+ (matmul (matmul F P) (transpose F)) Q))
               (v (m- (obs-vec (* {m} t) {m}) (matmul H xp)))
               (PHt (matmul Pp (transpose H)))
               (S (m+ (matmul H PHt) R))
               (Si (inv S))
               (K (matmul PHt Si))
               (xn (m+ xp (matmul K v)))
               (Pn (m- Pp (matmul K (matmul H Pp))))
               (term (* 0.5 (+ (logdet S) (mref (matmul (transpose v) (matmul Si v)) 0 0) {c}))))
          (loop (+ t 1) xn Pn (+ nll term))))))
"""


def _simulate_lgssm(rng, F, H, Q, R, P0, T):
    n = F.shape[0]
    x = rng.multivariate_normal(np.zeros(n), P0)
    ys = []
    for _ in range(T):
        x = F @ x + rng.multivariate_normal(np.zeros(n), Q)
        ys.append(H @ x + rng.multivariate_normal(np.zeros(H.shape[0]), R))
    return np.concatenate(ys)


def kalman_cv4(B: int = 8192, T: int = 200, seed: int = 1234) -> Workload:
    """4-state constant-velocity model (px, py, vx, vy), dt = 1, 2-d position observations."""
    rng = np.random.default_rng(seed)
    F = np.array([[1, 0, 1, 0], [0, 1, 0, 1], [0, 0, 1, 0], [0, 0, 0, 1]], dtype=float)
    H = np.array([[1, 0, 0, 0], [0, 1, 0, 0]], dtype=float)
    truth = np.log(np.array([0.5, 0.4, 1.0, 0.8]))
    qx, qy, rx, ry = np.exp(2 * truth)
    Q = np.array([[qx / 3, 0, qx / 2, 0], [0, qy / 3, 0, qy / 2], [qx / 2, 0, qx, 0], [0, qy / 2, 0, qy]])
    R = np.diag([rx, ry])
    P0 = 10.0 * np.eye(4)
    obs = _simulate_lgssm(rng, F, H, Q, R, P0, T)
    params = truth + rng.normal(0.0, 0.5, (B, 4))
    m = 2
    program = (
        ";; 4-state constant-velocity Kalman filter, Gaussian negative log-likelihood\n"
        f"(define F {_matrix_text(F)})\n"
        f"(define H {_matrix_text(H)})\n"
        + _KALMAN_LOOP.format(n=4, m=m, c=_fmt(m * math.log(2 * math.pi)))
        + "(model (params lqx lqy lrx lry)\n"
        "  (let* ((qx (exp (* 2.0 lqx))) (qy (exp (* 2.0 lqy)))\n"
        "         (rx (exp (* 2.0 lrx))) (ry (exp (* 2.0 lry)))\n"
        "         (Q (matrix 4 4 (/ qx 3.0) 0 (/ qx 2.0) 0\n"
        "                        0 (/ qy 3.0) 0 (/ qy 2.0)\n"
        "                        (/ qx 2.0) 0 qx 0\n"
        "                        0 (/ qy 2.0) 0 qy))\n"
        "         (R (matrix 2 2 rx 0 0 ry)))\n"
        f"    (kalman-nll Q R (mscale 10.0 (identity 4)) {T})))\n"
    )
    return Workload("kalman_cv4", program, FRONTEND_SCHEME, params, obs, truth, {"T": T, "n": 4, "m": m})


def random_stable_matrix(rng, n: int, radius: float = 0.95) -> np.ndarray:
    A = rng.normal(0.0, 1.0, (n, n))
    rho = float(np.max(np.abs(np.linalg.eigvals(A))))
    return A * (radius / rho)


def kalman_rand8(B: int = 65536, T: int = 1000, seed: int = 1234, n: int = 8, m: int = 3) -> Workload:
    """n-state linear-Gaussian model, random transition with spectral radius 0.95, H = [I_m 0]."""
    rng = np.random.default_rng(seed)
    F = random_stable_matrix(rng, n)
    H = np.zeros((m, n))
    H[:, :m] = np.eye(m)
    truth = np.concatenate([np.log(rng.uniform(0.1, 0.3, n)), np.log(np.full(m, 0.5)), [0.0]])
    Q = np.diag(np.exp(2 * truth[:n]))
    R = np.diag(np.exp(2 * truth[n:n + m]))
    P0 = np.exp(2 * truth[-1]) * np.eye(n)
    obs = _simulate_lgssm(rng, F, H, Q, R, P0, T)
    params = truth + rng.normal(0.0, 0.5, (B, n + m + 1))
    qn = " ".join(f"lq{i}" for i in range(n))
    rn = " ".join(f"lr{i}" for i in range(m))
    qdiag = []
    for i in range(n):
        row = ["0"] * n
        row[i] = f"(exp (* 2.0 lq{i}))"
        qdiag.append(" ".join(row))
    rdiag = []
    for i in range(m):
        row = ["0"] * m
        row[i] = f"(exp (* 2.0 lr{i}))"
        rdiag.append(" ".join(row))
    program = (
        f";; {n}-state random stable Kalman filter, {m}-d observations, Gaussian negative log-likelihood\n"
        f"(define F {_matrix_text(F)})\n"
        f"(define H {_matrix_text(H)})\n"
        + _KALMAN_LOOP.format(n=n, m=m, c=_fmt(m * math.log(2 * math.pi)))
        + f"(model (params {qn} {rn} lp0)\n"
        f"  (kalman-nll (matrix {n} {n} " + "\n      ".join(qdiag) + ")\n"
        f"              (matrix {m} {m} " + " ".join(rdiag) + ")\n"
        f"              (mscale (exp (* 2.0 lp0)) (identity {n}))\n"
        f"              {T}))\n"
    )
    return Workload(f"kalman_rand{n}", program, FRONTEND_SCHEME, params, obs, truth,
                    {"T": T, "n": n, "m": m, "F": F})


def kalman_highd(B: int = 1024, D: int = 64, m: int = 8, T: int = 50, seed: int = 1234) -> Workload:
    """A population of D-dimensional Kalman-filter likelihoods with shared dynamics,
    observation map and observations, differing in their noise parameters (the
    appendix's dense-numeric GPU workload, here with gradients): random transition
    with spectral radius 0.95, H = [I_m 0], Q = exp(2 lq) I, R = exp(2 lr) I,
    P0 = exp(2 lp0) I."""
    rng = np.random.default_rng(seed)
    F = random_stable_matrix(rng, D)
    H = np.zeros((m, D))
    H[:, :m] = np.eye(m)
    truth = np.array([np.log(0.2), np.log(0.5), 0.0])
    Q = np.exp(2 * truth[0]) * np.eye(D)
    R = np.exp(2 * truth[1]) * np.eye(m)
    P0 = np.exp(2 * truth[2]) * np.eye(D)
    obs = _simulate_lgssm(rng, F, H, Q, R, P0, T)
    params = truth + rng.normal(0.0, 0.3, (B, 3))
    program = (
        f";; {D}-state Kalman filter population, {m}-d observations, Gaussian negative log-likelihood\n"
        f"(define F {_matrix_text(F)})\n"
        f"(define H {_matrix_text(H)})\n"
        + _KALMAN_LOOP.format(n=D, m=m, c=_fmt(m * math.log(2 * math.pi)))
        + "(model (params lq lr lp0)\n"
        f"  (kalman-nll (mscale (exp (* 2.0 lq)) (identity {D}))\n"
        f"              (mscale (exp (* 2.0 lr)) (identity {m}))\n"
        f"              (mscale (exp (* 2.0 lp0)) (identity {D}))\n"
        f"              {T}))\n"
    )
    return Workload(f"kalman_highd{D}", program, FRONTEND_SCHEME, params, obs, truth,
                    {"T": T, "n": D, "m": m, "F": F})


def config(i: int, **kw):
    """Workload(s) of the five configurations at their full sizes (or overridden sizes)."""
    if i == 1:
        return exp_decay(**kw)
    if i == 2:
        return random_exprs(**kw)
    if i == 3:
        return logistic(**kw)
    if i == 4:
        return kalman_cv4(**kw)
    if i == 5:
        return kalman_rand8(**kw)
    if i == 6:
        return kalman_highd(**kw)
    raise ValueError(i)
