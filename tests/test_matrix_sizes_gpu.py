"""Inverse, determinant and log-determinant of every supported size (n = 1..8) on the GPU:
closed forms to 3 x 3, Gauss-Jordan elimination with partial pivoting above (with row
exchanges: one matrix is not symmetric and has a small leading element), their adjoints
(the inverse's through scratch slots), at lane counts that give the element-split kernel
1, 2, 8 and 16 threads per lane.  Sampled lanes match the oracle at 1e-12; every lane is
bit-identical across the launch shapes (each element has the same arithmetic whichever
thread of a lane's group computes it)."""
import numpy as np
import pytest

from conftest import oracle_ref, rel_check

pytestmark = pytest.mark.gpu

SIZES = [1, 2, 3, 4, 5, 6, 7, 8]
LANES = [1, 8192, 20000, 40000]


def program(n, rng):
    P = 4
    p = [f"p{i}" for i in range(P)]

    def mat(scale):
        els = []
        for _ in range(n * n):
            if rng.random() < 0.5:
                els.append(f"(* {round(float(rng.normal()) * scale, 3)} {rng.choice(p)})")
            else:
                els.append(repr(round(float(rng.normal()) * scale, 3)))
        return f"(matrix {n} {n} {' '.join(els)})"

    # M: parameter-dependent; A = M M^T + 2 I (SPD); N: not symmetric, moderately conditioned
    # (unit diagonal, small off-diagonal terms) with a tiny (0, 0) element, so that the
    # elimination exchanges rows while the 1e-12 bound still measures the arithmetic
    n_els = [f"(- (* 0.001 {p[0]}) 1.0)"] + [f"(+ {round(float(rng.normal()) * 0.15, 4)} (* 0.05 {rng.choice(p)}))"
                                             for _ in range(n * n - 1)]
    return (f"(model (params {' '.join(p)}) "
            f"(let* ((M {mat(0.7)}) (A (m+ (matmul M (transpose M)) (mscale 2.0 (identity {n})))) "
            f"(N (m+ (matrix {n} {n} {' '.join(n_els)}) (identity {n}))) "
            f"(Ai (inv A))) "
            f"(+ (logdet A) (trace Ai) (* 0.01 (det A)) (mref (matmul Ai M) 0 {n - 1}) "
            f"(* 0.1 (det N)) (trace (inv N)))))")


@pytest.mark.parametrize("n", SIZES)
def test_inverse_and_determinants_of_every_size(ndvm, oracle_mod, cuda, n):
    import torch
    rng = np.random.default_rng(1000 + n)
    prog = program(n, rng)
    tape = ndvm.trace_build(prog)
    params = rng.normal(0.0, 0.5, (max(LANES), 4))
    results = []
    for B in LANES:
        p = torch.tensor(params[:B], device=cuda)
        loss, grad = ndvm.value_and_grad(tape, p, None)
        torch.cuda.synchronize()
        results.append((loss.cpu().numpy(), grad.cpu().numpy()))
    for (l, g), B in zip(results[1:], LANES[1:]):  # the same lanes, bit for bit, at every launch shape
        k = min(B, LANES[1])
        assert np.array_equal(l[:k], results[1][0][:k]) and np.array_equal(g[:k], results[1][1][:k]), (n, B)
    assert np.array_equal(results[0][0], results[1][0][:1]) and np.array_equal(results[0][1], results[1][1][:1])
    l, g = results[-1]
    idx = np.concatenate([np.arange(40), rng.choice(len(l), 40, replace=False)])
    ol, og, sp = oracle_ref(oracle_mod, prog, params[idx], np.zeros(0))
    ok, rep = rel_check(l[idx], g[idx], ol, og, 1e-12, sp)
    assert ok, (n, rep)
