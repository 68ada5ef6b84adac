"""Divisions inside a data-axis body go through the divisor's correctly rounded
reciprocal and one correction step (and the reverse rule divides its adjoint with the
same reciprocal); outside a safe exponent range, and for zeros, infinities and NaNs, they
take the IEEE division.  Each lane here divides its own pair, so the loss is a / b and
the gradient is (1 / b, -a / b^2) as the replay computes them, compared with IEEE
arithmetic element by element."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu

PROGRAM = "(model (params a b) (data-sum 1 1 (/ (* a (dobs 0)) (* b (dobs 0)))))"


def _pairs(rng, n):
    a = rng.uniform(1, 2, n) * 2.0 ** rng.integers(-520, 520, n) * rng.choice([-1.0, 1.0], n)
    b = rng.uniform(1, 2, n) * 2.0 ** rng.integers(-520, 520, n) * rng.choice([-1.0, 1.0], n)
    special = np.array([0.0, -0.0, np.inf, -np.inf, np.nan, 5e-324, 1e-310, 2.0 ** 499, 2.0 ** 501,
                        2.0 ** -500, 2.0 ** -501, 1.0, 3.0, -7.0, 1.7976931348623157e308])
    sa, sb = np.meshgrid(special, special)
    return np.concatenate([a, sa.ravel()]), np.concatenate([b, sb.ravel()])


def test_body_division_matches_ieee(ndvm, cuda):
    import torch
    rng = np.random.default_rng(2468)
    a, b = _pairs(rng, 20000)
    tape = ndvm.trace_build(PROGRAM)
    params = torch.tensor(np.stack([a, b], 1), device=cuda)
    obs = torch.tensor([1.0], dtype=torch.float64, device=cuda)
    loss, grad = ndvm.value_and_grad(tape, params, obs)
    vloss = ndvm.forward(tape, params, obs)
    torch.cuda.synchronize()
    loss, grad, vloss = loss.cpu().numpy(), grad.cpu().numpy(), vloss.cpu().numpy()
    with np.errstate(all="ignore"):
        z = a / b
        ga = 1.0 / b
        gb = -(ga * z)
    # the value-only plan divides the same way as the gradient plan
    assert np.array_equal(loss.view(np.int64), vloss.view(np.int64)) or np.array_equal(loss, vloss, equal_nan=True)

    def ulps(x, y):
        d = np.zeros(len(x))
        neq = ~((x == y) | (np.isnan(x) & np.isnan(y)))
        xi, yi = x.view(np.int64), y.view(np.int64)
        same = np.signbit(x) == np.signbit(y)
        d[neq & same] = np.abs(xi[neq & same] - yi[neq & same])
        d[neq & ~same] = np.inf
        return d

    for name, got, want in (("a / b", loss, z), ("d/da = 1 / b", grad[:, 0], ga), ("d/db", grad[:, 1], gb)):
        # non-finite results keep their class
        assert np.array_equal(np.isnan(got), np.isnan(want)), name
        assert np.array_equal(np.isinf(got), np.isinf(want)), name
        assert np.array_equal(np.signbit(got[np.isinf(want)]), np.signbit(want[np.isinf(want)])), name
        fin = np.isfinite(want)
        d = ulps(got[fin], want[fin])
        assert d.max() <= 1, (name, d.max())
    # the quotient and the reciprocal are the correctly rounded IEEE values
    fin = np.isfinite(z)
    assert np.array_equal(loss[fin], z[fin])
    fin = np.isfinite(ga)
    assert np.array_equal(grad[fin, 0], ga[fin])
