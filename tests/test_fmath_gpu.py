"""Accuracy of the replay's exp, log, sin and cos (GPU, through the C ABI) in units in
the last place against the host's libm (numpy), over the full fast range and its edges."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


def replay(nd, prog, a):
    import torch
    t = nd.trace_build(prog)
    p = torch.tensor(a.reshape(-1, 1), dtype=torch.float64, device="cuda")
    loss, grad = nd.value_and_grad(t, p, None)
    torch.cuda.synchronize()
    return loss.cpu().numpy(), grad.cpu().numpy()[:, 0]


def ulps(x, ref):
    return np.abs(x - ref) / np.spacing(np.abs(ref))


def test_exp_within_two_ulp(ndvm, cuda):
    rng = np.random.default_rng(0)
    a = np.concatenate([rng.uniform(-707.9, 707.9, 400000), rng.uniform(-1, 1, 200000),
                        rng.uniform(-1e-6, 1e-6, 20000), np.linspace(-708.5, -707.5, 2001),
                        np.linspace(707.5, 708.5, 2001), [0.0, -0.0, 1e-300, -1e-300, 709.7, -745.0, -800.0, 800.0]])
    z, g = replay(ndvm, "(model (params a) (exp a))", a)
    ref = np.exp(a)
    fin = np.isfinite(ref) & (ref > 0)
    assert ulps(z[fin], ref[fin]).max() <= 2.0
    assert np.array_equal(z[~fin], ref[~fin])
    np.testing.assert_array_equal(g, z)  # d exp(a)/da = exp(a), the stored value


def test_log_within_two_ulp(ndvm, cuda):
    rng = np.random.default_rng(1)
    a = np.concatenate([np.exp(rng.uniform(-18.4, 690, 400000)), 1 + rng.uniform(-0.02, 0.02, 200000),
                        rng.uniform(0.74, 1.51, 200000), 1 + np.linspace(-1e-12, 1e-12, 2001),
                        [1.0, 2.0, 0.5, 0.75, 1.5, 1.5 - 2 ** -52, 2e-8, 1.7e308]])
    z, g = replay(ndvm, "(model (params a) (log a))", a)
    ref = np.log(a)
    nz = ref != 0
    assert ulps(z[nz], ref[nz]).max() <= 2.0
    assert np.all(z[~nz] == 0.0)
    np.testing.assert_allclose(g, 1.0 / a, rtol=1e-15)


def test_log_below_clamp_uses_the_clamp(ndvm, cuda):
    a = np.array([1e-8, 5e-9, 0.0, -3.0, 1e-300])
    z, g = replay(ndvm, "(model (params a) (log a))", a)
    assert np.all(z == np.log(1e-8)) or ulps(z, np.full(5, np.log(1e-8))).max() <= 2.0
    np.testing.assert_array_equal(g, 0.0)


def _trig_args(rng):
    k = rng.integers(-20000, 20000, 20000)
    return np.concatenate([
        rng.uniform(-32767.0, 32767.0, 300000), rng.uniform(-10, 10, 200000), rng.uniform(-1e-8, 1e-8, 20000),
        k * (np.pi / 2) + rng.uniform(-1e-6, 1e-6, 20000),  # near the zeros of sin and cos
        k * (np.pi / 64) + rng.uniform(-np.pi / 128, np.pi / 128, 20000),  # around the table points
        np.linspace(32766.0, 32769.0, 1001), -np.linspace(32766.0, 32769.0, 1001),  # the fast range's edge
        [np.pi, -np.pi, np.pi / 2, 2 * np.pi, 1e5, -3e7, 1e300, 5e-324, np.inf, -np.inf, np.nan]])


def _check_trig(z, ref):
    fin = np.isfinite(ref)
    assert np.array_equal(np.isnan(z), np.isnan(ref))
    big = np.abs(ref[fin]) > 1e-300
    assert ulps(z[fin][big], ref[fin][big]).max() <= 2.0


def test_sin_cos_within_two_ulp(ndvm, cuda):
    """sin (and its derivative, the cos that the forward sweep keeps) and cos."""
    a = _trig_args(np.random.default_rng(7))
    z, g = replay(ndvm, "(model (params a) (sin a))", a)
    _check_trig(z, np.sin(a))
    _check_trig(g, np.cos(a))
    z, g = replay(ndvm, "(model (params a) (cos a))", a)
    _check_trig(z, np.cos(a))
    _check_trig(g, -np.sin(a))
    # sin of a signed zero keeps its sign; cos of it is exactly 1
    z, _ = replay(ndvm, "(model (params a) (sin a))", np.array([0.0, -0.0]))
    assert np.array_equal(np.signbit(z), [False, True]) and np.all(z == 0.0)
    z, _ = replay(ndvm, "(model (params a) (cos a))", np.array([0.0, -0.0]))
    assert np.all(z == 1.0)
