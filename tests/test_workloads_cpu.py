"""The seeded input generators (no GPU): the same seed gives the same inputs, the shapes
and lane distributions follow the stated recipe, and the module holds none of the
method's arithmetic (it imports neither the oracle nor the replay package)."""
import os

import numpy as np
import pytest

import workloads as W

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def same(a, b):
    return a.program == b.program and a.frontend == b.frontend and np.array_equal(a.params, b.params) and \
        np.array_equal(a.obs, b.obs) and np.array_equal(a.truth, b.truth)


@pytest.mark.parametrize("cfg", [1, 3, 4, 6])
def test_configurations_are_seeded(cfg):
    small = {1: {}, 3: {"B": 256}, 4: {"B": 256}, 6: {"B": 8}}[cfg]
    assert same(W.config(cfg, **small), W.config(cfg, **small))
    a, b = W.config(cfg, seed=1, **small), W.config(cfg, seed=2, **small)
    assert not np.array_equal(a.params, b.params)


def test_random_programs_are_seeded():
    a, b = W.random_exprs(4, B=16, seed=7), W.random_exprs(4, B=16, seed=7)
    assert all(same(x, y) for x, y in zip(a, b))
    c = W.random_exprs(4, B=16, seed=8)
    assert any(x.program != y.program for x, y in zip(a, c))


def test_shapes_follow_the_recipe():
    w = W.config(1)
    assert w.params.shape == (64, 3) and w.obs.shape == (100,)
    t = w.obs[0::2]
    assert t.min() >= 0.0 and t.max() <= 5.0
    w = W.config(3)
    assert w.params.shape == (16384, 2) and w.obs.shape == (100,) and w.frontend == 1
    w = W.config(4)
    assert w.params.shape == (8192, 4) and w.obs.shape == (400,)
    w = W.config(5)
    assert w.params.shape == (65536, 12) and w.obs.shape == (3000,)
    w = W.config(6)
    assert w.params.shape == (1024, 3) and w.obs.shape == (400,)
    for w in W.random_exprs(5, B=4096):
        assert w.params.shape[0] == 4096 and 1 <= w.params.shape[1] <= 8 and w.obs.shape == (512,)
        x = w.obs[0::2]
        assert x.min() >= -2.0 and x.max() <= 2.0


def test_lane_distributions_follow_the_recipe():
    w = W.config(1)                                   # theta ~ N(1, 0.3^2)
    assert abs(w.params.mean() - 1.0) < 0.06 and abs(w.params.std() - 0.3) < 0.05
    w = W.config(3)                                   # theta* exp(0.25 N(0, 1))
    z = np.log(w.params / w.truth)
    assert abs(z.mean()) < 0.01 and abs(z.std() - 0.25) < 0.01
    w = W.config(4)                                   # theta* + N(0, 0.5^2)
    d = w.params - w.truth
    assert abs(d.mean()) < 0.02 and abs(d.std() - 0.5) < 0.01
    ds = np.concatenate([(w.params - w.truth).ravel() for w in W.random_exprs(8, B=4096)])
    assert abs(ds.std() - 0.3) < 0.01                 # theta* + N(0, 0.3^2)


def test_generators_hold_no_method_arithmetic():
    src = open(os.path.join(ROOT, "workloads", "__init__.py")).read()
    assert "import oracle" not in src and "from oracle" not in src
    assert "paper_2607_03574_gb300" not in src
