"""Batched replay of several tapes (ndvm_value_and_grad_multi) on the GPU.

The batched call runs each tape's replay with the arguments and launch shape that a
separate ndvm_value_and_grad call gives it (same kernel body, same threads per lane), so
its losses and gradients equal the separate calls' bit for bit; they also match the
oracle under the parity rule on sampled lanes.
"""
import numpy as np
import pytest

import workloads as W
from conftest import oracle_ref, rel_check

pytestmark = pytest.mark.gpu


def _tensors(ws, cuda, dtype=None):
    import torch
    dt = dtype or torch.float64
    params = [torch.tensor(w.params, dtype=dt, device=cuda) for w in ws]
    obs = [torch.tensor(w.obs, dtype=dt, device=cuda) for w in ws]
    return params, obs


def _separate(ndvm, tapes, params, obs):
    out = [ndvm.value_and_grad(t, p, o) for t, p, o in zip(tapes, params, obs)]
    return [l.cpu().numpy() for l, _ in out], [g.cpu().numpy() for _, g in out]


def _assert_same(ref, got, names):
    for k, name in enumerate(names):
        assert np.array_equal(ref[0][k], got[0][k], equal_nan=True), (name, "loss")
        assert np.array_equal(ref[1][k], got[1][k], equal_nan=True), (name, "grad")


def test_random_programs_batched_equal_separate_calls(ndvm, oracle_mod, cuda):
    """Forty random-expression programs (shared per-point values: a copy launch and a
    derive launch ahead of the replays) at assorted lane counts, one of them empty."""
    import torch
    ws = W.random_exprs(40, B=37, n_points=64, seed=4321)
    sizes = [37, 1, 5, 64, 129, 0, 300, 37] * 5
    ws = [W.Workload(w.name, w.program, w.frontend, w.params[:1].repeat(n, 0) + 0.01 * np.arange(n)[:, None],
                     w.obs, w.truth) if n != 37 else w for w, n in zip(ws, sizes)]
    tapes = [ndvm.trace_build(w.program, w.frontend) for w in ws]
    params, obs = _tensors(ws, cuda)
    ref = _separate(ndvm, tapes, params, obs)
    loss, grad = ndvm.value_and_grad_multi(tapes, params, obs)
    torch.cuda.synchronize()
    got = ([l.cpu().numpy() for l in loss], [g.cpu().numpy() for g in grad])
    _assert_same(ref, got, [w.name for w in ws])
    for k in (0, 3, 6):
        w = ws[k]
        ol, og, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs, frontend=w.frontend)
        ok, rep = rel_check(got[0][k], got[1][k], ol, og, 1e-12, sp)
        assert ok, (w.name, rep)


def test_mixed_kernel_variants_in_one_batch(ndvm, oracle_mod, cuda):
    """Data-axis, staged scalar (logistic, workspace), element-split matrix (Kalman) and
    block-cooperative (64-state) tapes in one call: one launch per kernel variant."""
    import torch
    ws = [W.config(1), W.logistic(B=300), W.kalman_cv4(B=100, T=20), W.kalman_rand8(B=40, T=8),
          W.kalman_highd(B=3, D=32, m=8, T=2), W.random_exprs(1, B=50, n_points=40, seed=8)[0],
          W.logistic(B=7)]
    tapes = [ndvm.trace_build(w.program, w.frontend) for w in ws]
    params, obs = _tensors(ws, cuda)
    ref = _separate(ndvm, tapes, params, obs)
    before = ndvm.launch_count()
    loss, grad = ndvm.value_and_grad_multi(tapes, params, obs)
    torch.cuda.synchronize()
    launches = ndvm.launch_count() - before
    assert launches < len(ws) + 2, launches
    got = ([l.cpu().numpy() for l in loss], [g.cpu().numpy() for g in grad])
    _assert_same(ref, got, [w.name for w in ws])
    for k in (1, 2):
        w = ws[k]
        sub = slice(0, 24)
        ol, og, sp = oracle_ref(oracle_mod, w.program, w.params[sub], w.obs, frontend=w.frontend)
        ok, rep = rel_check(got[0][k][sub], got[1][k][sub], ol, og, 1e-12, sp)
        assert ok, (w.name, rep)


def test_more_tapes_than_one_launch_holds(ndvm, cuda):
    """300 small tapes (more than the 240 members of one launch) and fp32."""
    import torch
    ws = W.random_exprs(300, B=6, n_points=16, seed=77)
    tapes = [ndvm.trace_build(w.program, w.frontend) for w in ws]
    params, obs = _tensors(ws, cuda, torch.float32)
    ref = _separate(ndvm, tapes, params, obs)
    before = ndvm.launch_count()
    loss, grad = ndvm.value_and_grad_multi(tapes, params, obs)
    torch.cuda.synchronize()
    assert 3 <= ndvm.launch_count() - before <= 12
    got = ([l.cpu().numpy() for l in loss], [g.cpu().numpy() for g in grad])
    _assert_same(ref, got, [w.name for w in ws])


def test_batched_argument_errors(ndvm, cuda):
    """Invalid entries are refused on the host, naming the tape, before any launch."""
    import torch
    ws = [W.logistic(B=8), W.config(1)]
    tapes = [ndvm.trace_build(w.program, w.frontend) for w in ws]
    params, obs = _tensors(ws, cuda)
    ndvm.value_and_grad_multi(tapes, params, obs)  # uploads the tapes
    torch.cuda.synchronize()
    before = ndvm.launch_count()
    small = torch.empty(256, dtype=torch.uint8, device=cuda)
    with pytest.raises(ndvm.NdvmError, match="workspace"):
        ndvm.value_and_grad_multi(tapes, params, obs, workspace=small)
    with pytest.raises(ndvm.NdvmError, match="tape 1"):
        ndvm.value_and_grad_multi(tapes, params, [obs[0], obs[1][:3]])
    assert ndvm.launch_count() == before
