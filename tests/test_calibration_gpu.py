"""Calibration through the PyTorch op: the replay as a differentiable op drives an
Adam maximum-likelihood fit of the 4-state Kalman model, and the trajectory equals the
one driven by the oracle's gradients (the paper's Kalman MLE calibration, section 6,
run here over a population of starting points).

Tolerance: with gradients perturbed by 1e-12 relative noise (the parity bound), the
30-step Adam trajectories of this problem move by about 7e-12 (measured with the
oracle alone); 1e-9 absolute leaves a factor 100.
"""
import numpy as np
import pytest

import workloads as W

pytestmark = pytest.mark.gpu

STEPS, LR, B1, B2, EPS = 30, 0.05, 0.9, 0.999, 1e-8


def adam(theta, grad_fn):
    """Adam written out (the same update on both sides); returns the trajectory and losses."""
    m, v = np.zeros_like(theta), np.zeros_like(theta)
    traj, losses = [theta.copy()], []
    for t in range(1, STEPS + 1):
        loss, g = grad_fn(theta)
        losses.append(loss)
        m = B1 * m + (1 - B1) * g
        v = B2 * v + (1 - B2) * g * g
        theta = theta - LR * (m / (1 - B1 ** t)) / (np.sqrt(v / (1 - B2 ** t)) + EPS)
        traj.append(theta.copy())
    return np.array(traj), np.array(losses)


def test_op_backward_is_the_replay_gradient(ndvm, cuda):
    import torch
    w = W.kalman_cv4(B=24, T=15)
    tape = ndvm.trace_build(w.program, w.frontend)
    obs = torch.tensor(w.obs, device="cuda")
    p = torch.tensor(w.params, device="cuda", requires_grad=True)
    op = ndvm.loss_op(tape)
    loss = op(p, obs)
    (loss * torch.arange(1, 25, device="cuda", dtype=torch.float64)).sum().backward()
    ref_loss, ref_grad = ndvm.value_and_grad(tape, p.detach().contiguous(), obs)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(loss.detach().cpu().numpy(), ref_loss.cpu().numpy())
    scale = np.arange(1, 25, dtype=np.float64)[:, None]
    np.testing.assert_array_equal(p.grad.cpu().numpy(), scale * ref_grad.cpu().numpy())


def test_adam_calibration_matches_oracle_trajectory(ndvm, oracle_mod, cuda):
    import torch
    w = W.kalman_cv4(B=16, T=30)
    tape = ndvm.trace_build(w.program, w.frontend)
    obs = torch.tensor(w.obs, device="cuda")
    op = ndvm.loss_op(tape)

    def gpu_grad(theta):
        p = torch.tensor(theta, device="cuda", requires_grad=True)
        loss = op(p, obs)
        loss.sum().backward()
        return loss.detach().cpu().numpy(), p.grad.cpu().numpy()

    def oracle_grad(theta):
        return oracle_mod.run(w.program, theta, w.obs, frontend=w.frontend, nthreads=8)

    tg, lg = adam(w.params.copy(), gpu_grad)
    to, lo = adam(w.params.copy(), oracle_grad)
    assert (lo[-1] < lo[0]).all()  # the fit makes progress on every lane
    np.testing.assert_allclose(lg, lo, rtol=1e-10, atol=0)
    assert np.abs(tg - to).max() <= 1e-9, np.abs(tg - to).max()
