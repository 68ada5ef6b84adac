"""The no-allocation entry point, checked against the regular one (GPU).

ndvm_value_and_grad_noalloc is for callers that may not allocate device memory while
they run -- a service whose device memory is planned up front and must not grow, or a
host runtime that owns every allocation.  It allocates nothing: the replay's workspace
is a fixed 32 MiB scratch array inside the library, and the tape must already be
resident on the device.  These tests call it through the C ABI and compare it with
ndvm_value_and_grad, twice in a row (the array keeps the previous call's contents).
"""
import ctypes

import numpy as np
import pytest

import workloads as W

pytestmark = pytest.mark.gpu


def _noalloc(nd, tape, p, o, loss, grad):
    import torch
    lib = nd.load()
    return lib.ndvm_value_and_grad_noalloc(
        tape.handle, 0 if p.dtype == torch.float64 else 1, p.shape[0], ctypes.c_void_p(p.data_ptr()),
        ctypes.c_void_p(o.data_ptr()) if o is not None else None, 0 if o is None else o.numel(),
        ctypes.c_void_p(loss.data_ptr()), ctypes.c_void_p(grad.data_ptr()),
        ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


SCRATCH_BYTES = 32 << 20


@pytest.mark.parametrize("make", [lambda: W.logistic(B=3000), lambda: W.random_exprs(1, B=3000, n_points=256)[0]],
                         ids=["workspace-tape", "data-axis-tape"])
def test_noalloc_matches_regular_entry_point_twice(ndvm, cuda, make):
    """Two calls in a row with different inputs and lane counts (3000 lanes; then the last
    1537 lanes with every parameter scaled by 1.05 and the observations by 0.9), each
    equal bit for bit to ndvm_value_and_grad on the same inputs: the second call must
    not read what the first left in the shared scratch.  The logistic tape keeps 4,099
    values per lane, so its 3000 lanes (98 MB) run in more than one launch over the
    32 MiB scratch; the random-expression tape keeps its per-point values shared by all
    lanes (computed from the observations) at the start of the scratch."""
    import torch
    w = make()
    tape = ndvm.trace_build(w.program, w.frontend)
    assert tape.cost()["save_elems"] > 0 or tape.cost()["work_shared"] > 0
    for params, obs in ((w.params, w.obs), (w.params[-1537:] * 1.05, w.obs * 0.9)):
        B = len(params)
        p = torch.tensor(params, dtype=torch.float64, device="cuda")
        o = torch.tensor(obs, dtype=torch.float64, device="cuda")
        ref_loss, ref_grad = ndvm.value_and_grad(tape, p, o)  # also makes the tape resident
        torch.cuda.synchronize()
        loss, grad = torch.full_like(ref_loss, float("nan")), torch.full_like(ref_grad, float("nan"))
        n0 = ndvm.launch_count()
        st = _noalloc(ndvm, tape, p, o, loss, grad)
        assert st == 0, ndvm.load().ndvm_last_error()
        launches = ndvm.launch_count() - n0
        torch.cuda.synchronize()
        ndvm.check_device(tape)
        np.testing.assert_array_equal(loss.cpu().numpy(), ref_loss.cpu().numpy())
        np.testing.assert_array_equal(grad.cpu().numpy(), ref_grad.cpu().numpy())
        saves = tape.cost()["save_elems"]
        if saves and B == 3000:
            assert saves * 8 * B > SCRATCH_BYTES and launches > 1, (saves, B, launches)


def test_noalloc_refuses_instead_of_allocating(ndvm, cuda):
    import torch
    # a tape whose workspace for one block of lanes exceeds the fixed scratch:
    # 20,000 Euler steps keep about 82,000 values per lane (84 MB per 128-lane block)
    big = W.logistic(B=64, n_obs=2000)
    tape = ndvm.trace_build(big.program, big.frontend)
    p = torch.tensor(big.params, dtype=torch.float64, device="cuda")
    o = torch.tensor(big.obs, dtype=torch.float64, device="cuda")
    loss, grad = torch.empty(64, dtype=torch.float64, device="cuda"), torch.empty_like(p)
    assert _noalloc(ndvm, tape, p, o, loss, grad) == 1
    assert b"fixed scratch" in ndvm.load().ndvm_last_error()
    # a tape never used on this device is not resident: refused, nothing uploaded
    w = W.logistic(B=8)
    fresh = ndvm.trace_build(w.program, w.frontend)
    p2 = torch.tensor(w.params, dtype=torch.float64, device="cuda")
    o2 = torch.tensor(w.obs, dtype=torch.float64, device="cuda")
    l2, g2 = torch.empty(8, dtype=torch.float64, device="cuda"), torch.empty_like(p2)
    assert _noalloc(ndvm, fresh, p2, o2, l2, g2) == 1
    assert b"not resident" in ndvm.load().ndvm_last_error()
    np.testing.assert_equal(np.isfinite(p2.cpu().numpy()).all(), True)
