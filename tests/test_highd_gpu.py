"""High-dimensional Kalman populations (GPU): D-state filters up to D = 64 with shared
dynamics and observations, lanes differing in their noise parameters.  Large lanes run
block-cooperatively (one lane per block, its threads splitting every matrix
instruction).  Compared with the oracle at 1e-12 (conftest.rel_check)."""
import numpy as np
import pytest

import workloads as W
from conftest import oracle_ref, rel_check

pytestmark = pytest.mark.gpu


def _gpu(nd, w, lanes=None):
    import torch
    tape = nd.trace_build(w.program, w.frontend)
    params = w.params if lanes is None else w.params[lanes]
    p = torch.tensor(params, device="cuda")
    o = torch.tensor(w.obs, device="cuda")
    loss, grad = nd.value_and_grad(tape, p, o)
    fl = nd.forward(tape, p, o)
    torch.cuda.synchronize()
    nd.check_device(tape)
    return loss.cpu().numpy(), grad.cpu().numpy(), fl.cpu().numpy()


@pytest.mark.parametrize("D,m,T", [(12, 4, 4), (32, 8, 3), (64, 8, 2)])
def test_highd_kalman_matches_oracle(ndvm, oracle_mod, cuda, D, m, T):
    w = W.kalman_highd(B=20, D=D, m=m, T=T)
    gl, gg, fl = _gpu(ndvm, w)
    ol, og, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs)
    ok, rep = rel_check(gl, gg, ol, og, 1e-12, sp)
    assert ok, rep
    np.testing.assert_array_equal(fl, gl)


def test_highd_kalman_full_size_sampled(ndvm, oracle_mod, cuda):
    """The benchmark's configuration (D = 64, 8-d observations, T = 50, 1024 lanes),
    four sampled lanes recomputed by the oracle."""
    w = W.kalman_highd()
    gl, gg, _ = _gpu(ndvm, w)
    idx = np.array([0, 341, 682, 1023])
    ol, og, sp = oracle_ref(oracle_mod, w.program, w.params[idx], w.obs, nthreads=4)
    ok, rep = rel_check(gl[idx], gg[idx], ol, og, 1e-12, sp)
    assert ok, rep


def test_highd_block_lanes_decompose_and_chunk(ndvm, cuda):
    """Block-cooperative lanes: a lane replayed alone, or in workspace chunks of a few
    lanes, gives the batched result bit for bit."""
    import torch
    w = W.kalman_highd(B=9, D=32, m=8, T=3)
    tape = ndvm.trace_build(w.program, w.frontend)
    p = torch.tensor(w.params, device="cuda")
    o = torch.tensor(w.obs, device="cuda")
    bl, bg = ndvm.value_and_grad(tape, p, o)
    per_lane = tape.workspace_bytes(1, 0)
    cl, cg = ndvm.value_and_grad(tape, p, o, ws_bytes=2 * per_lane + 8)  # chunks of two lanes
    sl, sg = ndvm.value_and_grad(tape, p[4:5].contiguous(), o)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(cl.cpu().numpy(), bl.cpu().numpy())
    np.testing.assert_array_equal(cg.cpu().numpy(), bg.cpu().numpy())
    np.testing.assert_array_equal(sl.cpu().numpy()[0], bl.cpu().numpy()[4])
    np.testing.assert_array_equal(sg.cpu().numpy()[0], bg.cpu().numpy()[4])


def test_highd_fp32_variant(ndvm, oracle_mod, cuda):
    """fp32 replay of a 32-state population against the oracle in binary32, 1e-5."""
    import torch
    w = W.kalman_highd(B=12, D=32, m=8, T=3)
    w.params = w.params.astype(np.float32).astype(np.float64)
    tape = ndvm.trace_build(w.program, w.frontend)
    p = torch.tensor(w.params, dtype=torch.float32, device="cuda")
    o = torch.tensor(w.obs, dtype=torch.float32, device="cuda")
    gl, gg = ndvm.value_and_grad(tape, p, o)
    torch.cuda.synchronize()
    ol, og, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs, f32=True)
    ok, rep = rel_check(gl.double().cpu().numpy(), gg.double().cpu().numpy(), ol, og, 1e-5, sp)
    assert ok, rep
