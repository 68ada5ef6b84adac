"""Control-flow fuzzing (GPU): seeded programs over let, let*, per-lane if, bounded
named-let loops and data sums, replayed on the GPU and compared with the oracle lane by
lane (1e-12, the comparison rule in conftest.rel_check), plus lane decomposition: a
lane replayed alone gives the batched result bit for bit (section 3.5: lanes share
nothing)."""
import numpy as np
import pytest

import workloads as W
from conftest import oracle_ref, rel_check

pytestmark = pytest.mark.gpu

PROGRAMS = W.control_fuzz(n_programs=40, B=96, seed=77)


def _gpu(nd, tape, params, obs):
    import torch
    p = torch.tensor(params, device="cuda")
    o = torch.tensor(obs, device="cuda")
    loss, grad = nd.value_and_grad(tape, p, o)
    torch.cuda.synchronize()
    return loss.cpu().numpy(), grad.cpu().numpy()


@pytest.mark.parametrize("k", range(len(PROGRAMS)))
def test_fuzz_program_matches_oracle(ndvm, oracle_mod, cuda, k):
    w = PROGRAMS[k]
    tape = ndvm.trace_build(w.program, w.frontend)
    gl, gg = _gpu(ndvm, tape, w.params, w.obs)
    ol, og, sp = oracle_ref(oracle_mod, w.program, w.params, w.obs, frontend=w.frontend)
    ok, rep = rel_check(gl, gg, ol, og, 1e-12, sp)
    assert ok, rep


@pytest.mark.parametrize("k", [0, 7, 19])
def test_fuzz_lane_decomposition(ndvm, cuda, k):
    w = PROGRAMS[k]
    tape = ndvm.trace_build(w.program, w.frontend)
    bl, bg = _gpu(ndvm, tape, w.params, w.obs)
    for b in (0, 31, 95):
        sl, sg = _gpu(ndvm, tape, w.params[b:b + 1], w.obs)
        np.testing.assert_array_equal(sl[0], bl[b])
        np.testing.assert_array_equal(sg[0], bg[b])
