"""Host-side sizing of the batched replay's workspace (ndvm_workspace_bytes_multi)."""
import ctypes

import workloads as W


def test_batch_workspace_is_the_aligned_sum_of_the_tapes(ndvm):
    ws = W.random_exprs(5, B=8, n_points=32, seed=3) + [W.logistic(B=4), W.kalman_cv4(B=4, T=5), W.config(1)]
    tapes = [ndvm.trace_build(w.program, w.frontend) for w in ws]
    lanes = [8, 0, 3, 1000, 5, 17, 2, 64]
    n = len(tapes)
    lib = ndvm.load()
    for dt in (ndvm.F64, ndvm.F32):
        expect = 0
        for t, b in zip(tapes, lanes):
            need = t.workspace_bytes(b, dt) if b > 0 else 0
            if need:
                expect = (expect + 255) // 256 * 256 + need
        got = lib.ndvm_workspace_bytes_multi((ctypes.c_void_p * n)(*[t.handle for t in tapes]), n,
                                             (ctypes.c_int64 * n)(*lanes), dt)
        assert got == expect, (dt, got, expect)
    # invalid arguments size nothing
    assert lib.ndvm_workspace_bytes_multi(None, 0, None, ndvm.F64) == 0
    assert lib.ndvm_workspace_bytes_multi((ctypes.c_void_p * 1)(tapes[0].handle), 1, (ctypes.c_int64 * 1)(-1),
                                          ndvm.F64) == 0
