"""Reference ("oracle") evaluator for the NDVM tape-replay path -- TEST INFRASTRUCTURE.

Only the test suite, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product path (the C-ABI library, its
host tracer, planner and CUDA kernels) never imports, links or calls it, and the
two share no code.

The oracle is plain C (``ndvm_oracle.c``): a per-lane tree-walking interpreter of
the program *text* in IEEE double, with a pointer-graph reverse mode and a
dual-number forward mode (paper section 2 problem statement, section 3.4, and
Appendix C's adjoint table).  This module only builds it with gcc and marshals
numpy arrays through ctypes.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "ndvm_oracle.c")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_OUT_DIR, "libndvm_oracle.so")

MODE_VALUE, MODE_REVERSE, MODE_DUAL = 0, 1, 2
FRONTEND_SCHEME, FRONTEND_BYTECODE = 0, 1

_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fused multiply-add: identical on every host)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=gnu11", "-ffp-contract=off", "-fPIC", "-shared",
               "-Wall", "-o", tmp, _SRC, "-lm", "-lpthread"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            lib = ctypes.CDLL(build())
            f = lib.ndvm_oracle_run
            f.restype = ctypes.c_int
            f.argtypes = [ctypes.c_char_p, ctypes.c_size_t, ctypes.c_int, ctypes.c_longlong, ctypes.c_int,
                          ctypes.c_void_p, ctypes.c_longlong, ctypes.c_void_p, ctypes.c_void_p,
                          ctypes.c_void_p, ctypes.c_int, ctypes.c_int, ctypes.c_char_p,
                          ctypes.c_size_t]
            _lib = lib
    return _lib


class OracleError(RuntimeError):
    pass


def run(program: str, params, obs, *, frontend: int = FRONTEND_SCHEME, mode: int = MODE_REVERSE,
        nthreads: int = 1, f32: bool = False):
    """Evaluate every lane.  params: (B, P) float64; obs: (n_obs,) float64.

    Returns (loss[B], grad[B, P]) (grad is None in value-only mode).  f32=True evaluates
    in binary32 arithmetic (each result rounded to float; inputs rounded first).
    """
    lib = _load()
    params = np.ascontiguousarray(params, dtype=np.float64)
    if params.ndim != 2:
        raise ValueError("params must be (B, P)")
    obs = np.ascontiguousarray(obs, dtype=np.float64).reshape(-1)
    if f32:
        obs = obs.astype(np.float32).astype(np.float64)
    B, P = params.shape
    loss = np.zeros(B, dtype=np.float64)
    grad = np.zeros((B, P), dtype=np.float64) if mode != MODE_VALUE else None
    err = ctypes.create_string_buffer(1024)
    text = program.encode()
    rc = lib.ndvm_oracle_run(text, len(text), frontend, B, P,
                             params.ctypes.data, obs.size, obs.ctypes.data if obs.size else None,
                             loss.ctypes.data, grad.ctypes.data if grad is not None else None,
                             mode | (4 if f32 else 0), nthreads,
                             err, len(err))
    if rc != 0:
        raise OracleError(err.value.decode(errors="replace"))
    return loss, grad
