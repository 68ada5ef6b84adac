"""NDVM tape replay on GB300: Python binding of the C-ABI library ``libndvm.so``.

Argument marshalling only: every step of the replay (tracing on the host, forward
sweep, reverse sweep, loss) runs inside the library; PyTorch supplies device
memory and streams.  The names follow the C ABI in ``include/ndvm.h``:

    tape = trace_build(program_text, frontend=FE_SCHEME)
    loss, grad = value_and_grad(tape, params, obs)     # params (B, P) CUDA tensor
    loss = loss_op(tape)(params, obs)                  # differentiable in params

There is no CPU fallback: if the library is missing or the device is not a CUDA
GPU, the calls raise.
"""
from __future__ import annotations

import ctypes
import os
import threading

FE_SCHEME, FE_BYTECODE = 0, 1
F64, F32 = 0, 1

STATUS = {0: "OK", 1: "INVALID_ARG", 2: "PARSE", 3: "UNSUPPORTED", 4: "SHAPE", 5: "OOM", 6: "CUDA", 7: "DEVICE_CHECK"}

_lib = None
_lock = threading.Lock()


class NdvmError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status


def library_path() -> str:
    from . import build as _b
    return _b.LIB


def load(build_if_missing: bool = True):
    """Load libndvm.so (building it first if needed and allowed)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        from . import build as _b
        path = _b.LIB
        if build_if_missing and _b._stale():
            _b.build()
        if not os.path.exists(path):
            raise NdvmError(6, f"the NDVM CUDA library is not built ({path}); run paper_2607_03574_gb300.build")
        lib = ctypes.CDLL(path)
        P, I64, I32, SZ, U64 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_size_t, ctypes.c_uint64
        sig = {
            "ndvm_trace_build": (ctypes.c_int, [ctypes.c_char_p, SZ, ctypes.c_int, ctypes.POINTER(P)]),
            "ndvm_tape_info": (ctypes.c_int, [P, ctypes.POINTER(I64), ctypes.POINTER(I32), ctypes.POINTER(I64),
                                              ctypes.POINTER(I64), ctypes.POINTER(U64)]),
            "ndvm_tape_cost": (ctypes.c_int, [P, ctypes.POINTER(ctypes.c_double), ctypes.POINTER(ctypes.c_double),
                                              ctypes.POINTER(I64), ctypes.POINTER(I32)]),
            "ndvm_tape_serialize": (ctypes.c_int, [P, P, SZ, ctypes.POINTER(SZ)]),
            "ndvm_tape_free": (None, [P]),
            "ndvm_workspace_bytes": (SZ, [P, I64, ctypes.c_int]),
            "ndvm_forward": (ctypes.c_int, [P, ctypes.c_int, I64, P, P, I64, P, P]),
            "ndvm_value_and_grad": (ctypes.c_int, [P, ctypes.c_int, I64, P, P, I64, P, P, P, SZ, P]),
            "ndvm_workspace_bytes_multi": (SZ, [P, I32, P, ctypes.c_int]),
            "ndvm_value_and_grad_multi": (ctypes.c_int, [P, I32, ctypes.c_int, P, P, P, P, P, P, P, SZ, P]),
            "ndvm_value_and_grad_host": (ctypes.c_int, [P, ctypes.c_int, I64, P, P, I64, P, P, P]),
            "ndvm_value_and_grad_noalloc": (ctypes.c_int, [P, ctypes.c_int, I64, P, P, I64, P, P, P]),
            "ndvm_value_and_grad_host_async": (ctypes.c_int, [P, ctypes.c_int, I64, P, P, I64, P, P, P]),
            "ndvm_tape_shared_work": (ctypes.c_int, [P, ctypes.POINTER(ctypes.c_double)]),
            "ndvm_check_device": (ctypes.c_int, [P]),
            "ndvm_launch_count": (ctypes.c_ulonglong, []),
            "ndvm_measure_fp64_peak": (ctypes.c_int, [ctypes.POINTER(ctypes.c_double), P]),
            "ndvm_measure_op_cost": (ctypes.c_int, [ctypes.c_int, ctypes.c_int, ctypes.POINTER(ctypes.c_double), P]),
            "ndvm_last_error": (ctypes.c_char_p, []),
            "ndvm_version": (ctypes.c_char_p, []),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _check(status: int):
    if status != 0:
        msg = load().ndvm_last_error()
        raise NdvmError(status, msg.decode(errors="replace") if msg else "")


class Tape:
    """Owning handle of an ``ndvm_tape``."""

    def __init__(self, handle):
        self._h = handle

    @property
    def handle(self):
        if not self._h:
            raise NdvmError(1, "tape already freed")
        return self._h

    def info(self) -> dict:
        lib = load()
        nn, no, ns = ctypes.c_int64(), ctypes.c_int64(), ctypes.c_int64()
        npar, h = ctypes.c_int32(), ctypes.c_uint64()
        _check(lib.ndvm_tape_info(self.handle, ctypes.byref(nn), ctypes.byref(npar), ctypes.byref(no),
                                  ctypes.byref(ns), ctypes.byref(h)))
        return {"n_nodes": nn.value, "n_params": npar.value, "n_obs": no.value, "n_slots": ns.value,
                "hash": h.value}

    def cost(self) -> dict:
        lib = load()
        wf, wr = ctypes.c_double(), ctypes.c_double()
        se, fl = ctypes.c_int64(), ctypes.c_int32()
        _check(lib.ndvm_tape_cost(self.handle, ctypes.byref(wf), ctypes.byref(wr), ctypes.byref(se),
                                  ctypes.byref(fl)))
        ws = ctypes.c_double()
        _check(lib.ndvm_tape_shared_work(self.handle, ctypes.byref(ws)))
        return {"work_fwd": wf.value, "work_rev": wr.value, "save_elems": se.value,
                "has_regions": bool(fl.value & 1), "spill": bool(fl.value & 2), "work_shared": ws.value}

    def serialize(self) -> bytes:
        lib = load()
        n = ctypes.c_size_t()
        _check(lib.ndvm_tape_serialize(self.handle, None, 0, ctypes.byref(n)))
        buf = ctypes.create_string_buffer(n.value)
        _check(lib.ndvm_tape_serialize(self.handle, buf, n.value, ctypes.byref(n)))
        return buf.raw[: n.value]

    def workspace_bytes(self, B: int, dtype: int = F64) -> int:
        return int(load().ndvm_workspace_bytes(self.handle, B, dtype))

    def free(self):
        if self._h:
            load().ndvm_tape_free(self._h)
            self._h = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


def trace_build(program: str, frontend: int = FE_SCHEME) -> Tape:
    lib = load()
    text = program.encode()
    h = ctypes.c_void_p()
    _check(lib.ndvm_trace_build(text, len(text), frontend, ctypes.byref(h)))
    return Tape(h.value)


def launch_count() -> int:
    return int(load().ndvm_launch_count())


def measure_fp64_peak(stream=None) -> float:
    """Measured FP64 FMA throughput of the current device in flop/s."""
    v = ctypes.c_double()
    _check(load().ndvm_measure_fp64_peak(ctypes.byref(v), _stream_ptr(stream) if stream is not None else None))
    return v.value


PROBES = ("dfma", "exp", "log", "sin", "cos", "sincos", "tanh", "sqrt", "div", "rcp", "pow", "log_lib", "exp_lib",
          "sin_lib", "sincos_lib")


def measure_op_cost(name: str, iters: int = 2000, stream=None) -> float:
    """Device time per call (ns, all SMs busy) of one probed function (PROBES)."""
    v = ctypes.c_double()
    _check(load().ndvm_measure_op_cost(PROBES.index(name), iters, ctypes.byref(v),
                                       _stream_ptr(stream) if stream is not None else None))
    return v.value


def _torch():
    import torch
    return torch


def _dtype_code(t) -> int:
    torch = _torch()
    if t.dtype == torch.float64:
        return F64
    if t.dtype == torch.float32:
        return F32
    raise NdvmError(1, f"unsupported dtype {t.dtype}")


def _stream_ptr(stream):
    torch = _torch()
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dev_ptr(t, name):
    if t is None:
        return None
    if not t.is_cuda:
        raise NdvmError(1, f"{name} must be a CUDA tensor (the replay has no CPU path)")
    if not t.is_contiguous():
        raise NdvmError(1, f"{name} must be contiguous")
    return ctypes.c_void_p(t.data_ptr())


def _on_stream(stream):
    """Context in which allocations belong to `stream` (the stream the replay runs on):
    torch's caching allocator then reuses a freed block only for later work on that
    stream, never while a kernel queued there may still use it."""
    torch = _torch()
    return torch.cuda.stream(stream if stream is not None else torch.cuda.current_stream())


def forward(tape: Tape, params, obs, loss=None, stream=None):
    """Per-lane loss.  params: (B, P) CUDA tensor; obs: 1-d CUDA tensor (same dtype).
    An output this call allocates belongs to `stream` (torch's allocator)."""
    torch = _torch()
    B = params.shape[0]
    if loss is None:
        with _on_stream(stream):
            loss = torch.empty(B, dtype=params.dtype, device=params.device)
    _check(load().ndvm_forward(tape.handle, _dtype_code(params), B, _dev_ptr(params, "params"),
                               _dev_ptr(obs, "obs"), 0 if obs is None else obs.numel(), _dev_ptr(loss, "loss"),
                               _stream_ptr(stream)))
    return loss


class Workspace:
    """Reusable device workspace for value_and_grad (grown on demand).  One per
    (device, stream): it is allocated on the stream its replays run on, so when it
    grows, the replaced block is not handed to other work while those replays may still
    read it."""

    def __init__(self):
        self.buf = None

    def get(self, nbytes: int, device, stream=None):
        torch = _torch()
        if nbytes == 0:
            return None
        if self.buf is None or self.buf.numel() < nbytes or self.buf.device != device:
            self.buf = None
            with _on_stream(stream):
                self.buf = torch.empty(nbytes, dtype=torch.uint8, device=device)
        return self.buf


_default_ws = {}  # (device, stream) -> Workspace: concurrent streams never share one


def value_and_grad(tape: Tape, params, obs, loss=None, grad=None, workspace=None, ws_bytes=None, stream=None):
    """Per-lane loss and gradient.  Returns (loss[B], grad[B, P]).  Outputs and the
    default workspace that this call allocates belong to `stream` (torch's allocator);
    a caller-given workspace must stay allocated until the replay on `stream` is done."""
    torch = _torch()
    B = params.shape[0]
    with _on_stream(stream):
        if loss is None:
            loss = torch.empty(B, dtype=params.dtype, device=params.device)
        if grad is None:
            grad = torch.empty_like(params)
    dt = _dtype_code(params)
    if workspace is None:
        need = tape.workspace_bytes(B, dt) if ws_bytes is None else ws_bytes
        key = (str(params.device), _stream_ptr(stream).value)
        workspace = _default_ws.setdefault(key, Workspace()).get(need, params.device, stream)
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    if ws_bytes is not None:
        nbytes = min(nbytes, ws_bytes)
    _check(load().ndvm_value_and_grad(tape.handle, dt, B, _dev_ptr(params, "params"), _dev_ptr(obs, "obs"),
                                      0 if obs is None else obs.numel(), _dev_ptr(loss, "loss"),
                                      _dev_ptr(grad, "grad"), _dev_ptr(workspace, "workspace"), nbytes,
                                      _stream_ptr(stream)))
    return loss, grad


def value_and_grad_multi(tapes, params, obs, loss=None, grad=None, workspace=None, stream=None):
    """Loss and gradient of several tapes in one batched call (ndvm_value_and_grad_multi).
    tapes: list of Tape; params[k]: (B_k, P_k) CUDA tensor; obs[k]: 1-d CUDA tensor (all of
    one dtype).  Returns (losses, grads), lists of tensors.  Outputs and the default
    workspace that this call allocates belong to `stream`."""
    torch = _torch()
    n = len(tapes)
    if not (len(params) == len(obs) == n):
        raise NdvmError(1, "tapes, params and obs must have the same length")
    if n == 0:
        return [], []
    dt = _dtype_code(params[0])
    for p in params:
        if _dtype_code(p) != dt:
            raise NdvmError(1, "every params tensor must have the same dtype")
    with _on_stream(stream):
        if loss is None:
            loss = [torch.empty(p.shape[0], dtype=p.dtype, device=p.device) for p in params]
        if grad is None:
            grad = [torch.empty_like(p) for p in params]
    Arr = ctypes.c_void_p * n
    I64A = ctypes.c_int64 * n
    th = Arr(*[t.handle for t in tapes])
    B = I64A(*[p.shape[0] for p in params])
    lib = load()
    need = lib.ndvm_workspace_bytes_multi(th, n, B, dt)
    if workspace is None:
        key = (str(params[0].device), _stream_ptr(stream).value, "multi")
        workspace = _default_ws.setdefault(key, Workspace()).get(need, params[0].device, stream)
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib.ndvm_value_and_grad_multi(
        th, n, dt, B, Arr(*[_dev_ptr(p, "params").value for p in params]),
        Arr(*[None if o is None else _dev_ptr(o, "obs").value for o in obs]),
        I64A(*[0 if o is None else o.numel() for o in obs]),
        Arr(*[_dev_ptr(l, "loss").value for l in loss]), Arr(*[_dev_ptr(g, "grad").value for g in grad]),
        _dev_ptr(workspace, "workspace"), nbytes, _stream_ptr(stream)))
    return loss, grad


def value_and_grad_noalloc(tape: Tape, params, obs, loss, grad, stream=None):
    """Loss and gradient into caller-given outputs with no device allocation (the
    library's fixed scratch array serves as workspace; the tape must already be
    resident on the device)."""
    _check(load().ndvm_value_and_grad_noalloc(tape.handle, _dtype_code(params), params.shape[0],
                                              _dev_ptr(params, "params"), _dev_ptr(obs, "obs"),
                                              0 if obs is None else obs.numel(), _dev_ptr(loss, "loss"),
                                              _dev_ptr(grad, "grad"), _stream_ptr(stream)))
    return loss, grad


def value_and_grad_host(tape: Tape, params_np, obs_np, want_grad: bool = True, stream=None):
    """Same computation through host numpy buffers (copies inside the call)."""
    import numpy as np
    dt = F32 if params_np.dtype == np.float32 else F64
    params_np = np.ascontiguousarray(params_np)
    obs_np = np.ascontiguousarray(obs_np, dtype=params_np.dtype)
    B = params_np.shape[0]
    loss = np.empty(B, dtype=params_np.dtype)
    grad = np.empty_like(params_np) if want_grad else None
    sp = None if stream is None else ctypes.c_void_p(stream.cuda_stream)
    _check(load().ndvm_value_and_grad_host(tape.handle, dt, B, params_np.ctypes.data, obs_np.ctypes.data,
                                           obs_np.size, loss.ctypes.data,
                                           grad.ctypes.data if grad is not None else None, sp))
    return loss, grad


def value_and_grad_host_async(tape: Tape, params_np, obs_np, loss_out, grad_out=None, stream=None):
    """Queue the host-buffer computation on `stream` and return: loss_out (and grad_out)
    hold the results after the stream is synchronized.  The arrays should be in
    page-locked memory (e.g. views of pinned torch tensors) and must stay alive and
    unchanged until then."""
    import numpy as np
    dt = F32 if params_np.dtype == np.float32 else F64
    for a in (params_np, obs_np, loss_out) + ((grad_out,) if grad_out is not None else ()):
        if not a.flags.c_contiguous or a.dtype != params_np.dtype:
            raise ValueError("host buffers must be C-contiguous and of the parameters' dtype")
    B = params_np.shape[0]
    if loss_out.shape != (B,) or (grad_out is not None and grad_out.shape != params_np.shape):
        raise ValueError("output shapes must be (B,) and params.shape")
    sp = None if stream is None else ctypes.c_void_p(stream.cuda_stream)
    _check(load().ndvm_value_and_grad_host_async(tape.handle, dt, B, params_np.ctypes.data, obs_np.ctypes.data,
                                                 obs_np.size, loss_out.ctypes.data,
                                                 grad_out.ctypes.data if grad_out is not None else None, sp))


_replay_fn = None


def loss_op(tape: Tape):
    """The replay as a differentiable PyTorch op (the paper exposes the evaluator as one,
    section 2): ``op(params, obs) -> loss[B]``.  Its backward returns the replay's
    per-lane gradient scaled by the incoming per-lane cotangent (the chain rule at the
    boundary); obs receive no gradient."""
    global _replay_fn
    torch = _torch()
    if _replay_fn is None:
        class _Replay(torch.autograd.Function):
            @staticmethod
            def forward(ctx, params, obs, tp):
                loss, grad = value_and_grad(tp, params.contiguous(), obs)
                ctx.save_for_backward(grad)
                return loss

            @staticmethod
            def backward(ctx, gloss):
                (grad,) = ctx.saved_tensors
                return grad * gloss.unsqueeze(1), None, None

        _replay_fn = _Replay.apply
    return lambda params, obs: _replay_fn(params, obs, tape)


def check_device(tape: Tape):
    _check(load().ndvm_check_device(tape.handle))
