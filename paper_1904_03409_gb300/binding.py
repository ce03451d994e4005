"""Thin ctypes binding of libstacklstm.so (include/stacklstm.h).

Argument marshalling only: every computation runs in the library's CUDA kernels.
PyTorch supplies device memory and the stream. Functions keep the C names; tensors are
passed as torch tensors (device, dtype and shape are checked here, then only their data
pointers cross the boundary). If the library is missing this module raises; there is no
fallback.
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Optional

from . import build as _build

SL_FP32, SL_BF16 = 0, 1
SL_MODE_HOMOGENIZED, SL_MODE_PUSH_ONLY = 0, 1
STATUS = {0: "SL_OK", 1: "SL_ERR_ARG", 2: "SL_ERR_OP", 3: "SL_ERR_UNDERFLOW", 4: "SL_ERR_STATE",
          5: "SL_ERR_CUDA", 6: "SL_ERR_TIMEOUT", 7: "SL_ERR_UNSUPPORTED", 8: "SL_ERR_OOM"}
HEADER = os.path.join(_build.ROOT, "include", "stacklstm.h")

_lib = None


class StackLSTMError(RuntimeError):
    def __init__(self, status: int, where: str, message: str = ""):
        super().__init__("%s: %s%s" % (where, STATUS.get(status, status), (" (%s)" % message) if message else ""))
        self.status = status


def header_functions():
    """Names of the functions include/stacklstm.h declares."""
    with open(HEADER) as f:
        text = f.read()
    return sorted(set(re.findall(r"^\s*(?:const\s+)?\w+\s*\*?\s*(stacklstm_\w+)\s*\(", text, re.M)))


def load(path: Optional[str] = None):
    """Load the library (built in-tree by ``build.build()``); raise if it is missing."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or _build.LIB
    if not os.path.exists(path):
        raise RuntimeError("libstacklstm.so is not built (%s); run paper_1904_03409_gb300.build.build()" % path)
    lib = ctypes.CDLL(path)
    vp, i, i32p = ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p
    lib.stacklstm_create.argtypes = [ctypes.POINTER(vp), i, i, i, i, i, i, vp]
    lib.stacklstm_forward.argtypes = [vp] * 13
    lib.stacklstm_backward.argtypes = [vp] * 8
    lib.stacklstm_set_stream.argtypes = [vp, vp]
    lib.stacklstm_set_async.argtypes = [vp, i]
    lib.stacklstm_status.argtypes = [vp]
    lib.stacklstm_destroy.argtypes = [vp]
    lib.stacklstm_status_string.argtypes = [i]
    lib.stacklstm_status_string.restype = ctypes.c_char_p
    lib.stacklstm_set_timing.argtypes = [vp, i]
    lib.stacklstm_get_timing.argtypes = [vp, vp, vp, i]
    lib.stacklstm_pointers_noalloc.argtypes = [i, i, vp, vp, vp, vp]
    lib.stacklstm_pointers_noalloc.restype = ctypes.c_int
    lib.stacklstm_forward_group.argtypes = [i, vp, vp]
    lib.stacklstm_backward_group.argtypes = [i, vp, vp]
    lib.stacklstm_set_mode.argtypes = [vp, i]
    lib.stacklstm_steps_run.argtypes = [vp, vp]
    lib.stacklstm_plan.argtypes = [vp]
    lib.stacklstm_plan.restype = ctypes.c_char_p
    lib.stacklstm_last_error.argtypes = [vp]
    lib.stacklstm_last_error.restype = ctypes.c_char_p
    lib.stacklstm_head_create.argtypes = [ctypes.POINTER(vp), i, i, i, i, i, i, i, vp]
    lib.stacklstm_head_run.argtypes = [vp] * 21
    lib.stacklstm_head_add_h0_grads.argtypes = [vp, vp, vp]
    lib.stacklstm_head_status.argtypes = [vp]
    lib.stacklstm_head_destroy.argtypes = [vp]
    lib.stacklstm_head_last_error.argtypes = [vp]
    lib.stacklstm_head_last_error.restype = ctypes.c_char_p
    for fn in ("stacklstm_create", "stacklstm_forward", "stacklstm_backward", "stacklstm_set_stream",
               "stacklstm_set_async", "stacklstm_status", "stacklstm_destroy", "stacklstm_set_timing",
               "stacklstm_get_timing", "stacklstm_forward_group", "stacklstm_backward_group", "stacklstm_set_mode", "stacklstm_steps_run", "stacklstm_head_create", "stacklstm_head_run", "stacklstm_head_add_h0_grads",
               "stacklstm_head_status", "stacklstm_head_destroy"):
        getattr(lib, fn).restype = ctypes.c_int
    _lib = lib
    return lib


def _check(handle, st: int, where: str):
    if st != 0:
        msg = load().stacklstm_last_error(handle).decode() if handle else ""
        raise StackLSTMError(st, where, msg)


def _ptr(t, device=None, dtype=None, shape=None, name="tensor"):
    if t is None:
        return None
    import torch
    if not isinstance(t, torch.Tensor):
        raise TypeError("%s must be a torch tensor" % name)
    if not t.is_cuda or (device is not None and t.device.index != device):
        raise ValueError("%s must live on cuda:%s" % (name, device))
    if dtype is not None and t.dtype != dtype:
        raise ValueError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError("%s must have shape %s, got %s" % (name, tuple(shape), tuple(t.shape)))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    return ctypes.c_void_p(t.data_ptr())


def stacklstm_status_string(st: int) -> str:
    return load().stacklstm_status_string(int(st)).decode()


def stacklstm_create(T: int, B: int, I: int, H: int, dtype: int, device: int = 0, stream=None):
    """Create a handle. ``stream`` is a torch.cuda.Stream, a raw cudaStream_t int, or None
    (the current torch stream of ``device``)."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(device)
    raw = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
    h = ctypes.c_void_p()
    _check(None, load().stacklstm_create(ctypes.byref(h), T, B, I, H, dtype, device, ctypes.c_void_p(raw)),
           "stacklstm_create")
    return StackLSTMHandle(h, T, B, I, H, dtype, device)


class StackLSTMHandle:
    """Owns one library handle; ``destroy`` (or garbage collection) frees it."""

    def __init__(self, h, T, B, I, H, dtype, device):
        self.h, self.T, self.B, self.I, self.H, self.dtype, self.device = h, T, B, I, H, dtype, device

    @property
    def tdtype(self):
        import torch
        return torch.bfloat16 if self.dtype == SL_BF16 else torch.float32

    def destroy(self):
        if self.h is not None and _lib is not None:
            _lib.stacklstm_destroy(self.h)
        self.h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def stacklstm_set_stream(hd: StackLSTMHandle, stream):
    raw = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
    _check(hd.h, load().stacklstm_set_stream(hd.h, ctypes.c_void_p(raw)), "stacklstm_set_stream")


def stacklstm_set_async(hd: StackLSTMHandle, on: bool):
    _check(hd.h, load().stacklstm_set_async(hd.h, int(bool(on))), "stacklstm_set_async")


def stacklstm_set_mode(hd: StackLSTMHandle, mode: int):
    """SL_MODE_HOMOGENIZED (Algorithm 1) or SL_MODE_PUSH_ONLY (dead writes skipped)."""
    _check(hd.h, load().stacklstm_set_mode(hd.h, int(mode)), "stacklstm_set_mode")


def stacklstm_steps_run(hd: StackLSTMHandle) -> int:
    """Steps the step kernels ran in the last forward (T, or the most pushes of any
    instance in push-only mode)."""
    n = ctypes.c_int(0)
    _check(hd.h, load().stacklstm_steps_run(hd.h, ctypes.byref(n)), "stacklstm_steps_run")
    return n.value


def stacklstm_status(hd: StackLSTMHandle):
    _check(hd.h, load().stacklstm_status(hd.h), "stacklstm_status")


FWD_FIELDS = ("x", "ops", "h0", "c0", "W", "bias", "h_stack", "c_stack", "p_final", "p_traj", "src", "y")
BWD_FIELDS = ("d_top_h", "dy", "dx", "dh0", "dc0", "dW", "dbias")


class _FwdArgs(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in FWD_FIELDS]


class _BwdArgs(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in BWD_FIELDS]


def stacklstm_forward(hd: StackLSTMHandle, x, ops, h0, c0, W, bias, h_stack=None, c_stack=None, p_final=None,
                      p_traj=None, src=None, y=None):
    """Forward over all T steps; see include/stacklstm.h for the layout of each tensor."""
    args = _forward_ptrs(hd, x, ops, h0, c0, W, bias, h_stack, c_stack, p_final, p_traj, src, y)
    _check(hd.h, load().stacklstm_forward(hd.h, *args), "stacklstm_forward")


def _forward_ptrs(hd, x, ops, h0, c0, W, bias, h_stack=None, c_stack=None, p_final=None, p_traj=None, src=None,
                  y=None):
    import torch
    T, B, I, H, d, dt = hd.T, hd.B, hd.I, hd.H, hd.device, hd.tdtype
    return [
        _ptr(x, d, dt, (T, B, I), "x"), _ptr(ops, d, torch.int8, (T, B), "ops"), _ptr(h0, d, dt, (B, H), "h0"),
        _ptr(c0, d, torch.float32, (B, H), "c0"), _ptr(W, d, dt, (I + H, 4 * H), "W"),
        _ptr(bias, d, torch.float32, (4 * H,), "bias"), _ptr(h_stack, d, dt, (T + 1, B, H), "h_stack"),
        _ptr(c_stack, d, torch.float32, (T + 1, B, H), "c_stack"), _ptr(p_final, d, torch.int32, (B,), "p_final"),
        _ptr(p_traj, d, torch.int32, (T + 1, B), "p_traj"), _ptr(src, d, torch.int32, (T + 1, B), "src"),
        _ptr(y, d, dt, (T, B, H), "y")]


def stacklstm_backward(hd: StackLSTMHandle, d_top_h=None, dy=None, dx=None, dh0=None, dc0=None, dW=None,
                       dbias=None):
    """Backward of the last forward; gradients are overwritten."""
    args = _backward_ptrs(hd, d_top_h, dy, dx, dh0, dc0, dW, dbias)
    _check(hd.h, load().stacklstm_backward(hd.h, *args), "stacklstm_backward")


def _backward_ptrs(hd, d_top_h=None, dy=None, dx=None, dh0=None, dc0=None, dW=None, dbias=None):
    import torch
    T, B, I, H, d, f = hd.T, hd.B, hd.I, hd.H, hd.device, torch.float32
    return [_ptr(d_top_h, d, f, (B, H), "d_top_h"), _ptr(dy, d, f, (T, B, H), "dy"),
            _ptr(dx, d, f, (T, B, I), "dx"), _ptr(dh0, d, f, (B, H), "dh0"), _ptr(dc0, d, f, (B, H), "dc0"),
            _ptr(dW, d, f, (I + H, 4 * H), "dW"), _ptr(dbias, d, f, (4 * H,), "dbias")]


def _group_call(fn, hds, args, ptrs_of, Struct, fields, where):
    n = len(hds)
    handles = (ctypes.c_void_p * n)(*[hd.h for hd in hds])
    arr = (Struct * n)()
    for i, (hd, a) in enumerate(zip(hds, args)):
        for name, p in zip(fields, ptrs_of(hd, **a)):
            setattr(arr[i], name, p.value if p is not None else None)
    st = fn(n, handles, arr)
    if st != 0:
        msg = "; ".join(m for m in (load().stacklstm_last_error(hd.h).decode() for hd in hds) if m)
        raise StackLSTMError(st, where, msg)


def stacklstm_forward_group(hds, args):
    """Forward of several handles in one call (include/stacklstm.h): ``args`` holds, per
    handle, a dict of stacklstm_forward's keyword arguments."""
    _group_call(load().stacklstm_forward_group, hds, args, _forward_ptrs, _FwdArgs, FWD_FIELDS,
                "stacklstm_forward_group")


def stacklstm_backward_group(hds, args):
    """Backward of several handles in one call: ``args`` as for stacklstm_backward."""
    _group_call(load().stacklstm_backward_group, hds, args, _backward_ptrs, _BwdArgs, BWD_FIELDS,
                "stacklstm_backward_group")


def stacklstm_pointers_noalloc(ops, p_traj, src, stream=None):
    """Pointer trajectory and read provenance of an op stream without a handle and without
    any device allocation (see include/stacklstm.h). ops [T, B] int8, p_traj and src
    [T+1, B] int32, all on one CUDA device, which is made current for the call."""
    import torch
    T, B = ops.shape
    d = ops.device.index
    if stream is None:
        stream = torch.cuda.current_stream(d)
    raw = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
    if hasattr(stream, "device") and stream.device.index != d:
        raise ValueError("stream must belong to cuda:%d, the device of ops" % d)
    args = [_ptr(ops, d, torch.int8, (T, B), "ops"), _ptr(p_traj, d, torch.int32, (T + 1, B), "p_traj"),
            _ptr(src, d, torch.int32, (T + 1, B), "src")]
    with torch.cuda.device(d):  # the library launches on the current device
        st = load().stacklstm_pointers_noalloc(T, B, *args, ctypes.c_void_p(raw))
    if st != 0:
        raise StackLSTMError(st, "stacklstm_pointers_noalloc")


PHASES = ("prepass", "forward", "outputs", "backward", "dx", "dw", "fwd_setup", "bwd_setup")


def stacklstm_set_timing(hd: StackLSTMHandle, on: bool):
    """Record CUDA events around each phase of later calls; resets the totals."""
    _check(hd.h, load().stacklstm_set_timing(hd.h, int(bool(on))), "stacklstm_set_timing")


def stacklstm_get_timing(hd: StackLSTMHandle) -> dict:
    """{phase: (milliseconds, kernel launches)} accumulated since the last set_timing."""
    n = len(PHASES)
    ms = (ctypes.c_double * n)()
    ln = (ctypes.c_longlong * n)()
    _check(hd.h, load().stacklstm_get_timing(hd.h, ms, ln, n), "stacklstm_get_timing")
    return {p: (ms[i], ln[i]) for i, p in enumerate(PHASES)}


def stacklstm_plan(hd: StackLSTMHandle) -> str:
    """How the handle runs (kernels, tiles, clusters, ring depths)."""
    return load().stacklstm_plan(hd.h).decode()


def stacklstm_destroy(hd: StackLSTMHandle):
    hd.destroy()


# ------------------------------------------------------------------ parser head
class StackLSTMHeadHandle:
    """Owns one parser-head handle (stacklstm_head_*); ``destroy`` frees it."""

    def __init__(self, h, T, Tb, B, H, P, A, device):
        self.h, self.T, self.Tb, self.B, self.H, self.P, self.A, self.device = h, T, Tb, B, H, P, A, device

    def destroy(self):
        if self.h is not None and _lib is not None:
            _lib.stacklstm_head_destroy(self.h)
        self.h = None

    def __del__(self):
        try:
            self.destroy()
        except Exception:
            pass


def _check_head(handle, st: int, where: str):
    if st != 0:
        msg = load().stacklstm_head_last_error(handle).decode() if handle else ""
        raise StackLSTMError(st, where, msg)


def stacklstm_head_create(T: int, Tb: int, B: int, H: int, P: int, A: int, device: int = 0, stream=None):
    """A parser head for T transitions, a Tb-step buffer StackLSTM, B instances, hidden H,
    state P, A transitions; ``stream`` as for stacklstm_create."""
    import torch
    if stream is None:
        stream = torch.cuda.current_stream(device)
    raw = stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)
    h = ctypes.c_void_p()
    _check_head(None, load().stacklstm_head_create(ctypes.byref(h), T, Tb, B, H, P, A, device, ctypes.c_void_p(raw)),
                "stacklstm_head_create")
    return StackLSTMHeadHandle(h, T, Tb, B, H, P, A, device)


def stacklstm_head_run(hh: StackLSTMHeadHandle, y_stack, h0_stack, y_buffer, y_action, h0_action, n, L, gold, Wp,
                       dp, Wz, q, loss_rows, dy_stack, dy_buffer, dy_action, dWp, ddp, dWz, dq):
    """Loss rows and gradients of the parser head; see include/stacklstm.h for layouts."""
    import torch
    T, Tb, B, H, P, A, d = hh.T, hh.Tb, hh.B, hh.H, hh.P, hh.A, hh.device
    bf, f = torch.bfloat16, torch.float32
    args = [_ptr(y_stack, d, bf, (T, B, H), "y_stack"), _ptr(h0_stack, d, bf, (B, H), "h0_stack"),
            _ptr(y_buffer, d, bf, (Tb, B, H), "y_buffer"), _ptr(y_action, d, bf, (T, B, H), "y_action"),
            _ptr(h0_action, d, bf, (B, H), "h0_action"), _ptr(n, d, torch.int32, (B,), "n"),
            _ptr(L, d, torch.int32, (B,), "L"), _ptr(gold, d, torch.int8, (T, B), "gold"),
            _ptr(Wp, d, bf, (P, 3 * H), "Wp"), _ptr(dp, d, f, (P,), "dp"), _ptr(Wz, d, f, (A, P), "Wz"),
            _ptr(q, d, f, (A,), "q"), _ptr(loss_rows, d, f, (T, B), "loss_rows"),
            _ptr(dy_stack, d, f, (T, B, H), "dy_stack"), _ptr(dy_buffer, d, f, (Tb, B, H), "dy_buffer"),
            _ptr(dy_action, d, f, (T, B, H), "dy_action"), _ptr(dWp, d, f, (P, 3 * H), "dWp"),
            _ptr(ddp, d, f, (P,), "ddp"), _ptr(dWz, d, f, (A, P), "dWz"), _ptr(dq, d, f, (A,), "dq")]
    _check_head(hh.h, load().stacklstm_head_run(hh.h, *args), "stacklstm_head_run")


def stacklstm_head_add_h0_grads(hh: StackLSTMHeadHandle, dh0_stack=None, dh0_action=None):
    import torch
    B, H, d, f = hh.B, hh.H, hh.device, torch.float32
    _check_head(hh.h, load().stacklstm_head_add_h0_grads(hh.h, _ptr(dh0_stack, d, f, (B, H), "dh0_stack"),
                                                         _ptr(dh0_action, d, f, (B, H), "dh0_action")),
                "stacklstm_head_add_h0_grads")


def stacklstm_head_status(hh: StackLSTMHeadHandle):
    _check_head(hh.h, load().stacklstm_head_status(hh.h), "stacklstm_head_status")


def stacklstm_head_destroy(hh: StackLSTMHeadHandle):
    hh.destroy()
