"""fp64 CPU oracle of the homogenized StackLSTM step (test infrastructure).

TEST INFRASTRUCTURE ONLY: the test suite, the smoke check and the benchmark's
CPU-baseline leg are the only users. The product library never imports, links or
runs anything here, and this package imports nothing from the product package.

``run`` wraps the plain-C oracle in ``stacklstm_oracle.c`` (one instance at a time,
explicit stack, analytic backward, fp64). ``build`` compiles it with gcc.
Modes: ``"homogenized"`` is Algorithm 1 taken literally; ``"definition"`` is the
original push/pop semantics of Sec. 2 (plus hold, Sec. 3).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from typing import Iterable, Optional

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "stacklstm_oracle.c")
_LIB_DIR = os.path.join(_HERE, "_build")
_LIB = os.path.join(_LIB_DIR, "libstacklstm_oracle.so")

MODES = {"homogenized": 0, "definition": 1}
ERRORS = {1: "bad op", 2: "stack underflow", 3: "out of memory", 4: "bad argument"}
OUTPUTS = ("p_traj", "src", "y", "h_stack", "c_stack", "dx", "dh0", "dc0", "dW", "dbias")

_lib = None


class OracleError(RuntimeError):
    def __init__(self, code: int):
        super().__init__("oracle error %d: %s" % (code, ERRORS.get(code, "?")))
        self.code = code


def build(force: bool = False) -> str:
    """Compile the oracle into a shared library (gcc, fp64, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        os.makedirs(_LIB_DIR, exist_ok=True)
        tmp = _LIB + ".%d.tmp" % os.getpid()
        subprocess.check_call(["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared",
                               "-o", tmp, _SRC, "-lm"])
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    if _lib is None:
        lib = ctypes.CDLL(build())
        dp, ip, bp = ctypes.c_void_p, ctypes.c_int, ctypes.c_void_p
        lib.oracle_stacklstm.argtypes = [ip, ip, ip, ip, ip] + [dp] * 8 + [bp] * 10 + [ip]
        lib.oracle_stacklstm.restype = ctypes.c_int
        lib.oracle_pointers.argtypes = [ip, ip, bp, bp, bp]
        lib.oracle_pointers.restype = ctypes.c_int
        _lib = lib
    return _lib


def _in(a, dtype, shape):
    if a is None:
        return None
    a = np.ascontiguousarray(a, dtype=dtype)
    if a.shape != tuple(shape):
        raise ValueError("shape %s != %s" % (a.shape, tuple(shape)))
    return a


def _ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def run(x, ops, h0, c0, W, bias, d_top_h=None, dy=None, mode: str = "homogenized",
        nthreads: int = 1, outputs: Iterable[str] = OUTPUTS) -> dict:
    """Forward (and, when gradients are requested, backward) of every instance.

    Shapes: x [T, B, I], ops [T, B] int in {-1, 0, 1}, h0/c0 [B, H], W [I+H, 4H]
    (gate column blocks i, f, g, o), bias [4H], d_top_h [B, H], dy [T, B, H].
    Returns a dict with the requested ``outputs`` (fp64 / int32 numpy arrays):
    p_traj [T+1, B], src [T+1, B] (history index of the top at each time: 0 is the
    initial state, t+1 the state written at step t), y [T, B, H], h_stack/c_stack
    [T+1, B, H] (final slot-indexed stack, never-written slots 0), dx [T, B, I],
    dh0/dc0 [B, H], dW [I+H, 4H], dbias [4H].
    """
    ops = np.ascontiguousarray(ops)
    T, B = ops.shape
    H = np.shape(h0)[1]
    I = np.shape(W)[0] - H
    if np.shape(W) != (I + H, 4 * H) or I < 1:
        raise ValueError("W must be [I+H, 4H]")
    if not np.all((ops >= -1) & (ops <= 1)):
        raise OracleError(1)
    ops8 = ops.astype(np.int8)
    args = dict(x=_in(x, np.float64, (T, B, I)), h0=_in(h0, np.float64, (B, H)),
                c0=_in(c0, np.float64, (B, H)), W=_in(W, np.float64, (I + H, 4 * H)),
                bias=_in(bias, np.float64, (4 * H,)), d_top_h=_in(d_top_h, np.float64, (B, H)),
                dy=_in(dy, np.float64, (T, B, H)))
    shapes = {"p_traj": ((T + 1, B), np.int32), "src": ((T + 1, B), np.int32),
              "y": ((T, B, H), np.float64), "h_stack": ((T + 1, B, H), np.float64),
              "c_stack": ((T + 1, B, H), np.float64), "dx": ((T, B, I), np.float64),
              "dh0": ((B, H), np.float64), "dc0": ((B, H), np.float64),
              "dW": ((I + H, 4 * H), np.float64), "dbias": ((4 * H,), np.float64)}
    outputs = tuple(outputs)
    out = {k: np.zeros(*shapes[k]) if k in outputs else None for k in OUTPUTS}
    rc = _load().oracle_stacklstm(
        T, B, I, H, MODES[mode], _ptr(args["x"]), _ptr(ops8), _ptr(args["h0"]), _ptr(args["c0"]),
        _ptr(args["W"]), _ptr(args["bias"]), _ptr(args["d_top_h"]), _ptr(args["dy"]),
        *[_ptr(out[k]) for k in OUTPUTS], int(nthreads))
    if rc != 0:
        raise OracleError(rc)
    return {k: v for k, v in out.items() if v is not None}


def pointers(ops) -> dict:
    """Pointer trajectory p_traj [T+1, B] and read provenance src [T+1, B] of every
    instance, without the cell arithmetic (same explicit stack of slot tags)."""
    ops = np.ascontiguousarray(ops)
    T, B = ops.shape
    if not np.all((ops >= -1) & (ops <= 1)):
        raise OracleError(1)
    ops8 = ops.astype(np.int8)
    p = np.zeros((T + 1, B), np.int32)
    s = np.zeros((T + 1, B), np.int32)
    rc = _load().oracle_pointers(T, B, _ptr(ops8), _ptr(p), _ptr(s))
    if rc != 0:
        raise OracleError(rc)
    return {"p_traj": p, "src": s}


def run_instances(inst, x, ops, h0, c0, W, bias, d_top_h=None, dy=None, **kw) -> dict:
    """``run`` on the instances listed in ``inst`` only (instances are independent,
    Sec. 3). Per-instance outputs come back with the batch axis restricted to ``inst``
    in the given order; dW/dbias are the sums over those instances."""
    inst = np.asarray(inst, dtype=np.int64)
    sel = lambda a, ax: None if a is None else np.take(np.asarray(a), inst, axis=ax)
    return run(sel(x, 1), sel(ops, 1), sel(h0, 0), sel(c0, 0), W, bias,
               sel(d_top_h, 0), sel(dy, 1), **kw)
