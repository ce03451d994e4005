"""Comparison of the CUDA path's results with the oracle's.

Integer results (pointer trajectories, read provenance, final pointers) must match
bit for bit. Floats: fp32 path max-abs error <= 1e-4; bf16 path max-abs error <=
3e-2 times the tensor's largest oracle magnitude.
"""
import json
import os

import numpy as np

FP32_TOL = 1e-4
BF16_REL = 3e-2
INT_KEYS = ("p_traj", "src", "p_final")
FLOAT_KEYS = ("y", "h_stack", "c_stack", "dx", "dh0", "dc0", "dW", "dbias")


def tol_for(dtype, ref):
    if dtype == "fp32":
        return FP32_TOL
    return BF16_REL * max(float(np.abs(ref).max()), 1e-30)


def compare(got, ref, dtype, keys=None, inst=None):
    """Assert parity; ``inst`` restricts per-instance tensors of ``got`` to those
    instances (the oracle ran on them only). Returns {key: (max abs err, tol)}."""
    report = {}
    ref = dict(ref)
    if "p_traj" in ref:
        ref["p_final"] = ref["p_traj"][-1]
    batch_axis = {"p_traj": 1, "src": 1, "p_final": 0, "y": 1, "h_stack": 1, "c_stack": 1, "dx": 1,
                  "dh0": 0, "dc0": 0}
    for k in keys or (INT_KEYS + FLOAT_KEYS):
        if k not in ref or k not in got:
            continue
        g = got[k]
        if inst is not None and k in batch_axis:
            g = np.take(g, inst, axis=batch_axis[k])
        if k in INT_KEYS:
            assert np.array_equal(g, ref[k]), "%s differs (%d entries)" % (k, int((g != ref[k]).sum()))
            report[k] = (0, 0)
        else:
            err = float(np.abs(g.astype(np.float64) - ref[k]).max()) if ref[k].size else 0.0
            tol = tol_for(dtype, ref[k])
            assert np.isfinite(err) and err <= tol, "%s: max abs err %.3g > tol %.3g" % (k, err, tol)
            report[k] = (err, tol)
    log = os.environ.get("PARITY_LOG")
    if log:
        import inspect
        who = os.environ.get("PYTEST_CURRENT_TEST", inspect.stack()[1].function).split(" ")[0]
        with open(log, "a") as f:
            f.write(json.dumps({"test": who, "dtype": dtype,
                                "max_abs_err": {k: v[0] for k, v in report.items() if k not in INT_KEYS},
                                "tol": {k: v[1] for k, v in report.items() if k not in INT_KEYS}}) + "\n")
    return report
