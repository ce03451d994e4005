"""GPU parity of the small-batch CUDA-core kernels (bf16_small.cu) against the fp64 oracle.

For batches up to 32 the forward and the backward can run as one thread-block cluster on
CUDA cores (FFMA contraction, weights resident in shared memory) instead of the
tensor-core cluster kernels; the planner picks them below a measured crossover batch
size. Both paths are run here at the same shapes (STACKLSTM_CUDA_CORE=1 forces the
CUDA-core kernels, =0 the tensor-core ones), into NaN-filled outputs, and compared with
the oracle element by element: every row-count tier of the kernels (1, 2, 4, 8, 16, 32
rows), ragged hidden widths (H not a multiple of the 16-unit slice), narrow and wide
inputs, dy seeds, push-only mode, and run-to-run bitwise reproducibility.
"""
import os

import numpy as np
import pytest

import oracle
from paper_1904_03409_gb300 import binding as bd
from paper_1904_03409_gb300 import runner, workloads as wl
from parity import compare

pytestmark = pytest.mark.gpu
NTHREADS = max(1, len(os.sched_getaffinity(0)))


def oracle_all(w, mode="homogenized"):
    return oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h, dy=w.dy, mode=mode,
                      nthreads=NTHREADS)


def case(T, B, I, H, seed, probs=(0.5, 0.3, 0.2), **kw):
    return wl.make_workload("case", T=T, B=B, I=I, H=H, dtype="bf16", seed=seed, ops_kind="random_walk",
                            probs=probs, **kw)


def run_with(w, value, mode=bd.SL_MODE_HOMOGENIZED):
    old = os.environ.get("STACKLSTM_CUDA_CORE")
    os.environ["STACKLSTM_CUDA_CORE"] = value
    try:
        hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16, 0)
        plan = bd.stacklstm_plan(hd)
        hd.destroy()
        return plan, runner.run(w, mode=mode)
    finally:
        if old is None:
            os.environ.pop("STACKLSTM_CUDA_CORE", None)
        else:
            os.environ["STACKLSTM_CUDA_CORE"] = old


@pytest.mark.parametrize("T,B,I,H,seed", [
    (15, 1, 200, 200, 51),   # one row, parser widths
    (12, 2, 24, 40, 52),     # ragged H (the last slice half empty), narrow x
    (20, 3, 8, 16, 53),      # smallest widths, one CTA
    (16, 8, 200, 200, 54),
    (10, 13, 136, 72, 55),   # 16-row tier with 3 rows idle
    (9, 32, 64, 256, 56),    # 32-row tier, the widest hidden layer (16 CTAs)
])
def test_cuda_core_path_matches_oracle(T, B, I, H, seed):
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    plan, got = run_with(w, "1")
    assert "forward cuda-core" in plan and "backward cuda-core" in plan, plan
    compare(got, oracle_all(w), "bf16")


@pytest.mark.parametrize("B", [1, 8, 32])
def test_both_paths_at_the_sweep_batch_sizes(B):
    """The sweep workload (arc-standard op streams, I = H = 200) on both paths."""
    w = wl.config_workload("sweep", B=B)
    ref = oracle_all(w)
    plan1, cc = run_with(w, "1")
    plan0, tc = run_with(w, "0")
    assert "forward cuda-core" in plan1, plan1
    assert "forward cluster" in plan0 and "cuda-core" not in plan0, plan0
    compare(cc, ref, "bf16")
    compare(tc, ref, "bf16")
    for k in ("p_traj", "src"):
        assert np.array_equal(cc[k], tc[k])


def test_push_only_on_the_cuda_core_path():
    w = case(24, 6, 40, 56, 57, bias_scale=0.3, h0_scale=0.5, dy_scale=0.5)
    _, got = run_with(w, "1", mode=bd.SL_MODE_PUSH_ONLY)
    compare(got, oracle_all(w, mode="definition"), "bf16")
    assert got["steps_run"] == max(1, int((w.ops == 1).sum(0).max()))


def test_cuda_core_backward_is_bitwise_reproducible():
    w = case(18, 5, 32, 48, 58, dy_scale=1.0)
    _, a = run_with(w, "1")
    _, b = run_with(w, "1")
    for k in ("y", "h_stack", "c_stack", "dx", "dW", "dbias", "dh0", "dc0"):
        assert np.array_equal(a[k], b[k]), k


def test_planner_default_by_batch_size():
    """Unforced, the planner gives one row up to the crossover to the CUDA-core kernels and
    a 64-row batch to the tensor-core cluster kernels."""
    for B, want in ((1, "forward cuda-core"), (64, "forward cluster")):
        hd = bd.stacklstm_create(40, B, 200, 200, bd.SL_BF16, 0)
        try:
            assert want in bd.stacklstm_plan(hd)
        finally:
            hd.destroy()
