"""GPU parity of the fp32 CUDA-core path against the fp64 oracle, and the device-side
error statuses. Runs through the C ABI on cuda:0."""
import numpy as np
import pytest
import torch

import oracle
from paper_1904_03409_gb300 import binding as bd
from paper_1904_03409_gb300 import runner, workloads as wl
from parity import compare

pytestmark = pytest.mark.gpu


def oracle_of(w, d_top_h=None):
    return oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h if d_top_h is None else d_top_h,
                      dy=w.dy)


def test_tiny_config():
    w = wl.config_workload("tiny")
    got = runner.run(w)
    compare(got, oracle_of(w), "fp32")


@pytest.mark.parametrize("T,B,I,H,seed,probs", [
    (33, 37, 24, 40, 1, (0.5, 0.3, 0.2)),    # ragged B, H not a multiple of 32
    (50, 5, 7, 33, 2, (0.4, 0.4, 0.2)),      # odd sizes
    (20, 130, 16, 160, 3, (0.6, 0.3, 0.1)),  # several thread blocks per instance
    (1, 3, 4, 5, 4, (1.0, 0.0, 0.0)),        # a single step
])
def test_random_cases(T, B, I, H, seed, probs):
    w = wl.make_workload("case", T=T, B=B, I=I, H=H, dtype="fp32", seed=seed, ops_kind="random_walk",
                         probs=probs, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    got = runner.run(w)
    compare(got, oracle_of(w), "fp32")


@pytest.mark.parametrize("T,B,I,H,seed", [(12, 4, 16, 16, 10), (20, 16, 16, 32, 11), (9, 20, 8, 48, 12)])
def test_one_cta_and_per_step_kernels_agree_bit_for_bit(T, B, I, H, seed):
    """Small problems run each direction's steps in one CTA; the per-step kernels
    (STACKLSTM_STEP_KERNELS=1) do the same arithmetic per element, so every output is
    bit-identical, and both match the oracle."""
    import os
    w = wl.make_workload("case", T=T, B=B, I=I, H=H, dtype="fp32", seed=seed, ops_kind="random_walk",
                         probs=(0.5, 0.3, 0.2), bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    hd = bd.stacklstm_create(T, B, I, H, bd.SL_FP32, 0)
    try:
        assert "one CTA" in bd.stacklstm_plan(hd)
    finally:
        hd.destroy()
    one = runner.run(w)
    os.environ["STACKLSTM_STEP_KERNELS"] = "1"
    try:
        hd = bd.stacklstm_create(T, B, I, H, bd.SL_FP32, 0)
        try:
            assert "one launch per step" in bd.stacklstm_plan(hd)
        finally:
            hd.destroy()
        per = runner.run(w)
    finally:
        os.environ.pop("STACKLSTM_STEP_KERNELS", None)
    for k in ("y", "h_stack", "c_stack", "dx", "dW", "dbias", "dh0", "dc0"):
        assert np.array_equal(one[k], per[k], equal_nan=False), k
    compare(one, oracle_of(w), "fp32")


def test_holds_only_and_all_push():
    for probs in ((0.0, 0.0, 1.0), (1.0, 0.0, 0.0)):
        w = wl.make_workload("case", T=16, B=9, I=8, H=12, dtype="fp32", seed=7, ops_kind="random_walk",
                             probs=probs, h0_scale=0.5)
        got = runner.run(w)
        compare(got, oracle_of(w), "fp32")
        if probs[2] == 1.0:
            assert np.all(got["dx"] == 0.0) and np.all(got["dW"] == 0.0)


def test_dead_writes_have_exactly_zero_input_gradient():
    w = wl.make_workload("case", T=40, B=16, I=8, H=12, dtype="fp32", seed=8, ops_kind="random_walk",
                         probs=(0.4, 0.4, 0.2))
    got = runner.run(w)
    assert np.all(got["dx"][w.ops != 1] == 0.0)


def test_backward_is_bitwise_reproducible():
    w = wl.make_workload("case", T=25, B=20, I=8, H=16, dtype="fp32", seed=9, ops_kind="random_walk",
                         probs=(0.5, 0.3, 0.2), dy_scale=1.0)
    a, b = runner.run(w), runner.run(w)
    for k in ("dx", "dW", "dbias", "dh0", "dc0"):
        assert np.array_equal(a[k], b[k]), k


def _statuses(ops_np):
    T, B = ops_np.shape
    hd = bd.stacklstm_create(T, B, 4, 4, bd.SL_FP32, 0)
    dev = torch.device("cuda", 0)
    z = lambda *s: torch.zeros(*s, device=dev)
    ops = torch.from_numpy(ops_np.astype(np.int8)).to(dev)
    pf = torch.zeros(B, dtype=torch.int32, device=dev)
    try:
        with pytest.raises(bd.StackLSTMError) as e:
            bd.stacklstm_forward(hd, z(T, B, 4), ops, z(B, 4), z(B, 4), z(8, 16), z(16), p_final=pf)
        return e.value.status, hd
    except BaseException:
        hd.destroy()
        raise


def test_bad_op_and_underflow_statuses():
    st, hd = _statuses(np.array([[1, 2], [0, 0]]))
    hd.destroy()
    assert st == 2
    st, hd = _statuses(np.array([[1, 0], [-1, -1]]))
    assert st == 3
    # the handle stays usable: a valid stream now succeeds
    dev = torch.device("cuda", 0)
    z = lambda *s: torch.zeros(*s, device=dev)
    pf = torch.zeros(2, dtype=torch.int32, device=dev)
    bd.stacklstm_forward(hd, z(2, 2, 4), torch.ones(2, 2, dtype=torch.int8, device=dev), z(2, 4), z(2, 4),
                         z(8, 16), z(16), p_final=pf)
    assert pf.tolist() == [2, 2]
    hd.destroy()


def test_backward_before_forward():
    hd = bd.stacklstm_create(3, 2, 4, 4, bd.SL_FP32, 0)
    try:
        with pytest.raises(bd.StackLSTMError) as e:
            bd.stacklstm_backward(hd)
        assert e.value.status == 4
    finally:
        hd.destroy()
