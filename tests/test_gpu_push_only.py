"""GPU parity of the push-only mode (dead writes skipped) against the fp64 oracle.

Observation 2 of Sec. 3: a pop or hold step writes slot p + 1 above the new top, and the
next push overwrites that slot before the pointer reaches it, so only push steps' writes
are ever read. In SL_MODE_PUSH_ONLY the library runs the cell for push steps only, each
instance's pushes forming a virtual timeline. Its results are checked against the
oracle's definition mode (the push/pop semantics of Sec. 2: push runs the cell on the top
and writes above it, pop and hold only move the pointer), whose slot-indexed stack holds
each slot's last pushed state, and against the homogenized mode on the GPU: y and dx bit
for bit (the same per-row arithmetic), the live part of the stack, and the number of
steps the kernels ran (the most pushes of any instance). Outputs are NaN-filled first.
"""
import os

import numpy as np
import pytest
import torch

import oracle
from paper_1904_03409_gb300 import binding as bd
from paper_1904_03409_gb300 import runner, workloads as wl
from parity import compare

pytestmark = pytest.mark.gpu
NTHREADS = max(1, len(os.sched_getaffinity(0)))
PUSH = bd.SL_MODE_PUSH_ONLY
PERSISTENT = {"STACKLSTM_FWD_CLUSTER": "0", "STACKLSTM_BWD_CLUSTER": "0"}


def definition(w, d_top_h=None, inst=None):
    seed = w.d_top_h if d_top_h is None else d_top_h
    if inst is None:
        return oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=seed, dy=w.dy, mode="definition",
                          nthreads=NTHREADS)
    return oracle.run_instances(inst, w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=seed, dy=w.dy,
                                mode="definition", nthreads=NTHREADS)


def case(T, B, I, H, seed, probs=(0.5, 0.3, 0.2), **kw):
    return wl.make_workload("case", T=T, B=B, I=I, H=H, dtype="bf16", seed=seed, ops_kind="random_walk",
                            probs=probs, **kw)


def with_env(env, fn):
    old = {k: os.environ.get(k) for k in env}
    os.environ.update(env)
    try:
        return fn()
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v


def check_against_homogenized(w, got, env=None):
    """y and dx bit for bit, the live stack, and the virtual step count."""
    hom = with_env(env or {}, lambda: runner.run(w))
    assert np.array_equal(got["y"], hom["y"])
    assert np.array_equal(got["dx"], hom["dx"])
    for k in ("p_traj", "src", "p_final"):
        assert np.array_equal(got[k], hom[k]), k
    live = np.arange(w.T + 1)[:, None] <= got["p_final"][None, :]
    for k in ("h_stack", "c_stack"):
        assert np.array_equal(got[k][live], hom[k][live]), k
    assert got["steps_run"] == max(1, int((w.ops == 1).sum(0).max()))
    assert hom["steps_run"] == w.T


@pytest.mark.parametrize("T,B,I,H,seed,env", [
    (17, 40, 8, 16, 31, {}),                                  # one row tile: thread-block cluster kernels
    (24, 64, 200, 200, 32, {}),                               # parser widths, cluster kernels
    (20, 200, 24, 40, 33, {}),                                # clusters, four row tiles
    (20, 200, 24, 40, 33, dict(PERSISTENT)),                  # persistent kernels, ragged tiles
    (30, 300, 136, 72, 34, dict(PERSISTENT)),                 # three row tiles
    (11, 200, 264, 64, 35, dict(PERSISTENT)),                 # dx on the spare SMs of the backward launch
    (12, 200, 64, 256, 36, dict(PERSISTENT, STACKLSTM_BWD_SPLIT="4")),  # split-contraction backward
    (20, 200, 24, 40, 37, {"STACKLSTM_STEP_KERNELS": "1"}),   # one launch per step
    (11, 200, 264, 64, 38, dict(PERSISTENT, STACKLSTM_DX_SPARE="0")),   # dx in its own launch
])
def test_push_only_matches_definition_mode(T, B, I, H, seed, env):
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    got = with_env(env, lambda: runner.run(w, mode=PUSH))
    compare(got, definition(w), "bf16")
    check_against_homogenized(w, got, env)


@pytest.mark.parametrize("T,B", [(900, 40), (900, 64), (2000, 64)])
def test_long_sequences_take_every_index_prepass(T, B):
    """The index prepass has three forms by sequence length: up to several hundred steps one
    kernel walks the ops with its slot tags (and, push-only mode, the real-to-virtual index
    map) on chip; at T = 900 the push-only map no longer fits beside the tags and the
    compaction runs as a kernel of its own; at T = 2000 the slot tags live in a global
    scratch. Each with a ragged 32-instance block (B = 40) or whole ones (B = 64), both modes."""
    w = case(T, B, 8, 16, 42 + T + B, probs=(0.45, 0.35, 0.2), bias_scale=0.3, h0_scale=0.5)
    ptr = oracle.pointers(w.ops)
    hom = runner.run(w)
    assert np.array_equal(hom["p_traj"], ptr["p_traj"]) and np.array_equal(hom["src"], ptr["src"])
    got = runner.run(w, mode=PUSH)
    compare(got, definition(w), "bf16")
    check_against_homogenized(w, got)


def test_no_push_at_all_runs_one_unread_step():
    w = case(16, 40, 16, 24, 39, probs=(0.0, 0.0, 1.0), h0_scale=0.5)
    got = runner.run(w, mode=PUSH)
    compare(got, definition(w), "bf16")
    assert got["steps_run"] == 1
    assert np.all(got["dx"] == 0.0) and np.all(got["dW"] == 0.0)


def test_all_push_is_the_homogenized_run():
    w = case(14, 150, 32, 48, 40, probs=(1.0, 0.0, 0.0), bias_scale=0.3, h0_scale=0.5)
    got = runner.run(w, mode=PUSH)
    compare(got, definition(w), "bf16")
    hom = runner.run(w)
    assert got["steps_run"] == w.T
    for k in ("y", "h_stack", "c_stack", "dx", "dh0", "dc0", "dW", "dbias"):
        assert np.array_equal(got[k], hom[k]), k


@pytest.mark.parametrize("name", ["parser64", "sweep:1", "sweep:128"])
def test_parser_workloads(name):
    w = wl.config_workload("sweep", B=int(name.split(":")[1])) if ":" in name else wl.config_workload(name)
    got = runner.run(w, mode=PUSH)
    compare(got, definition(w), "bf16")
    check_against_homogenized(w, got)


@pytest.mark.parametrize("name,inst", [("large", [0, 77, 128, 255]), ("stress", [0, 1, 2047, 4095])])
def test_full_size_workloads_sampled(name, inst):
    w = wl.config_workload(name)
    seed = np.zeros_like(w.d_top_h)
    seed[inst] = w.d_top_h[inst]
    got = runner.run(w, d_top_h=seed, mode=PUSH)
    ptr = oracle.pointers(w.ops)
    assert np.array_equal(got["p_traj"], ptr["p_traj"]) and np.array_equal(got["src"], ptr["src"])
    compare(got, definition(w, inst=inst), "bf16", inst=np.asarray(inst))
    rest = np.setdiff1d(np.arange(w.B), inst)
    assert np.all(got["dx"][:, rest] == 0.0) and np.all(got["dh0"][rest] == 0.0)
    assert got["steps_run"] == int((w.ops == 1).sum(0).max())
    torch.cuda.empty_cache()


def test_mode_switch_needs_a_new_forward_and_fp32_is_refused():
    w = case(6, 20, 8, 16, 41)
    hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16, 0)
    try:
        ins, out = runner.upload(w), runner.alloc_outputs(w)
        runner.forward_backward(hd, ins, out)
        bd.stacklstm_set_mode(hd, PUSH)
        with pytest.raises(bd.StackLSTMError) as e:
            bd.stacklstm_backward(hd, ins["d_top_h"], None, out["dx"])
        assert e.value.status == 4
        runner.forward_backward(hd, ins, out)
        assert bd.stacklstm_steps_run(hd) == max(1, int((w.ops == 1).sum(0).max()))
        bd.stacklstm_set_mode(hd, bd.SL_MODE_HOMOGENIZED)
        assert "push-only" not in bd.stacklstm_plan(hd)
    finally:
        hd.destroy()
    hf = bd.stacklstm_create(4, 4, 16, 16, bd.SL_FP32, 0)
    try:
        with pytest.raises(bd.StackLSTMError) as e:
            bd.stacklstm_set_mode(hf, PUSH)
        assert e.value.status == 7
    finally:
        hf.destroy()
