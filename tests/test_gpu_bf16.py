"""GPU parity of the bf16 tensor-core path against the fp64 oracle, through the C ABI.

Small shapes compare every output element (they span several tiles with ragged tails:
B not a multiple of the 128-row tile, H not a multiple of the unit tile, I + H and 4H
not multiples of the 64-wide contraction chunk). The five named workloads run at their
full sizes in the launch configuration the benchmark times; where the oracle cannot
finish every instance in seconds, it runs a sample of instances and the loss seed is
restricted to them, so dW and dbias are the sums over exactly those instances.
Pointer trajectories and read provenance are compared bit for bit for all instances.
"""
import os
import re

import numpy as np
import pytest
import torch

import oracle
from paper_1904_03409_gb300 import binding as bd
from paper_1904_03409_gb300 import runner, workloads as wl
from parity import compare

pytestmark = pytest.mark.gpu
NTHREADS = max(1, len(os.sched_getaffinity(0)))


def oracle_all(w, d_top_h=None):
    return oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h if d_top_h is None else d_top_h,
                      dy=w.dy, nthreads=NTHREADS)


def case(T, B, I, H, seed, probs=(0.5, 0.3, 0.2), **kw):
    return wl.make_workload("case", T=T, B=B, I=I, H=H, dtype="bf16", seed=seed, ops_kind="random_walk",
                            probs=probs, **kw)


def test_single_step_all_push():
    w = case(1, 130, 64, 64, 11, probs=(1.0, 0.0, 0.0), bias_scale=0.5, h0_scale=0.8, c0_scale=0.8)
    compare(runner.run(w), oracle_all(w), "bf16")


@pytest.mark.parametrize("T,B,I,H,seed", [
    (12, 128, 64, 64, 1),     # exact tiles
    (20, 200, 24, 40, 2),     # ragged rows, I + H not a multiple of 64, partial unit tile
    (17, 37, 8, 16, 3),       # smallest widths
    (30, 300, 136, 72, 4),    # three row tiles, mixed x / h contraction chunk
    (9, 129, 256, 256, 5),    # one extra row past a tile
])
def test_small_shapes(T, B, I, H, seed):
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    compare(runner.run(w), oracle_all(w), "bf16")


def test_holds_only_and_dead_writes():
    w = case(16, 40, 16, 24, 6, probs=(0.0, 0.0, 1.0), h0_scale=0.5)
    got = runner.run(w)
    compare(got, oracle_all(w), "bf16")
    assert np.all(got["dx"] == 0.0) and np.all(got["dW"] == 0.0)
    w = case(40, 50, 16, 24, 7, probs=(0.4, 0.4, 0.2))
    got = runner.run(w)
    compare(got, oracle_all(w), "bf16")
    assert np.all(got["dx"][w.ops != 1] == 0.0)


def test_backward_is_bitwise_reproducible():
    w = case(25, 150, 32, 48, 8, dy_scale=1.0)
    a, b = runner.run(w), runner.run(w)
    for k in ("dx", "dW", "dbias", "dh0", "dc0", "y", "h_stack"):
        assert np.array_equal(a[k], b[k]), k


def test_parser64_config():
    w = wl.config_workload("parser64")
    compare(runner.run(w), oracle_all(w), "bf16")


@pytest.mark.parametrize("B", [1, 8, 32, 128])
def test_sweep_config_small_batches(B):
    w = wl.config_workload("sweep", B=B)
    compare(runner.run(w), oracle_all(w), "bf16")


def sampled_check(w, inst):
    """Full-size GPU run; oracle on the sampled instances (loss seed restricted to them)."""
    seed = np.zeros_like(w.d_top_h)
    seed[inst] = w.d_top_h[inst]
    got = runner.run(w, d_top_h=seed)
    ptr = oracle.pointers(w.ops)
    assert np.array_equal(got["p_traj"], ptr["p_traj"])
    assert np.array_equal(got["src"], ptr["src"])
    ref = oracle.run_instances(inst, w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h, dy=w.dy,
                               nthreads=NTHREADS)
    rep = compare(got, ref, "bf16", inst=np.asarray(inst))
    # instances outside the sample had a zero loss seed: exactly zero input gradient
    rest = np.setdiff1d(np.arange(w.B), inst)
    assert np.all(got["dx"][:, rest] == 0.0) and np.all(got["dh0"][rest] == 0.0)
    torch.cuda.empty_cache()
    return rep


@pytest.mark.parametrize("B", [512, 1024])
def test_sweep_config_large_batches_sampled(B):
    w = wl.config_workload("sweep", B=B)
    sampled_check(w, [0, 1, 127, 128, B // 2 + 3, B - 1])


def test_large_config_sampled():
    w = wl.config_workload("large")
    sampled_check(w, [0, 77, 128, 200, 254, 255])


def test_stress_config_sampled():
    w = wl.config_workload("stress")
    sampled_check(w, [0, 1, 127, 128, 2047, 3000, 4094, 4095])


@pytest.mark.parametrize("T,B,I,H,seed", [(16, 4096, 256, 256, 26), (16, 4000, 256, 248, 27)])
def test_four_lanes_per_row_backward_epilogue(T, B, I, H, seed):
    """The persistent backward with 32-unit column tiles and one epilogue warp group takes
    each row's units four lanes at a time, after a shared-memory transpose of the
    accumulator rows. The stress shape, and a ragged one (B = 4000: the last row tile a
    quarter full; H = 248: the last column tile 24 units); the oracle on instances at
    every warp, round and lane position of a row tile, in three row tiles."""
    w = case(T, B, I, H, seed, probs=(0.6, 0.3, 0.1), bias_scale=0.3, h0_scale=0.5, c0_scale=0.5)
    hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16, 0)
    try:
        plan = bd.stacklstm_plan(hd)
    finally:
        hd.destroy()
    assert "backward persistent U=32 [EP 1" in plan and "contraction parts 1" in plan, plan
    last = (B - 1) // 128 * 128
    inst = sorted({base + r for base in (0, 17 * 128, last) for r in range(0, 128, 9) if base + r < B} | {B - 1})
    sampled_check(w, inst)


PERSISTENT = {"STACKLSTM_FWD_CLUSTER": "0", "STACKLSTM_BWD_CLUSTER": "0"}


@pytest.mark.parametrize("B,env", [(130, PERSISTENT), (40, {}), (130, {})])
def test_wait_timeout_is_reported_and_context_survives(B, env):
    """With a zero wait budget the bounded device-side waits run out: forward (persistent
    kernel at B = 130, thread-block clusters at B = 40 and at B = 130, three row tiles)
    reports SL_ERR_TIMEOUT instead of hanging, and the device stays usable."""
    w = case(4, B, 16, 32, 9)
    old = {k: os.environ.get(k) for k in env}
    os.environ.update(env)
    os.environ["STACKLSTM_WAIT_LIMIT_CYCLES"] = "0"
    try:
        hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16, 0)
    finally:
        del os.environ["STACKLSTM_WAIT_LIMIT_CYCLES"]
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    try:
        ins = runner.upload(w)
        out = runner.alloc_outputs(w)
        with pytest.raises(bd.StackLSTMError) as e:
            bd.stacklstm_forward(hd, ins["x"], ins["ops"], ins["h0"], ins["c0"], ins["W"], ins["bias"],
                                 p_final=out["p_final"])
        assert e.value.status == 6
    finally:
        hd.destroy()
    compare(runner.run(w), oracle_all(w), "bf16")


@pytest.mark.parametrize("T,B,I,H,env,want", [
    (6, 200, 64, 256, dict(PERSISTENT, STACKLSTM_BWD_SPLIT="4"), "cluster 4 "),  # split contraction, clusters
    (4, 4096, 256, 256, {}, "U=32 [EP 1"),                                      # the release warp's plan
    (6, 200, 64, 256, dict(PERSISTENT, STACKLSTM_BWD_SPLIT="4", STACKLSTM_SPLIT_CLUSTER="0"), "cluster 1 "),
    (6, 40, 64, 64, {}, "cluster U=16 ["),                                       # one-row-tile cluster
])
def test_backward_wait_timeout_is_reported_and_context_survives(T, B, I, H, env, want):
    """With a zero wait budget for the backward's kernels only, the forward completes and the
    backward reports SL_ERR_TIMEOUT instead of hanging: the persistent backward with its
    contraction split in thread-block clusters (partials in flight between the parts) or
    through L2, the one whose release warp waits at a barrier with the epilogue, and the
    cluster backward. The device stays usable: a new handle then reproduces a normal run
    bit for bit."""
    w = case(T, B, I, H, 10, bias_scale=0.3, h0_scale=0.5)

    def with_env(extra, fn):
        keys = dict(env, **extra)
        old = {k: os.environ.get(k) for k in keys}
        os.environ.update(keys)
        try:
            return fn()
        finally:
            for k, v in old.items():
                if v is None:
                    os.environ.pop(k, None)
                else:
                    os.environ[k] = v

    ref = with_env({}, lambda: runner.run(w))
    hd = with_env({"STACKLSTM_WAIT_LIMIT_BWD_CYCLES": "0"},
                  lambda: bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16, 0))
    try:
        assert want in bd.stacklstm_plan(hd).split("; backward ")[1], bd.stacklstm_plan(hd)
        ins, out = runner.upload(w), runner.alloc_outputs(w)
        bd.stacklstm_forward(hd, ins["x"], ins["ops"], ins["h0"], ins["c0"], ins["W"], ins["bias"],
                             p_final=out["p_final"])
        bd.stacklstm_status(hd)
        with pytest.raises(bd.StackLSTMError) as e:
            bd.stacklstm_backward(hd, ins["d_top_h"], None, out["dx"], out["dh0"], out["dc0"], out["dW"],
                                  out["dbias"])
            bd.stacklstm_status(hd)
        assert e.value.status == 6
    finally:
        hd.destroy()
    again = with_env({}, lambda: runner.run(w))
    for k in ("y", "h_stack", "c_stack", "dx", "dW", "dbias", "dh0", "dc0"):
        assert np.array_equal(again[k], ref[k]), k


@pytest.mark.parametrize("T,B,I,H,seed", [(20, 200, 24, 40, 12), (9, 300, 136, 72, 13)])
def test_per_step_kernels_match_oracle(T, B, I, H, seed):
    """The one-launch-per-step kernels (used when a persistent grid cannot be
    co-resident) stay parity-green too."""
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    os.environ["STACKLSTM_STEP_KERNELS"] = "1"
    try:
        got = runner.run(w)
    finally:
        del os.environ["STACKLSTM_STEP_KERNELS"]
    compare(got, oracle_all(w), "bf16")


@pytest.mark.parametrize("T,B,I,H,seed,cl", [(12, 200, 64, 256, 14, 4), (10, 130, 40, 200, 15, 4),
                                            (6, 1300, 16, 256, 26, 1)])
def test_split_contraction_backward_matches_oracle(T, B, I, H, seed, cl):
    """The backward with its 4H contraction split over four CTAs per column tile stays
    parity-green, including parts of unequal length (H = 200: 13 chunks over 4 parts), into
    NaN-filled outputs. Where each CTA keeps one row tile the four parts run as one
    thread-block cluster and trade their partial sums in shared memory; with several row
    tiles a CTA (B = 1300: 11 row tiles) they go through an L2 scratch. Both sum the parts in
    part order, so the two exchanges agree bit for bit, and a rerun repeats them."""
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    env = dict(PERSISTENT, STACKLSTM_BWD_SPLIT="4")
    plan, got = run_nan_filled(w, env)
    plan0, l2 = run_nan_filled(w, dict(env, STACKLSTM_SPLIT_CLUSTER="0"))
    _, again = run_nan_filled(w, env)
    bwd, bwd0 = plan.split("; backward ")[1], plan0.split("; backward ")[1]
    assert "persistent U=64" in bwd and "contraction parts 4" in bwd and "cluster %d " % cl in bwd, plan
    assert "contraction parts 4" in bwd0 and "cluster 1 " in bwd0, plan0
    compare(got, oracle_all(w), "bf16")
    for k in ("dx", "dW", "dbias", "dh0", "dc0"):
        assert np.array_equal(got[k], l2[k]), k
        assert np.array_equal(got[k], again[k]), k


@pytest.mark.parametrize("T,B,I,H,seed", [(20, 200, 24, 40, 27), (9, 300, 136, 72, 28), (12, 130, 264, 64, 29)])
def test_weight_gradient_tile_shapes_match_oracle(T, B, I, H, seed):
    """The weight gradient with 128 x 256 tiles (two CTAs an SM) and with 256 x 256 tiles
    (two accumulators over one dG operand, one CTA an SM), into NaN-filled outputs: x and h
    blocks of W in one tile, constant zero blocks past I + H (I = 264: five x blocks and one
    h block), ragged gate columns (4H = 160, 288)."""
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    ref = oracle_all(w)
    for m in ("128", "256"):
        plan, got = run_nan_filled(w, {"STACKLSTM_DW_M": m})
        assert "tiles of %sx256" % m in plan, plan
        compare(got, ref, "bf16")


def run_nan_filled(w, env):
    """Forward + backward with every output buffer filled with NaN first (an element the
    path fails to write cannot pass), under extra environment settings; (plan, dx)."""
    old = {k: os.environ.get(k) for k in env}
    os.environ.update(env)
    try:
        hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16, 0)
    finally:
        for k, v in old.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    try:
        plan = bd.stacklstm_plan(hd)
        ins = runner.upload(w)
        out = runner.alloc_outputs(w)
        for v in out.values():
            if v.is_floating_point():
                v.fill_(float("nan"))
        runner.forward_backward(hd, ins, out)
        torch.cuda.synchronize()
        bd.stacklstm_status(hd)
        return plan, runner.to_numpy(out)
    finally:
        hd.destroy()


@pytest.mark.parametrize("T,B,I,H,seed", [(11, 200, 264, 64, 16), (9, 129, 256, 256, 17), (40, 512, 256, 256, 18)])
def test_input_gradient_on_spare_sms_matches_oracle(T, B, I, H, seed):
    """dx computed by the extra CTAs of the backward launch, on the SMs the step chain
    leaves idle (128-row tiles that straddle two steps; I = 264: a second, partial
    256-column tile; B = 512: several tiles per extra CTA), into NaN-filled outputs,
    matches the oracle and equals bit for bit the separate dx launch (same contraction
    chunk order). A single extra CTA, trailing the whole chain, too."""
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    plan, got = run_nan_filled(w, dict(PERSISTENT))
    m = re.search(r"dx CTAs (\d+)", plan)
    assert m and int(m.group(1)) >= 4, plan
    compare(got, oracle_all(w), "bf16")
    plan0, sep = run_nan_filled(w, dict(PERSISTENT, STACKLSTM_DX_SPARE="0"))
    assert "dx CTAs 0" in plan0, plan0
    assert np.array_equal(got["dx"], sep["dx"])
    # one extra CTA is no whole cluster: a split contraction's parts then trade through L2
    # (which may change the plan, so its own separate-launch dx is the reference)
    l2 = dict(PERSISTENT, STACKLSTM_SPLIT_CLUSTER="0")
    _, sep1 = run_nan_filled(w, dict(l2, STACKLSTM_DX_SPARE="0"))
    plan1, one = run_nan_filled(w, dict(l2, STACKLSTM_DX_SPARE="1"))
    assert "dx CTAs 1" in plan1, plan1
    assert np.array_equal(one["dx"], sep1["dx"])


@pytest.mark.parametrize("T,B,I,H,seed", [(17, 40, 8, 16, 19), (24, 64, 200, 200, 20), (9, 8, 64, 136, 21),
                                         (12, 37, 24, 40, 22), (14, 100, 24, 40, 23), (10, 200, 64, 136, 24),
                                         (8, 450, 16, 32, 25)])
def test_cluster_kernels_match_oracle(T, B, I, H, seed):
    """Up to 8 row tiles of 64 instances: the forward and the backward as one thread-block
    cluster per row tile, their defaults (a ragged last tile: B = 100, 200, 450), into
    NaN-filled outputs, match the oracle, as do the persistent kernels they replace."""
    w = case(T, B, I, H, seed, bias_scale=0.3, h0_scale=0.5, c0_scale=0.5, dy_scale=0.5)
    plan, got = run_nan_filled(w, {})
    assert "forward cluster U=16" in plan and "backward cluster U=16" in plan, plan
    assert "slots %d" % ((B + 63) // 64) in plan, plan
    ref = oracle_all(w)
    compare(got, ref, "bf16")
    plan_p, per = run_nan_filled(w, {"STACKLSTM_BWD_CLUSTER": "0", "STACKLSTM_FWD_CLUSTER": "0"})
    assert "forward persistent" in plan_p and "backward persistent" in plan_p, plan_p
    compare(per, ref, "bf16")
    # one cluster kernel beside a persistent one: the saved gates keep the row-major layout
    for env, want in (({"STACKLSTM_BWD_CLUSTER": "0"}, ("forward cluster", "backward persistent")),
                      ({"STACKLSTM_FWD_CLUSTER": "0"}, ("forward persistent", "backward cluster"))):
        plan_m, mixed = run_nan_filled(w, env)
        assert all(x in plan_m for x in want), plan_m
        compare(mixed, ref, "bf16")
