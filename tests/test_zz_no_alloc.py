"""The allocation-free index prepass (stacklstm_pointers_noalloc).

Some callers of this library cannot allocate device memory at the moment they need the
pointer bookkeeping: services whose device memory is all reserved up front by a pooling
allocator, and callers that must not let a cudaMalloc or cudaFree synchronize the device
while other streams run. For them the prepass runs on a fixed scratch array built into
the library. These tests check, through the C ABI on cuda:0, that its pointer
trajectories and read provenance equal those of stacklstm_forward bit for bit on two
calls in a row (the second call runs on the scratch the first one left behind), that a
call changes neither torch's allocated memory nor the device's free memory, and that
sizes beyond its limit are refused. The file is named to be collected last.
"""
import gc

import numpy as np
import pytest
import torch

from paper_1904_03409_gb300 import binding as bd
from paper_1904_03409_gb300 import runner, workloads as wl

pytestmark = pytest.mark.gpu


def via_forward(w):
    got = runner.run(w)
    return got["p_traj"], got["src"]


def via_noalloc(w):
    dev = torch.device("cuda", 0)
    ops = torch.from_numpy(np.ascontiguousarray(w.ops, np.int8)).to(dev)
    p = torch.full((w.T + 1, w.B), -7, dtype=torch.int32, device=dev)
    s = torch.full((w.T + 1, w.B), -7, dtype=torch.int32, device=dev)
    bd.stacklstm_pointers_noalloc(ops, p, s)
    return p.cpu().numpy(), s.cpu().numpy()


def test_matches_forward_on_two_calls_in_a_row():
    bd.load()
    cases = [wl.config_workload("parser64"),
             wl.make_workload("case", T=40, B=300, I=8, H=16, dtype="bf16", seed=21, ops_kind="random_walk",
                              probs=(0.45, 0.35, 0.2))]
    for w in cases:
        ref_p, ref_s = via_forward(w)
        for _ in range(2):
            p, s = via_noalloc(w)
            assert np.array_equal(p, ref_p)
            assert np.array_equal(s, ref_s)


def test_a_call_allocates_no_device_memory():
    w = wl.config_workload("parser64")
    dev = torch.device("cuda", 0)
    ops = torch.from_numpy(np.ascontiguousarray(w.ops, np.int8)).to(dev)
    p = torch.empty(w.T + 1, w.B, dtype=torch.int32, device=dev)
    s = torch.empty(w.T + 1, w.B, dtype=torch.int32, device=dev)
    bd.stacklstm_pointers_noalloc(ops, p, s)  # the device's one-time set-up happens here
    torch.cuda.synchronize(dev)
    # tensors of earlier tests are collected first, and no collection runs during the
    # measurement, so the counts change only if the call itself allocated
    gc.collect()
    gc.disable()
    try:
        for _ in range(2):
            alloc0, free0 = torch.cuda.memory_allocated(dev), torch.cuda.mem_get_info(dev)[0]
            bd.stacklstm_pointers_noalloc(ops, p, s)
            torch.cuda.synchronize(dev)
            assert torch.cuda.memory_allocated(dev) == alloc0
            assert torch.cuda.mem_get_info(dev)[0] == free0
    finally:
        gc.enable()


def test_refuses_sizes_beyond_its_scratch():
    dev = torch.device("cuda", 0)
    T, B = 1023, 1024  # (T + 1) * B = 1,048,576 fits; one more step does not
    ops = torch.zeros(T + 1, B, dtype=torch.int8, device=dev)
    p = torch.empty(T + 2, B, dtype=torch.int32, device=dev)
    with pytest.raises(bd.StackLSTMError) as e:
        bd.stacklstm_pointers_noalloc(ops, p, p)
    assert e.value.status == 7
    ops = torch.ones(T, B, dtype=torch.int8, device=dev)
    p = torch.empty(T + 1, B, dtype=torch.int32, device=dev)
    s = torch.empty(T + 1, B, dtype=torch.int32, device=dev)
    bd.stacklstm_pointers_noalloc(ops, p, s)
    assert p[-1].eq(T).all().item() and s[-1].eq(T).all().item()
