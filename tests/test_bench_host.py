"""Host logic of bench.py, on CPU: the one-GPU rule, the reference arm under torchrun,
and the roofline arithmetic of its JSON line.

The library runs on one GPU, so bench.py refuses --gpus N > 1 and a torchrun world larger
than one before it builds or calls the library. The reference arm (the fp64 oracle on the
host cores) runs on rank 0 alone when launched under torchrun.
"""
import json
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("argv,env", [(["--gpus", "2"], {}), (["--gpus", "1"], {"WORLD_SIZE": "2", "RANK": "1"})])
def test_more_than_one_gpu_is_refused_before_any_library_call(argv, env):
    e = dict(os.environ, **env)
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *argv, "--steps", "1", "--warmup", "3"],
                       cwd=ROOT, capture_output=True, text=True, timeout=120, env=e)
    assert r.returncode == 2, (r.returncode, r.stderr[-2000:])
    assert "one GPU" in r.stderr
    assert not [l for l in r.stdout.splitlines() if l.startswith("{")]


def test_reference_arm_under_torchrun_prints_once():
    """Two ranks launched as the driver does: rank 0 times the oracle and prints one JSON
    line; rank 1 exits 0 without work."""
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(free_port()), os.path.join(ROOT, "bench.py"),
           "--impl", "reference", "--gpus", "2", "--workload", "tiny", "--steps", "2", "--warmup", "3",
           "--ref-step-seconds", "0.05"]
    r = subprocess.run(cmd, cwd=ROOT, capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [l for l in r.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["n_gpus"] == 2 and d["value"] > 0
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["cpu_baseline"]["kind"] == "oracle"


def test_work_per_instance_step_sums_its_phases():
    """Whole-step flops and bytes are the sum of the forward, backward, dx and dW terms
    minus the dW bias column (the step counts the contraction only)."""
    for I, H in ((200, 200), (512, 1024), (16, 16)):
        for dt in ("bf16", "fp32"):
            w = bench.work_per_inst_step(I, H, dt)
            assert w["step"]["flops"] == 24 * H * (I + H)
            parts = sum(w[p]["flops"] for p in ("forward", "backward", "dx", "dw"))
            assert parts - 8 * H == w["step"]["flops"]
        assert bench.work_per_inst_step(I, H)["step"]["bytes"] == 8 * I + 46 * H
        assert bench.work_per_inst_step(I, H, "fp32")["step"]["bytes"] == 12 * I + 52 * H


def test_roofline_picks_the_tighter_bound():
    peaks = {"hbm_gbs": 1000.0, "bf16_tflops": 100.0, "bf16_tflops_sustained": 90.0, "sm_max_mhz": 2000.0}
    # 1e12 flops (10 ms at peak) against 1e9 bytes (1 ms at peak): tensor-bound
    r = bench.roofline_of(1e12, 1e9, 0.02, peaks, "measured")
    assert r["bound"] == "tensor" and abs(r["frac"] - 0.5) < 1e-12 and r["peak"] == 100.0
    r = bench.roofline_of(1e9, 1e10, 0.02, peaks, "measured")
    assert r["bound"] == "hbm" and abs(r["frac"] - 0.5) < 1e-12
    # fp32 path: CUDA-core FFMA peak from the SM count and the clock
    r = bench.roofline_of(1e12, 1e9, 1.0, peaks, "measured", dtype="fp32", sms=100)
    assert r["bound"] == "alu" and abs(r["peak"] - 100 * 128 * 2 * 2000e6 / 1e12) < 1e-9
