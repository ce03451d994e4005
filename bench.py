#!/usr/bin/env python
"""Forward + backward throughput of the homogenized StackLSTM step on GB300.

One "step" is one pass of the whole hot path over one batch: forward over all T time
steps (Algorithm 1) and the reverse-time backward with dx, dW and dbias. The metric is
instance-steps per second, B * T per step (hold padding included: the homogenized
method computes padded steps too).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Prints ONE JSON line (rank 0). Under torchrun each rank runs its own replica of the
workload on its own GPU (instances are independent; no collective on the data path);
the job value is all ranks' instance-steps over the slowest rank's time.
--impl reference times the fp64 CPU oracle on the host cores on the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import re
import math
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "fwd+bwd StackLSTM instance-steps/s"
UNIT = "instance-steps/s"
L2_FLUSH_BYTES = 256 << 20  # > the 129 MB L2
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}


# ----------------------------------------------------------------------------- setup
def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def get_workload(name, T=None):
    from paper_1904_03409_gb300 import workloads as wl
    if name.startswith("sweep:"):
        return wl.config_workload("sweep", B=int(name.split(":")[1]))
    return wl.config_workload(name, T=T)


def describe(w):
    ops = {"tiny": "uniform valid push/pop/hold", "parser64": "random valid arc-standard sequences flattened to "
           "push/pop (n~U[10,60]), hold-padded", "large": "push/pop/hold .5/.3/.2, ragged lengths U[64,256], "
           "hold-padded", "stress": "push/pop/hold .6/.3/.1, all real steps", "sweep": "as parser64"}
    return ("%s: B=%d T=%d I=%d H=%d, %s, seed %d" % (w.name, w.B, w.T, w.I, w.H, ops.get(w.name, ""), w.seed))


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {k: float(d[k]) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ---------------------------------------------------------------- algorithmic work
def work_per_inst_step(I, H):
    """Flops and bytes per instance-step, per kernel phase and for the whole step (bf16
    path). Whole step: F = 24 H (I + H), Q = 8 I + 46 H."""
    return {
        "forward": {"flops": 8 * H * (I + H), "bytes": 2 * I + 12 * H},
        "backward": {"flops": 8 * H * H, "bytes": 34 * H},
        "dx": {"flops": 8 * H * I, "bytes": 4 * I},
        "dw": {"flops": 8 * H * (I + H + 1), "bytes": 2 * I},
        "step": {"flops": 24 * H * (I + H), "bytes": 8 * I + 46 * H},
    }


def roofline_of(work_flops, work_bytes, seconds, peaks, src, sustained):
    tf_peak = peaks["bf16_tflops_sustained" if sustained else "bf16_tflops"]
    t_tensor = work_flops / (tf_peak * 1e12)
    t_hbm = work_bytes / (peaks["hbm_gbs"] * 1e9)
    if t_tensor >= t_hbm:
        ach = work_flops / seconds / 1e12
        return {"bound": "tensor", "achieved": ach, "peak": tf_peak, "unit": "TFLOP/s", "frac": ach / tf_peak,
                "peak_source": "%s bf16 %s" % (src, "sustained" if sustained else "burst")}
    ach = work_bytes / seconds / 1e9
    return {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": ach / peaks["hbm_gbs"], "peak_source": "%s HBM copy" % src}


def phase_kernel(plan, phase):
    """(kernel name, source file) of the kernel that does a phase's work, from the plan."""
    if phase in ("forward", "backward"):
        m = re.search(phase + r" (persistent|per-step|cluster) U=(\d+)", plan)
        if m and m.group(1) == "cluster":
            return "%s<U=%s,%s>" % ("step_cl" if phase == "forward" else "step_clb", m.group(2), phase), "bf16_cluster.cu"
        if m and m.group(1) == "persistent":
            return "step_ws<U=%s,%s>" % (m.group(2), phase), "bf16_persist.cu"
        return ("fwd_step_tc" if phase == "forward" else "bwd_step_tc"), "bf16_path.cu"
    if phase == "dx":
        return "dx_tc", "bf16_path.cu"
    return "dw_ws", "bf16_dw.cu"


def source_sha(fname):
    src = os.path.join(ROOT, "paper_1904_03409_gb300", "csrc", fname)
    return hashlib.sha256(open(src, "rb").read()).hexdigest()[:16]


def kernel_traffic(kernel, fname, workload):
    """DRAM bytes per launch of `kernel` from the committed ncu summary, if it was taken
    on this workload with the kernel source as it is now (or a later revision listed as
    changing host code only); else None."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    sha = source_sha(fname)
    for e in d.get("entries", []):
        same = e.get("source_sha") == sha or sha in e.get("host_only_revisions", [])
        if e.get("kernel") == kernel and e.get("workload") == workload and same:
            return e.get("dram_bytes_per_launch")
    return None


# ---------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples every 100 ms; keeps those taken inside [start, stop]."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.device, self.rows, self.t0, self.t1 = device, [], None, None
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(device), "--query-gpu=" + self.FIELDS,
                                       "--format=csv,noheader,nounits", "-lms", "100"],
                                      stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.th = threading.Thread(target=self._read, daemon=True)
            self.th.start()
        except OSError:
            self.p = None

    def _read(self):
        for line in self.p.stdout:
            self.rows.append((time.time(), [v.strip() for v in line.split(",")]))

    def start(self):
        self.t0 = time.time()

    def stop(self):
        self.t1 = time.time()
        time.sleep(0.25)
        if self.p:
            self.p.terminate()
            try:
                self.p.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.p.kill()

    def summary(self):
        win = [r for t, r in self.rows if self.t0 is not None and self.t0 <= t <= (self.t1 or t)]
        if not win:  # a short timed region: fall back to the samples nearest to it
            win = [r for _, r in self.rows][-3:]
        if not win:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no nvidia-smi samples"], "samples": 0}
        def num(v):
            try:
                return float(v)
            except ValueError:
                return None
        sm = [num(r[1]) for r in win if len(r) > 2 and num(r[1]) is not None]
        smax = [num(r[2]) for r in win if len(r) > 2 and num(r[2]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in win for i in range(4) if len(r) > 5 + i and r[5 + i] == "Active"})
        power = [num(r[3]) for r in win if len(r) > 3 and num(r[3]) is not None]
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "reasons": reasons, "samples": len(win), "power_w_max": max(power) if power else None}


# ------------------------------------------------------------------------- our arm
def run_ours(args, rank, world, local):
    import torch
    from paper_1904_03409_gb300 import binding as bd
    from paper_1904_03409_gb300 import build, runner

    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("gloo")
        if rank == 0:
            build.build()
        dist.barrier()
    else:
        build.build()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    w = get_workload(args.workload, args.T)
    res = measure_workload(w, args.steps, args.warmup, local, world, sample_clocks=True, e2e=True)

    line = {"metric": METRIC, "value": res["value"], "unit": UNIT, "n_gpus": world, "steps": res["steps"],
            "warmup": args.warmup, "ms_per_step": res["ms_per_step"], "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "fp32",
            "data": "synthetic (seeded; shapes and op statistics of the parsing workloads, no treebank)",
            "config": {"workload": describe(w), "B": w.B, "T": w.T, "I": w.I, "H": w.H,
                       "real_step_share": round(w.real_step_share, 4),
                       "l2": "flushed between timed steps (256 MiB write outside the timed events)",
                       "parallelism": "replicas" if world > 1 else "single GPU"},
            "roofline": res["roofline"], "step_roofline": res["step_roofline"], "phases_ms_per_step":
            res["phases"], "e2e": res["e2e"], "gpu_launches": res["gpu_launches"], "clocks": res["clocks"],
            "plan": res["plan"]}
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, args.cpu_seconds)
    if rank == 0 and world == 1 and not args.no_extra and args.workload == "parser64":
        line["other_workloads"] = {}
        for name in ("large", "stress"):
            torch.cuda.empty_cache()
            wx = get_workload(name)
            r = measure_workload(wx, 5, 3, local, 1, sample_clocks=False, e2e=False)
            line["other_workloads"][name] = {"workload": describe(wx), "value": r["value"],
                                             "ms_per_step": r["ms_per_step"], "steps": 5, "warmup": 3,
                                             "roofline": r["roofline"], "step_roofline": r["step_roofline"],
                                             "phases_ms_per_step": r["phases"]}
            del wx
        torch.cuda.empty_cache()
        line["other_workloads"]["arc_hybrid64"] = measure_group("arc_hybrid64", 20, 3, local)
        torch.cuda.empty_cache()
        line["other_workloads"]["parser_step64"] = measure_parser("arc_hybrid64", 20, 3, local)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.barrier()
        dist.destroy_process_group()


def measure_workload(w, steps, warmup, local, world, sample_clocks, e2e):
    import torch
    from paper_1904_03409_gb300 import binding as bd
    from paper_1904_03409_gb300 import runner

    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16 if w.dtype == "bf16" else bd.SL_FP32, local, stream)
    plan = bd.stacklstm_plan(hd)
    bd.stacklstm_set_async(hd, True)
    ins = runner.upload(w, local)
    out = runner.alloc_outputs(w, local, forward_outputs=False)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def step():
        runner.forward_backward(hd, ins, out)

    for _ in range(max(1, warmup)):
        step()
    bd.stacklstm_status(hd)
    if steps <= 0:  # auto: about 2 s of timed work
        t0 = time.time()
        step()
        bd.stacklstm_status(hd)
        steps = int(min(2000, max(10, math.ceil(2.0 / max(time.time() - t0, 1e-4)))))

    bd.stacklstm_set_timing(hd, True)
    launches0 = hd_launches(hd)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    clocks = ClockSampler(local) if sample_clocks else None
    if clocks:
        time.sleep(0.3)
    barrier(world)
    torch.cuda.synchronize(dev)
    if clocks:
        clocks.start()
    for i in range(steps):
        flush.zero_()
        evs[i][0].record(stream)
        step()
        evs[i][1].record(stream)
    torch.cuda.synchronize(dev)
    if clocks:
        clocks.stop()
    barrier(world)
    bd.stacklstm_status(hd)
    total_ms = sum(a.elapsed_time(b) for a, b in evs)
    total_ms = max_over_ranks(total_ms, world)
    timing = bd.stacklstm_get_timing(hd)
    n_launch = hd_launches(hd) - launches0
    bd.stacklstm_set_timing(hd, False)

    peaks, src = load_peaks()
    wk = work_per_inst_step(w.I, w.H)
    phase_ms = {p: timing[p][0] / steps for p in timing}
    dom = max(("forward", "backward", "dx", "dw"), key=lambda p: phase_ms[p])
    kname, kfile = phase_kernel(plan, dom)
    # a persistent step kernel is one launch over all T steps; the per-step kernels are T
    # launches of B instance-steps each; dx and dW are one contraction over all T * B rows
    # (dW: plus its fixed-order reduction of the split partials)
    per_step_kernels = dom in ("forward", "backward") and "step_ws" not in kname and "step_cl" not in kname
    per_launch_units = w.B if per_step_kernels else w.B * w.T
    launches_per_step = w.T if per_step_kernels else 1
    launch_s = phase_ms[dom] / 1e3 / launches_per_step
    fl, by = wk[dom]["flops"], wk[dom]["bytes"]
    m = re.search(r"dx CTAs (\d+)", plan)
    if dom == "backward" and m and int(m.group(1)) > 0:
        # the backward launch also computed dx on the SMs its step chain leaves idle
        fl, by = fl + wk["dx"]["flops"], by + wk["dx"]["bytes"]
        kname += "+dx"
    rf = roofline_of(fl * per_launch_units, by * per_launch_units, launch_s, peaks, src, sustained=True)
    rf.update({"kernel": kname, "phase": dom, "launch_us": launch_s * 1e6,
               "units_per_launch": per_launch_units, "unit_of_work": "instance-step",
               "algorithmic_flops_per_unit": fl, "algorithmic_bytes_per_unit": by,
               "traffic": kernel_traffic(kname, kfile, w.name)})
    sec = total_ms / 1e3 / steps
    srf = roofline_of(wk["step"]["flops"] * w.B * w.T, wk["step"]["bytes"] * w.B * w.T, sec, peaks, src,
                      sustained=True)
    res = {"value": world * w.B * w.T * steps / (total_ms / 1e3), "ms_per_step": total_ms / steps, "steps": steps,
           "roofline": rf, "step_roofline": srf, "phases": {p: round(v, 4) for p, v in phase_ms.items()},
           "plan": plan,
           "gpu_launches": int(n_launch), "clocks": clocks.summary() if clocks else None}
    if e2e:
        res["e2e"] = measure_e2e(w, hd, ins, out, steps, world, local, flush)
    hd.destroy()
    del ins, out, flush
    torch.cuda.empty_cache()
    return res


def measure_group(name, steps, warmup, local):
    """The three StackLSTMs of an arc-hybrid parser batch (stack, buffer, action history),
    forward + backward at the same time, one stream each; against the same three timed one
    at a time. value = instance-steps of all three / second."""
    import torch
    from paper_1904_03409_gb300 import runner, workloads as wl

    g = wl.make_arc_hybrid(**wl.GROUPS[name])
    dev = torch.device("cuda", local)
    cur = torch.cuda.current_stream(dev)
    hds = runner.create_group(g, local)
    ins = {k: runner.upload(g[k], local) for k in runner.GROUP_MEMBERS}
    outs = {k: runner.alloc_outputs(g[k], local, forward_outputs=False) for k in runner.GROUP_MEMBERS}
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    for _ in range(max(1, warmup)):
        runner.group_forward_backward(hds, ins, outs)
    torch.cuda.synchronize(dev)
    runner.group_status(hds)

    def timed(members):
        evs = []
        for _ in range(steps):
            flush.zero_()
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record(cur)
            if members is None:
                runner.group_forward_backward(hds, ins, outs)
            else:
                hd, st = hds[members]
                st.wait_stream(cur)
                runner.forward_backward(hd, ins[members], outs[members])
                cur.wait_stream(st)
            b.record(cur)
            evs.append((a, b))
        torch.cuda.synchronize(dev)
        runner.group_status(hds)
        return sum(x.elapsed_time(y) for x, y in evs) / steps

    ms = timed(None)
    alone = {k: timed(k) for k in runner.GROUP_MEMBERS}
    units = sum(g[k].B * g[k].T for k in runner.GROUP_MEMBERS)
    peaks, src = load_peaks()
    fl = sum(work_per_inst_step(g[k].I, g[k].H)["step"]["flops"] * g[k].B * g[k].T for k in runner.GROUP_MEMBERS)
    by = sum(work_per_inst_step(g[k].I, g[k].H)["step"]["bytes"] * g[k].B * g[k].T for k in runner.GROUP_MEMBERS)
    res = {"workload": "%s: arc-hybrid parser batch, B=%d, n~U[10,60]; stack LSTM T=%d I=%d, buffer LSTM T=%d I=%d "
                       "(n pushes, then a pop per Shift), action LSTM T=%d I=%d; H=%d; seed %d" % (
                           name, g["stack"].B, g["stack"].T, g["stack"].I, g["buffer"].T, g["buffer"].I,
                           g["action"].T, g["action"].I, g["stack"].H, g["stack"].seed),
           "value": units / (ms / 1e3), "unit": "instance-steps/s (three StackLSTMs)",
           "transitions_per_s": g["stack"].B * g["stack"].T / (ms / 1e3),
           "ms_per_step": ms, "ms_one_at_a_time": {k: round(v, 4) for k, v in alone.items()},
           "overlap_speedup": round(sum(alone.values()) / ms, 3), "steps": steps, "warmup": warmup,
           "step_roofline": roofline_of(fl, by, ms / 1e3, peaks, src, sustained=True)}
    for hd, _ in hds.values():
        hd.destroy()
    del ins, outs, flush
    torch.cuda.empty_cache()
    return res


def measure_parser(name, steps, warmup, local):
    """A whole parser training step of the recurrent part on an arc-hybrid batch: the three
    StackLSTM forwards at the same time, the parser head (200-wide ReLU state, softmax over
    the transitions, cross-entropy), the three backwards seeded by the head's gradients.
    value = instance-transitions / second."""
    import torch
    from paper_1904_03409_gb300 import runner, workloads as wl

    g = wl.make_arc_hybrid(**wl.GROUPS[name])
    dev = torch.device("cuda", local)
    cur = torch.cuda.current_stream(dev)
    ps = runner.create_parser(g, local)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    for _ in range(max(1, warmup)):
        runner.parser_step(ps)
    torch.cuda.synchronize(dev)
    runner.group_status(ps["hds"])
    evs = []
    for _ in range(steps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(cur)
        runner.parser_step(ps)
        b.record(cur)
        evs.append((a, b))
    torch.cuda.synchronize(dev)
    runner.group_status(ps["hds"])
    ms = sum(x.elapsed_time(y) for x, y in evs) / steps
    st = g["stack"]
    hp = g["head"]
    res = {"workload": "%s: arc-hybrid parser batch B=%d (as arc_hybrid64) plus the parser head: P=%d ReLU state "
                       "over [stack; buffer; action] tops, softmax over %d transitions, cross-entropy; the "
                       "StackLSTMs' backward seeded only by the head" % (name, st.B, hp["P"], hp["A"]),
           "value": st.B * st.T / (ms / 1e3), "unit": "instance-transitions/s (padded, T=%d)" % st.T,
           "real_transitions_per_s": float(g["L"].sum()) / (ms / 1e3), "ms_per_step": ms, "steps": steps,
           "warmup": warmup}
    runner.destroy_parser(ps)
    del ps, flush
    torch.cuda.empty_cache()
    return res


def hd_launches(hd):
    from paper_1904_03409_gb300 import binding as bd
    return sum(v[1] for v in bd.stacklstm_get_timing(hd).values())


def measure_e2e(w, hd, ins, out, steps, world, local, flush):
    """Same metric through the ABI with the step's inputs copied from pinned host memory
    and its results (all gradients, final pointers) read back, inside the timed events."""
    import torch
    from paper_1904_03409_gb300 import runner

    dev = torch.device("cuda", local)
    stream = torch.cuda.current_stream(dev)
    keys_in = ["x", "ops", "h0", "c0", "W", "bias", "d_top_h"]
    keys_out = ["p_final", "dx", "dh0", "dc0", "dW", "dbias"]
    host_in = {k: ins[k].cpu().pin_memory() for k in keys_in}
    host_out = {k: torch.empty(out[k].shape, dtype=out[k].dtype).pin_memory() for k in keys_out}
    h2d = sum(t.numel() * t.element_size() for t in host_in.values())
    d2h = sum(t.numel() * t.element_size() for t in host_out.values())
    n = max(3, min(steps, 50))
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    barrier(world)
    torch.cuda.synchronize(dev)
    for i in range(n):
        flush.zero_()
        evs[i][0].record(stream)
        for k in keys_in:
            ins[k].copy_(host_in[k], non_blocking=True)
        runner.forward_backward(hd, ins, out)
        for k in keys_out:
            host_out[k].copy_(out[k], non_blocking=True)
        evs[i][1].record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    total = max_over_ranks(sum(a.elapsed_time(b) for a, b in evs), world)
    return {"value": world * w.B * w.T * n / (total / 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": n}


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(v, world):
    if world == 1:
        return v
    import torch
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ CPU (oracle)
def oracle_sample(w, seconds):
    """Instances for about `seconds` of oracle work on all host cores (the whole batch
    when it fits), from a one-instance timing."""
    import oracle
    cores = len(os.sched_getaffinity(0))
    one = [0]
    t0 = time.time()
    oracle.run_instances(one, w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h, nthreads=1)
    t1 = max(time.time() - t0, 1e-6)
    n = int(max(1, min(w.B, math.floor(seconds * cores / t1))))
    return list(range(n)), cores


def run_oracle(w, inst, cores):
    import oracle
    t0 = time.time()
    oracle.run_instances(inst, w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h, dy=w.dy, nthreads=cores)
    return time.time() - t0


def cpu_baseline(w, seconds):
    inst, cores = oracle_sample(w, seconds)
    reps, el = 0, 0.0
    while el < seconds or reps == 0:
        el += run_oracle(w, inst, cores)
        reps += 1
    return {"value": reps * len(inst) * w.T / el, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": "%d of %d instances x %d repetitions (all T=%d steps, forward + backward, fp64), %.1f s"
                      % (len(inst), w.B, reps, w.T, el)}


def run_reference(args, rank, world):
    if rank != 0:
        return
    w = get_workload(args.workload, args.T)
    inst, cores = oracle_sample(w, args.ref_step_seconds)
    for _ in range(args.warmup):
        run_oracle(w, inst, cores)
    times = [run_oracle(w, inst, cores) for _ in range(args.steps if args.steps > 0 else 10)]
    el = sum(times)
    value = len(times) * len(inst) * w.T / el
    sample = "%d of %d instances per step (all T=%d steps, forward + backward, fp64)" % (len(inst), w.B, w.T)
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world,
            "steps": len(times), "warmup": args.warmup, "ms_per_step": 1e3 * el / len(times),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded; shapes and op statistics of the parsing workloads, no treebank)",
            "config": {"workload": describe(w), "B": w.B, "T": w.T, "I": w.I, "H": w.H,
                       "reference": "fp64 CPU oracle (plain C, one instance at a time), host cores"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=0, help="timed steps (0: about 2 s of work)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default="parser64", help="tiny | parser64 | large | stress | sweep:B")
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="oracle CPU-baseline budget")
    ap.add_argument("--ref-step-seconds", type=float, default=3.0, help="oracle work per reference step")
    ap.add_argument("--no-extra", action="store_true", help="skip the large/stress side measurements")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--T", type=int, default=None,
                    help="fewer steps for tiny/large/stress (a smaller case of the same shape, for profiling)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank, world, local = dist_env()
    if world != args.gpus and world > 1:
        print("warning: WORLD_SIZE=%d but --gpus %d" % (world, args.gpus), file=sys.stderr)
    if args.impl == "reference":
        run_reference(args, rank, world)
    else:
        run_ours(args, rank, world, local)


if __name__ == "__main__":
    main()
