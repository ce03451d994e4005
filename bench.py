#!/usr/bin/env python
"""Forward + backward throughput of the homogenized StackLSTM step on GB300.

One "step" is one pass of the whole hot path over one batch: forward over all T time
steps (Algorithm 1) and the reverse-time backward with dx, dW and dbias. The metric is
instance-steps per second, B * T per step (hold padding included: the homogenized
method computes padded steps too).

  python bench.py [--gpus 1] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

Prints ONE JSON line. The headline is the parser-scale workload (B=64, I=H=200); unless
--workload names one workload or --no-extra is given, the line also carries a full record
(throughput, roofline, clocks, end-to-end rate, CPU baseline, step latency) for every
other workload: tiny, each batch size of the sweep, large, stress, and the arc-hybrid
parser batch. The library runs on one GPU: its one-row-tile kernels deliver operands
between the CTAs of a thread-block cluster with multicast copies, which are for a
process on one GPU; --gpus N > 1 (or a torchrun world larger than one) is refused
before any library call.
--impl reference times the fp64 CPU oracle on the host cores on the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import re
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
# fp32 FFMA peak (the fp32 path runs on CUDA cores, TF32 off): 128 fp32 lanes per SM,
# 2 flops per FFMA, at the maximum SM clock
FP32_LANES_PER_SM = 128
SIDE_WORKLOADS = ("tiny", "sweep:1", "sweep:8", "sweep:32", "sweep:128", "sweep:512", "sweep:1024", "large",
                  "stress")
DATA = "synthetic (seeded; shapes and op statistics of the parsing workloads, no treebank)"


# ----------------------------------------------------------------------------- setup
def dist_env():
    return int(os.environ.get("RANK", 0)), int(os.environ.get("WORLD_SIZE", 1)), int(os.environ.get("LOCAL_RANK", 0))


def get_workload(name, T=None):
    from paper_1904_03409_gb300 import workloads as wl
    if name.startswith("sweep:"):
        return wl.config_workload("sweep", B=int(name.split(":")[1]))
    return wl.config_workload(name, T=T)


def wkey(w):
    """Workload key: the config name, with the batch size for the sweep."""
    return "sweep:%d" % w.B if w.name == "sweep" else w.name


def describe(w):
    ops = {"tiny": "uniform valid push/pop/hold", "parser64": "random valid arc-standard sequences flattened to "
           "push/pop (n~U[10,60]), hold-padded", "large": "push/pop/hold .5/.3/.2, ragged lengths U[64,256], "
           "hold-padded", "stress": "push/pop/hold .6/.3/.1, all real steps", "sweep": "as parser64"}
    return ("%s: B=%d T=%d I=%d H=%d, %s, seed %d" % (wkey(w), w.B, w.T, w.I, w.H, ops.get(w.name, ""), w.seed))


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        peaks = {k: float(d[k]) for k in FALLBACK_PEAKS}
        peaks["sm_max_mhz"] = float(d.get("sm_max_mhz", 2070.0))
        return peaks, "measured"
    peaks = dict(FALLBACK_PEAKS)
    peaks["sm_max_mhz"] = 2070.0
    return peaks, "fallback"


# ---------------------------------------------------------------- algorithmic work
def work_per_inst_step(I, H, dtype="bf16"):
    """Flops and bytes per instance-step, per kernel phase and for the whole step.
    bf16 path: whole step F = 24 H (I + H), Q = 8 I + 46 H. fp32 path: the same flops,
    Q = 12 I + 52 H (4-byte x, h and gates)."""
    if dtype == "fp32":
        return {"forward": {"flops": 8 * H * (I + H), "bytes": 4 * I + 16 * H},
                "backward": {"flops": 8 * H * H, "bytes": 36 * H},
                "dx": {"flops": 8 * H * I, "bytes": 4 * I},
                "dw": {"flops": 8 * H * (I + H + 1), "bytes": 4 * I},
                "step": {"flops": 24 * H * (I + H), "bytes": 12 * I + 52 * H}}
    return {
        "forward": {"flops": 8 * H * (I + H), "bytes": 2 * I + 12 * H},
        "backward": {"flops": 8 * H * H, "bytes": 34 * H},
        "dx": {"flops": 8 * H * I, "bytes": 4 * I},
        "dw": {"flops": 8 * H * (I + H + 1), "bytes": 2 * I},
        "step": {"flops": 24 * H * (I + H), "bytes": 8 * I + 46 * H},
    }


def roofline_of(work_flops, work_bytes, seconds, peaks, src, dtype="bf16", sms=152):
    """The tighter of the contraction's compute roofline and the HBM byte roofline.
    bf16: tensor cores at the measured burst bf16 rate (every timed region here is
    milliseconds long). fp32: CUDA-core FFMA at the peak derived from the SM count, the
    fp32 lanes per SM and the maximum SM clock."""
    if dtype == "fp32":
        peak_t = sms * FP32_LANES_PER_SM * 2 * peaks["sm_max_mhz"] * 1e6 / 1e12
        bound_c, psrc = "alu", "derived fp32 FFMA: %d SMs x %d lanes x 2 flops x %.0f MHz" % (
            sms, FP32_LANES_PER_SM, peaks["sm_max_mhz"])
    else:
        peak_t = peaks["bf16_tflops"]
        bound_c, psrc = "tensor", "%s bf16 burst" % src
    t_c = work_flops / (peak_t * 1e12)
    t_hbm = work_bytes / (peaks["hbm_gbs"] * 1e9)
    if t_c >= t_hbm:
        ach = work_flops / seconds / 1e12
        return {"bound": bound_c, "achieved": ach, "peak": peak_t, "unit": "TFLOP/s", "frac": ach / peak_t,
                "peak_source": psrc}
    ach = work_bytes / seconds / 1e9
    return {"bound": "hbm", "achieved": ach, "peak": peaks["hbm_gbs"], "unit": "GB/s",
            "frac": ach / peaks["hbm_gbs"], "peak_source": "%s HBM copy" % src}


def phase_kernel(plan, phase, dtype):
    """(kernel name, source file, launches per pass) of the kernel that does a phase's
    work, from the plan."""
    if dtype == "fp32":
        if "one CTA" in plan:
            return {"forward": ("fwd_seq_f32", "fp32_path.cu", 1), "backward": ("bwd_seq_f32", "fp32_path.cu", 1),
                    "dx": ("dx_f32", "fp32_path.cu", 1), "dw": ("dw_f32", "fp32_path.cu", 1)}[phase]
        return {"forward": ("fwd_step_f32", "fp32_path.cu", "T"),
                "backward": ("bwd_pointwise_f32+bwd_contract_f32", "fp32_path.cu", "2T"),
                "dx": ("dx_f32", "fp32_path.cu", 1), "dw": ("dw_f32", "fp32_path.cu", 1)}[phase]
    if phase in ("forward", "backward"):
        m = re.search(phase + r" (persistent|per-step|cluster|cuda-core) U=(\d+)", plan)
        if m and m.group(1) == "cuda-core":
            return "%s<BT>" % ("step_ccf" if phase == "forward" else "step_ccb"), "bf16_small.cu", 1
        if m and m.group(1) == "cluster":
            return ("%s<U=%s,%s>" % ("step_cl" if phase == "forward" else "step_clb", m.group(2), phase),
                    "bf16_cluster.cu", 1)
        if m and m.group(1) == "persistent":
            return "step_ws<U=%s,%s>" % (m.group(2), phase), "bf16_persist.cu", 1
        return ("fwd_step_tc" if phase == "forward" else "bwd_step_tc"), "bf16_path.cu", "T"
    if phase == "dx":
        return "dx_tc", "bf16_path.cu", 1
    return "dw_ws", "bf16_dw.cu", 1


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
def run_ours(args):
    import torch
    from paper_1904_03409_gb300 import build

    build.build()
    torch.cuda.set_device(0)
    if args.workload in ("arc_hybrid64", "parser_step64"):
        # the parser workloads alone (their records otherwise ride on the headline line)
        fn = measure_group if args.workload == "arc_hybrid64" else measure_parser
        rec = fn("arc_hybrid64", max(1, args.steps), args.warmup)
        print(json.dumps({"metric": METRIC, "value": rec["value"], "unit": rec["unit"], "n_gpus": 1,
                          "steps": rec["steps"], "warmup": args.warmup, "ms_per_step": rec["ms_per_step"],
                          "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
                          "data": DATA, "config": {"workload": rec["workload"]}, "record": rec}), flush=True)
        return
    w = get_workload(args.workload, args.T)
    rec = measure_record(w, args.steps, args.warmup, args.cpu_seconds, not args.no_cpu_baseline, min_seconds=0.0)
    line = {"metric": METRIC, "value": rec.pop("value"), "unit": UNIT, "n_gpus": 1, "steps": rec.pop("steps"),
            "warmup": args.warmup, "ms_per_step": rec.pop("ms_per_step"), "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16" if w.dtype == "bf16" else "f32",
            "data": DATA, "config": rec.pop("config")}
    line.update(rec)
    if not args.no_extra and args.workload == "parser64" and args.T is None:
        line["workloads"] = {}
        for name in SIDE_WORKLOADS:
            torch.cuda.empty_cache()
            wx = get_workload(name)
            line["workloads"][name] = measure_record(wx, max(20, args.steps), args.warmup, args.side_cpu_seconds,
                                                     not args.no_cpu_baseline, min_seconds=0.3)
            del wx
        torch.cuda.empty_cache()
        line["workloads"]["arc_hybrid64"] = measure_group("arc_hybrid64", max(20, args.steps), args.warmup)
        torch.cuda.empty_cache()
        line["workloads"]["parser_step64"] = measure_parser("arc_hybrid64", max(20, args.steps), args.warmup)
    print(json.dumps(line), flush=True)


def measure_record(w, steps, warmup, cpu_seconds, with_cpu, min_seconds):
    """One workload's full record: device-timed throughput with the clocks seen during
    the timed region, the roofline of its dominant kernel and of the whole step, the
    end-to-end rate through host buffers, per-step latency, and the oracle on the host
    cores as a baseline."""
    res = measure_workload(w, steps, warmup, min_seconds)
    if w.dtype == "bf16":
        # the push-only mode (dead writes skipped, Observation 2 of Sec. 3) on the same
        # workload: same metric (real B * T instance-steps per second), its own roofline
        # over the B * steps_run virtual steps it computes
        res["push_only"] = measure_workload(w, steps, warmup, min_seconds, push_only=True, with_e2e=False)
    res["config"] = {"workload": describe(w), "B": w.B, "T": w.T, "I": w.I, "H": w.H,
                     "real_step_share": round(w.real_step_share, 4),
                     "l2": "flushed between timed steps (256 MiB write outside the timed events)",
                     "parallelism": "single GPU"}
    if with_cpu:
        res["cpu_baseline"] = cpu_baseline(w, cpu_seconds)
    return res


def measure_workload(w, steps, warmup, min_seconds=0.0, push_only=False, with_e2e=True):
    import torch
    from paper_1904_03409_gb300 import binding as bd
    from paper_1904_03409_gb300 import runner

    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(dev)
    hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16 if w.dtype == "bf16" else bd.SL_FP32, 0, stream)
    if push_only:
        bd.stacklstm_set_mode(hd, bd.SL_MODE_PUSH_ONLY)
    plan = bd.stacklstm_plan(hd)
    bd.stacklstm_set_async(hd, True)
    ins = runner.upload(w, 0)
    out = runner.alloc_outputs(w, 0, forward_outputs=False)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)

    def step():
        runner.forward_backward(hd, ins, out)

    for _ in range(max(1, warmup)):
        step()
    bd.stacklstm_status(hd)
    if steps <= 0 or min_seconds > 0:  # auto (or a floor): time enough steps for the clock samples
        t0 = time.time()
        step()
        bd.stacklstm_status(hd)
        one = max(time.time() - t0, 1e-5)
        want = 2.0 if steps <= 0 else min_seconds
        steps = int(min(2000, max(steps, 10, math.ceil(want / one))))

    launches0 = hd_launches(hd)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    clocks = ClockSampler(0)
    time.sleep(0.3)
    torch.cuda.synchronize(dev)
    clocks.start()
    for i in range(steps):
        flush.zero_()
        evs[i][0].record(stream)
        step()
        evs[i][1].record(stream)
    torch.cuda.synchronize(dev)
    clocks.stop()
    bd.stacklstm_status(hd)
    total_ms = sum(a.elapsed_time(b) for a, b in evs)
    n_launch = hd_launches(hd) - launches0
    # the per-phase breakdown (the library's own events around each phase) from separate
    # passes, so that its event records stay out of the timed ones
    n_ph = min(steps, 20)
    bd.stacklstm_set_timing(hd, True)
    for i in range(n_ph):
        flush.zero_()
        step()
    torch.cuda.synchronize(dev)
    bd.stacklstm_status(hd)
    timing = bd.stacklstm_get_timing(hd)
    bd.stacklstm_set_timing(hd, False)
    Tr = bd.stacklstm_steps_run(hd)  # T, or the virtual steps of the push-only mode

    peaks, src = load_peaks()
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    wk = work_per_inst_step(w.I, w.H, w.dtype)
    phase_ms = {p: timing[p][0] / n_ph for p in timing}
    dom = max(("forward", "backward", "dx", "dw"), key=lambda p: phase_ms[p])
    kname, kfile, lpp = phase_kernel(plan, dom, w.dtype)
    # a persistent or cluster step kernel is one launch over all T steps; the per-step
    # kernels are T (or 2T) launches of B instance-steps each; dx and dW are one
    # contraction over all T * B rows (dW: plus its fixed-order reduction of the partials)
    launches_per_pass = {"T": Tr, "2T": 2 * Tr}.get(lpp, lpp)
    per_launch_units = w.B * Tr / launches_per_pass
    launch_s = phase_ms[dom] / 1e3 / launches_per_pass
    fl, by = wk[dom]["flops"], wk[dom]["bytes"]
    m = re.search(r"dx CTAs (\d+)", plan)
    if dom == "backward" and m and int(m.group(1)) > 0:
        # the backward launch also computed dx on the SMs its step chain leaves idle
        fl, by = fl + wk["dx"]["flops"], by + wk["dx"]["bytes"]
        kname += "+dx"
    rf = roofline_of(fl * per_launch_units, by * per_launch_units, launch_s, peaks, src, w.dtype, sms)
    rf.update({"kernel": kname, "phase": dom, "launch_us": launch_s * 1e6,
               "launches_per_pass": launches_per_pass, "units_per_launch": per_launch_units,
               "unit_of_work": "instance-step", "algorithmic_flops_per_unit": fl,
               "algorithmic_bytes_per_unit": by, "traffic": kernel_traffic(kname, kfile, wkey(w))})
    sec = total_ms / 1e3 / steps
    srf = roofline_of(wk["step"]["flops"] * w.B * Tr, wk["step"]["bytes"] * w.B * Tr, sec, peaks, src, w.dtype, sms)
    res = {"value": w.B * w.T * steps / (total_ms / 1e3), "ms_per_step": total_ms / steps, "steps": steps,
           "roofline": rf, "step_roofline": srf, "phases_ms_per_step": {p: round(v, 4) for p, v in phase_ms.items()},
           "step_latency_us": {"forward": 1e3 * phase_ms["forward"] / Tr,
                               "backward": 1e3 * (phase_ms["backward"] + phase_ms["dx"]) / Tr},
           "steps_run": Tr, "plan": plan, "gpu_launches": int(n_launch), "clocks": clocks.summary()}
    if with_e2e:
        res["e2e"] = measure_e2e(w, hd, ins, out, steps, flush)
    hd.destroy()
    del ins, out, flush
    torch.cuda.empty_cache()
    return res


def measure_group(name, steps, warmup):
    """The three StackLSTMs of an arc-hybrid parser batch (stack, buffer, action history),
    forward + backward through the grouped calls (their step kernels as one launch each
    way); beside it, the same three as separate calls on three streams, and each timed
    alone. value = instance-steps of all three / second through the grouped calls."""
    import torch
    from paper_1904_03409_gb300 import runner, workloads as wl

    g = wl.make_arc_hybrid(**wl.GROUPS[name])
    dev = torch.device("cuda", 0)
    cur = torch.cuda.current_stream(dev)
    hds = runner.create_group(g, 0)
    ins = {k: runner.upload(g[k], 0) for k in runner.GROUP_MEMBERS}
    outs = {k: runner.alloc_outputs(g[k], 0, forward_outputs=False) for k in runner.GROUP_MEMBERS}
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
            if members == "one_call":
                runner.group_forward_backward_one_call(hds, ins, outs)
            elif members is None:
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

    clocks = ClockSampler(0)
    time.sleep(0.3)
    clocks.start()
    ms = timed("one_call")
    clocks.stop()
    ms_streams = timed(None)
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
           "ms_per_step": ms, "ms_three_streams_separate_calls": ms_streams,
           "ms_one_at_a_time": {k: round(v, 4) for k, v in alone.items()},
           "overlap_speedup": round(sum(alone.values()) / ms, 3), "steps": steps, "warmup": warmup,
           "step_roofline": roofline_of(fl, by, ms / 1e3, peaks, src), "clocks": clocks.summary()}
    for hd, _ in hds.values():
        hd.destroy()
    del ins, outs, flush
    torch.cuda.empty_cache()
    return res


def measure_parser(name, steps, warmup):
    """A whole parser training step of the recurrent part on an arc-hybrid batch: the three
    StackLSTM forwards at the same time, the parser head (200-wide ReLU state, softmax over
    the transitions, cross-entropy), the three backwards seeded by the head's gradients.
    value = instance-transitions / second."""
    import torch
    from paper_1904_03409_gb300 import runner, workloads as wl

    g = wl.make_arc_hybrid(**wl.GROUPS[name])
    dev = torch.device("cuda", 0)
    cur = torch.cuda.current_stream(dev)
    ps = runner.create_parser(g, 0)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    for _ in range(max(1, warmup)):
        runner.parser_step(ps)
    torch.cuda.synchronize(dev)
    runner.group_status(ps["hds"])
    evs = []
    clocks = ClockSampler(0)
    time.sleep(0.3)
    clocks.start()
    for _ in range(steps):
        flush.zero_()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(cur)
        runner.parser_step(ps)
        b.record(cur)
        evs.append((a, b))
    torch.cuda.synchronize(dev)
    clocks.stop()
    runner.group_status(ps["hds"])
    ms = sum(x.elapsed_time(y) for x, y in evs) / steps
    st = g["stack"]
    hp = g["head"]
    res = {"workload": "%s: arc-hybrid parser batch B=%d (as arc_hybrid64) plus the parser head: P=%d ReLU state "
                       "over [stack; buffer; action] tops, softmax over %d transitions, cross-entropy; the "
                       "StackLSTMs' backward seeded only by the head" % (name, st.B, hp["P"], hp["A"]),
           "value": st.B * st.T / (ms / 1e3), "unit": "instance-transitions/s (padded, T=%d)" % st.T,
           "real_transitions_per_s": float(g["L"].sum()) / (ms / 1e3), "ms_per_step": ms, "steps": steps,
           "warmup": warmup, "clocks": clocks.summary()}
    runner.destroy_parser(ps)
    del ps, flush
    torch.cuda.empty_cache()
    return res


def hd_launches(hd):
    from paper_1904_03409_gb300 import binding as bd
    return sum(v[1] for v in bd.stacklstm_get_timing(hd).values())


def packed(tensors: dict, keys, device=None, align: int = 256):
    """One buffer (pinned host memory, or device memory) holding the given tensors back to
    back at 256-byte-aligned offsets; returns (buffer, {key: view of the buffer with that
    tensor's dtype and shape})."""
    import torch
    offs, n = {}, 0
    for k in keys:
        t = tensors[k]
        n = (n + align - 1) // align * align
        offs[k] = n
        n += t.numel() * t.element_size()
    buf = (torch.empty(n, dtype=torch.uint8, device=device) if device is not None
           else torch.empty(n, dtype=torch.uint8).pin_memory())
    views = {k: buf[offs[k]:offs[k] + tensors[k].numel() * tensors[k].element_size()].view(tensors[k].dtype)
             .view(tensors[k].shape) for k in keys}
    return buf, views


def measure_e2e(w, hd, ins, out, steps, flush):
    """Same metric through the ABI with the step's inputs copied from pinned host memory
    and its results (all gradients, final pointers) read back, inside the timed events. The
    inputs live in one pinned host buffer and one device buffer, and so do the results (each
    tensor a 256-byte-aligned view the library reads or writes in place): one copy each way
    a step, the same bytes as a copy per tensor, without a copy's fixed cost per tensor."""
    import torch
    from paper_1904_03409_gb300 import runner

    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(dev)
    keys_in = ["x", "ops", "h0", "c0", "W", "bias", "d_top_h"]
    keys_out = ["p_final", "dx", "dh0", "dc0", "dW", "dbias"]
    host_in_buf, host_in = packed(ins, keys_in)
    for k in keys_in:
        host_in[k].copy_(ins[k].cpu())
    dev_in_buf, dev_in = packed(ins, keys_in, dev)
    host_out_buf, _ = packed(out, keys_out)
    dev_out_buf, dev_out = packed(out, keys_out, dev)
    ins_e = dict(ins, **dev_in)
    out_e = dict(out, **dev_out)
    h2d = host_in_buf.numel()
    d2h = host_out_buf.numel()
    n = max(3, min(steps, 50))
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(n)]
    torch.cuda.synchronize(dev)
    for i in range(n):
        flush.zero_()
        evs[i][0].record(stream)
        dev_in_buf.copy_(host_in_buf, non_blocking=True)
        runner.forward_backward(hd, ins_e, out_e)
        host_out_buf.copy_(dev_out_buf, non_blocking=True)
        evs[i][1].record(stream)
    torch.cuda.synchronize(dev)
    total = sum(a.elapsed_time(b) for a, b in evs)
    return {"value": w.B * w.T * n / (total / 1e3), "unit": UNIT, "h2d_bytes_per_step": int(h2d),
            "d2h_bytes_per_step": int(d2h), "steps": n}


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
    return list(range(n)), min(cores, n)


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


def run_reference(args, world):
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
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": DATA,
            "config": {"workload": describe(w), "B": w.B, "T": w.T, "I": w.I, "H": w.H,
                       "reference": "fp64 CPU oracle (plain C, one instance at a time), host cores"},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1, help="must be 1: the library runs on one GPU")
    ap.add_argument("--steps", type=int, default=0, help="timed steps (0: about 2 s of work)")
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=("ours", "reference"), default="ours")
    ap.add_argument("--workload", default="parser64",
                    help="tiny | parser64 | large | stress | sweep:B | arc_hybrid64 | parser_step64")
    ap.add_argument("--cpu-seconds", type=float, default=10.0, help="oracle CPU-baseline budget (headline)")
    ap.add_argument("--side-cpu-seconds", type=float, default=3.0, help="oracle CPU-baseline budget (others)")
    ap.add_argument("--ref-step-seconds", type=float, default=3.0, help="oracle work per reference step")
    ap.add_argument("--no-extra", action="store_true", help="the named workload only")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--T", type=int, default=None,
                    help="fewer steps for tiny/large/stress (a smaller case of the same shape, for profiling)")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    rank, world, _ = dist_env()
    if args.impl == "reference":
        # the oracle runs on the host cores: rank 0 alone under torchrun
        if rank == 0:
            run_reference(args, world)
        return
    if args.gpus != 1 or world > 1:
        print("bench.py: this library runs on one GPU (its one-row-tile kernels use cluster multicast "
              "copies, which are for a process on one GPU); run it with --gpus 1 and no torchrun world",
              file=sys.stderr)
        sys.exit(2)
    run_ours(args)


if __name__ == "__main__":
    main()
