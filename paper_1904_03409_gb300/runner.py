"""Move a synthetic workload onto the device, run it through the C ABI, read results back.

Marshalling only (numpy <-> torch device tensors); the computation is the library's.
"""
from __future__ import annotations

from typing import Optional

import numpy as np

from . import binding as bd


def upload(w, device: int = 0) -> dict:
    """Device tensors of a workload: inputs in the workload's dtype, c0/bias/seeds fp32."""
    import torch
    dev = torch.device("cuda", device)
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    f = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)
    return dict(x=f(w.x).to(dt), ops=torch.from_numpy(np.ascontiguousarray(w.ops, np.int8)).to(dev),
                h0=f(w.h0).to(dt), c0=f(w.c0), W=f(w.W).to(dt), bias=f(w.bias), d_top_h=f(w.d_top_h),
                dy=None if w.dy is None else f(w.dy))


def alloc_outputs(w, device: int = 0, forward_outputs: bool = True) -> dict:
    import torch
    dev = torch.device("cuda", device)
    dt = torch.bfloat16 if w.dtype == "bf16" else torch.float32
    T, B, I, H = w.T, w.B, w.I, w.H
    e = lambda *s, d=torch.float32: torch.empty(*s, dtype=d, device=dev)
    out = dict(p_final=e(B, d=torch.int32), dx=e(T, B, I), dh0=e(B, H), dc0=e(B, H), dW=e(I + H, 4 * H),
               dbias=e(4 * H))
    if forward_outputs:
        out.update(h_stack=e(T + 1, B, H, d=dt), c_stack=e(T + 1, B, H), p_traj=e(T + 1, B, d=torch.int32),
                   src=e(T + 1, B, d=torch.int32), y=e(T, B, H, d=dt))
    return out


def forward_backward(hd, ins: dict, out: dict, d_top_h=None, dy=None):
    bd.stacklstm_forward(hd, ins["x"], ins["ops"], ins["h0"], ins["c0"], ins["W"], ins["bias"],
                         out.get("h_stack"), out.get("c_stack"), out["p_final"], out.get("p_traj"),
                         out.get("src"), out.get("y"))
    bd.stacklstm_backward(hd, ins["d_top_h"] if d_top_h is None else d_top_h, ins.get("dy") if dy is None else dy,
                          out.get("dx"), out.get("dh0"), out.get("dc0"), out.get("dW"), out.get("dbias"))


def to_numpy(out: dict) -> dict:
    import torch
    res = {}
    for k, v in out.items():
        if v is None:
            continue
        res[k] = (v.float() if v.dtype == torch.bfloat16 else v).cpu().numpy()
    return res


def run(w, device: int = 0, d_top_h: Optional[np.ndarray] = None, mode: int = bd.SL_MODE_HOMOGENIZED) -> dict:
    """Forward + backward of workload ``w`` on ``cuda:device`` in the given mode; numpy
    results (plus ``steps_run``, the steps the step kernels ran)."""
    import torch
    hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16 if w.dtype == "bf16" else bd.SL_FP32, device)
    try:
        if mode != bd.SL_MODE_HOMOGENIZED:
            bd.stacklstm_set_mode(hd, mode)
        ins = upload(w, device)
        out = alloc_outputs(w, device)
        for v in out.values():  # an element the path does not write cannot match the oracle
            if v.is_floating_point():
                v.fill_(float("nan"))
        seed = None if d_top_h is None else torch.from_numpy(np.ascontiguousarray(d_top_h, np.float32)).to(
            ins["x"].device)
        forward_backward(hd, ins, out, d_top_h=seed)
        torch.cuda.synchronize(device)
        res = to_numpy(out)
        res["steps_run"] = bd.stacklstm_steps_run(hd)
        return res
    finally:
        hd.destroy()


GROUP_MEMBERS = ("stack", "buffer", "action")


def create_group(group: dict, device: int = 0) -> dict:
    """One handle per StackLSTM of a parser workload group, each on its own CUDA stream and
    in asynchronous mode, so that their launches can run at the same time."""
    import torch
    hds = {}
    for k in GROUP_MEMBERS:
        w = group[k]
        st = torch.cuda.Stream(device)
        hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16 if w.dtype == "bf16" else bd.SL_FP32, device, st)
        bd.stacklstm_set_async(hd, True)
        hds[k] = (hd, st)
    return hds


def group_forward_backward(hds: dict, ins: dict, outs: dict):
    """Enqueue forward + backward of every member on its own stream, after the current
    stream's work; the current stream then waits for all of them."""
    import torch
    cur = torch.cuda.current_stream()
    for k in GROUP_MEMBERS:
        hd, st = hds[k]
        st.wait_stream(cur)
        forward_backward(hd, ins[k], outs[k])
    for k in GROUP_MEMBERS:
        cur.wait_stream(hds[k][1])


def group_forward_backward_one_call(hds: dict, ins: dict, outs: dict):
    """The same as ``group_forward_backward`` through the grouped calls: one forward call
    and one backward call for the three StackLSTMs, whose step kernels then run as one
    launch each way."""
    import torch
    cur = torch.cuda.current_stream()
    hs = [hds[k][0] for k in GROUP_MEMBERS]
    for k in GROUP_MEMBERS:
        hds[k][1].wait_stream(cur)
    fwd = [dict(x=ins[k]["x"], ops=ins[k]["ops"], h0=ins[k]["h0"], c0=ins[k]["c0"], W=ins[k]["W"], bias=ins[k]["bias"],
                h_stack=outs[k].get("h_stack"), c_stack=outs[k].get("c_stack"), p_final=outs[k]["p_final"],
                p_traj=outs[k].get("p_traj"), src=outs[k].get("src"), y=outs[k].get("y")) for k in GROUP_MEMBERS]
    bwd = [dict(d_top_h=ins[k]["d_top_h"], dy=ins[k].get("dy"), dx=outs[k].get("dx"), dh0=outs[k].get("dh0"),
                dc0=outs[k].get("dc0"), dW=outs[k].get("dW"), dbias=outs[k].get("dbias")) for k in GROUP_MEMBERS]
    bd.stacklstm_forward_group(hs, fwd)
    bd.stacklstm_backward_group(hs, bwd)
    for k in GROUP_MEMBERS:
        cur.wait_stream(hds[k][1])


def group_status(hds: dict):
    for hd, _ in hds.values():
        bd.stacklstm_status(hd)


def run_group(group: dict, device: int = 0, one_call: bool = False) -> dict:
    """Forward + backward of the three StackLSTMs of a parser workload group at the same
    time (one stream each; with ``one_call`` through the grouped calls), into NaN-filled
    outputs; numpy results per member."""
    import torch
    hds = create_group(group, device)
    try:
        ins = {k: upload(group[k], device) for k in GROUP_MEMBERS}
        outs = {k: alloc_outputs(group[k], device) for k in GROUP_MEMBERS}
        for o in outs.values():
            for v in o.values():
                if v.is_floating_point():
                    v.fill_(float("nan"))
        (group_forward_backward_one_call if one_call else group_forward_backward)(hds, ins, outs)
        torch.cuda.synchronize(device)
        group_status(hds)
        return {k: to_numpy(outs[k]) for k in GROUP_MEMBERS}
    finally:
        for hd, _ in hds.values():
            hd.destroy()


def create_parser(group: dict, device: int = 0) -> dict:
    """The three StackLSTM handles of ``create_group`` plus a parser head on the current
    stream, and the device tensors of a whole parser step."""
    import torch
    dev = torch.device("cuda", device)
    hds = create_group(group, device)
    hp, st, bu = group["head"], group["stack"], group["buffer"]
    head = bd.stacklstm_head_create(st.T, bu.T, st.B, st.H, hp["P"], hp["A"], device)
    f = lambda a, dt=torch.float32: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev).to(dt)
    hin = dict(n=torch.from_numpy(group["n"].astype(np.int32)).to(dev), L=torch.from_numpy(group["L"].astype(np.int32)).to(dev),
               gold=torch.from_numpy(group["transitions"].astype(np.int8)).to(dev), Wp=f(hp["Wp"], torch.bfloat16),
               dp=f(hp["dp"]), Wz=f(hp["Wz"]), q=f(hp["q"]))
    e = lambda *s: torch.empty(*s, dtype=torch.float32, device=dev)
    T, Tb, B, H, P, A = st.T, bu.T, st.B, st.H, hp["P"], hp["A"]
    hout = dict(loss_rows=e(T, B), dy_stack=e(T, B, H), dy_buffer=e(Tb, B, H), dy_action=e(T, B, H),
                dWp=e(P, 3 * H), ddp=e(P), dWz=e(A, P), dq=e(A))
    ins = {k: upload(group[k], device) for k in GROUP_MEMBERS}
    outs = {k: alloc_outputs(group[k], device) for k in GROUP_MEMBERS}
    return dict(hds=hds, head=head, hin=hin, hout=hout, ins=ins, outs=outs)


def parser_step(ps: dict):
    """One training step of the parser's recurrent part: the three StackLSTM forwards at
    the same time, the head on the current stream, the three backwards (seeded only by
    the head's gradients) at the same time, then the head's initial-state gradients."""
    import torch
    cur = torch.cuda.current_stream()
    hds, ins, outs, hin, hout = ps["hds"], ps["ins"], ps["outs"], ps["hin"], ps["hout"]
    for k in GROUP_MEMBERS:
        hd, st = hds[k]
        st.wait_stream(cur)
        o, i = outs[k], ins[k]
        bd.stacklstm_forward(hd, i["x"], i["ops"], i["h0"], i["c0"], i["W"], i["bias"], o.get("h_stack"),
                             o.get("c_stack"), o["p_final"], o.get("p_traj"), o.get("src"), o["y"])
    for k in GROUP_MEMBERS:
        cur.wait_stream(hds[k][1])
    bd.stacklstm_head_run(ps["head"], outs["stack"]["y"], ins["stack"]["h0"], outs["buffer"]["y"],
                          outs["action"]["y"], ins["action"]["h0"], hin["n"], hin["L"], hin["gold"], hin["Wp"],
                          hin["dp"], hin["Wz"], hin["q"], hout["loss_rows"], hout["dy_stack"], hout["dy_buffer"],
                          hout["dy_action"], hout["dWp"], hout["ddp"], hout["dWz"], hout["dq"])
    for k in GROUP_MEMBERS:
        hd, st = hds[k]
        st.wait_stream(cur)
        o = outs[k]
        bd.stacklstm_backward(hd, None, hout["dy_" + k], o["dx"], o["dh0"], o["dc0"], o["dW"], o["dbias"])
    for k in GROUP_MEMBERS:
        cur.wait_stream(hds[k][1])
    bd.stacklstm_head_add_h0_grads(ps["head"], outs["stack"]["dh0"], outs["action"]["dh0"])


def destroy_parser(ps: dict):
    for hd, _ in ps["hds"].values():
        hd.destroy()
    ps["head"].destroy()


def run_parser(group: dict, device: int = 0) -> dict:
    """One parser step into NaN-filled outputs; numpy results: {member: outputs} and
    ``head`` (loss rows and the head's gradients)."""
    import torch
    ps = create_parser(group, device)
    try:
        for d in list(ps["outs"].values()) + [ps["hout"]]:
            for v in d.values():
                if v.is_floating_point():
                    v.fill_(float("nan"))
        parser_step(ps)
        torch.cuda.synchronize(device)
        group_status(ps["hds"])
        bd.stacklstm_head_status(ps["head"])
        res = {k: to_numpy(ps["outs"][k]) for k in GROUP_MEMBERS}
        res["head"] = to_numpy(ps["hout"])
        return res
    finally:
        destroy_parser(ps)
