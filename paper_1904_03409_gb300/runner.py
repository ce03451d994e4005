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


def run(w, device: int = 0, d_top_h: Optional[np.ndarray] = None) -> dict:
    """Forward + backward of workload ``w`` on ``cuda:device``; numpy results."""
    import torch
    hd = bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16 if w.dtype == "bf16" else bd.SL_FP32, device)
    try:
        ins = upload(w, device)
        out = alloc_outputs(w, device)
        for v in out.values():  # an element the path does not write cannot match the oracle
            if v.is_floating_point():
                v.fill_(float("nan"))
        seed = None if d_top_h is None else torch.from_numpy(np.ascontiguousarray(d_top_h, np.float32)).to(
            ins["x"].device)
        forward_backward(hd, ins, out, d_top_h=seed)
        torch.cuda.synchronize(device)
        return to_numpy(out)
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


def group_status(hds: dict):
    for hd, _ in hds.values():
        bd.stacklstm_status(hd)


def run_group(group: dict, device: int = 0) -> dict:
    """Forward + backward of the three StackLSTMs of a parser workload group at the same
    time (one stream each), into NaN-filled outputs; numpy results per member."""
    import torch
    hds = create_group(group, device)
    try:
        ins = {k: upload(group[k], device) for k in GROUP_MEMBERS}
        outs = {k: alloc_outputs(group[k], device) for k in GROUP_MEMBERS}
        for o in outs.values():
            for v in o.values():
                if v.is_floating_point():
                    v.fill_(float("nan"))
        group_forward_backward(hds, ins, outs)
        torch.cuda.synchronize(device)
        group_status(hds)
        return {k: to_numpy(outs[k]) for k in GROUP_MEMBERS}
    finally:
        for hd, _ in hds.values():
            hd.destroy()
