"""The arc-hybrid parser workload: three StackLSTMs (stack, buffer, action history) driven
by one transition sequence per instance (Table 1, arc-hybrid rows).

CPU tests pin the op-stream generator against a brute-force parser-state replay and the
oracle's pointer trajectories; the GPU test runs the three StackLSTMs at the same time
(one stream each) through the C ABI and compares each with the oracle.
"""
import numpy as np
import pytest

import oracle
from paper_1904_03409_gb300 import workloads as wl
from parity import compare


def replay(seq, n):
    """Explicit token stack and buffer: checks each transition's precondition and returns
    the token each Shift moves and the arcs (head, dependent)."""
    stack, buf, shifted, arcs = [], list(range(n)), [], []
    for tr in seq:
        if tr == "S":
            assert buf
            shifted.append(buf[0])
            stack.append(buf.pop(0))
        elif tr == "LA":
            assert stack and buf
            arcs.append((buf[0], stack.pop()))
        else:
            assert tr == "RA" and len(stack) >= 2
            dep = stack.pop()
            arcs.append((stack[-1], dep))
    assert not buf and len(stack) == 1
    return shifted, arcs


def read_golden(name):
    import os
    out = {}
    with open(os.path.join(os.path.dirname(__file__), "golden", name)) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                k, v = line.split(":", 1)
                out[k.strip()] = v.split()
    return out


def test_golden_arc_hybrid_trace():
    """A hand-derived arc-hybrid trace (tests/golden/arc_hybrid_trace.txt, from Table 1,
    Sec. 3 and Algorithm 1): op streams, input tokens, pointer provenance, the arcs, and
    the buffer top the head reads before each transition."""
    g = read_golden("arc_hybrid_trace.txt")
    seq, n = g["transitions"], 3
    ints = lambda v: [int(x) for x in v]
    tok = lambda v: [-1 if x == "-" else int(x) for x in v]
    st = wl.arc_hybrid_op_streams(seq, n)
    for k in ("stack_ops", "buffer_ops", "action_ops"):
        assert st[k] == ints(g[k]), k
    assert st["stack_tok"] == tok(g["stack_tok"]) and st["buffer_tok"] == tok(g["buffer_tok"])
    src = {}
    for name in ("stack", "buffer"):
        ops = np.array(st[name + "_ops"], np.int8)[:, None]
        src[name] = oracle.pointers(ops)["src"][:, 0]
        assert list(src[name]) == ints(g[name + "_src"]), name
    _, arcs = replay(seq, n)
    assert ["%d>%d" % a for a in arcs] == g["arcs"]
    for k in range(len(seq)):
        row = n - 1 + k
        assert row == int(g["head_buffer_row"][k])
        h = int(src["buffer"][row + 1])  # the top after buffer step `row`
        assert (st["buffer_tok"][h - 1] if h > 0 else -1) == tok(g["head_buffer_token"])[k]


@pytest.mark.parametrize("seed", range(5))
def test_arc_hybrid_transitions_are_valid_trees(seed):
    rng = np.random.default_rng(seed)
    for n in (1, 2, 3, 7, 30):
        seq = wl.arc_hybrid_transitions(rng, n)
        assert len(seq) == 2 * n - 1
        shifted, arcs = replay(seq, n)
        assert shifted == list(range(n))
        # every token but the root gets exactly one head: a tree over the n tokens
        deps = [d for _, d in arcs]
        assert sorted(deps) == sorted(set(deps)) and len(deps) == n - 1


def test_arc_hybrid_choices_cover_all_valid_transitions():
    # uniform choice among the valid transitions: each appears, at a plausible rate
    rng = np.random.default_rng(11)
    counts = {"S": 0, "LA": 0, "RA": 0}
    for _ in range(200):
        for tr in wl.arc_hybrid_transitions(rng, 20):
            counts[tr] += 1
    assert counts["S"] == 200 * 20
    assert counts["LA"] > 0.25 * 200 * 19 and counts["RA"] > 0.25 * 200 * 19


def test_arc_hybrid_streams_follow_table1():
    g = wl.make_arc_hybrid(B=9, seed=3, H=16, I_tok=16, I_act=8, dtype="fp32", n_range=(1, 12))
    st, bf, ac, trans, ns = g["stack"], g["buffer"], g["action"], g["transitions"], g["n"]
    ps, pb, pa = (oracle.pointers(w.ops)["p_traj"] for w in (st, bf, ac))
    for b in range(st.B):
        n, L = int(ns[b]), 2 * int(ns[b]) - 1
        seq = [wl.ARC_HYBRID_ACTIONS[i] for i in trans[:L, b]]
        assert np.all(trans[L:, b] == -1)
        shifted, _ = replay(seq, n)
        # stack: push per Shift, pop per arc, one token (the root) at the end
        assert ps[L, b] == 1 and ps[-1, b] == 1 and np.all(ps[:, b] >= 0)
        # buffer: n pushes (last token first), then a pop per Shift; empty at the end
        assert np.all(bf.ops[:n, b] == 1) and pb[n, b] == n and pb[-1, b] == 0
        for k, tr in enumerate(seq):
            assert bf.ops[n + k, b] == (-1 if tr == "S" else 0)
            assert st.ops[k, b] == (1 if tr == "S" else -1)
        # action history: a push per transition
        assert np.all(ac.ops[:L, b] == 1) and pa[-1, b] == L
        # the token a Shift pushes on the stack is the buffer's top, which the buffer
        # pushed (bit for bit) at step n - 1 - token
        k_shift = [k for k, tr in enumerate(seq) if tr == "S"]
        for k, tok in zip(k_shift, shifted):
            assert np.array_equal(st.x[k, b], bf.x[n - 1 - tok, b])
        # holds past each stream's end
        assert np.all(st.ops[L:, b] == 0) and np.all(bf.ops[n + L:, b] == 0) and np.all(ac.ops[L:, b] == 0)


def test_arc_hybrid_oracle_buffer_top_is_forward_lstm_over_reversed_suffix():
    """After the buffer's n pushes and k Shifts, its top is the state built by pushing
    tokens n - 1 .. k: with pushes only up to that point, a plain LSTM over them (the
    oracle's definition mode on the truncated stream gives the same top)."""
    g = wl.make_arc_hybrid(B=4, seed=8, H=8, I_tok=8, I_act=8, dtype="fp32", n_range=(3, 9))
    bf = g["buffer"]
    hom = oracle.run(bf.x, bf.ops, bf.h0, bf.c0, bf.W, bf.bias, d_top_h=bf.d_top_h)
    dfn = oracle.run(bf.x, bf.ops, bf.h0, bf.c0, bf.W, bf.bias, d_top_h=bf.d_top_h, mode="definition")
    np.testing.assert_array_equal(hom["y"], dfn["y"])
    for b in range(bf.B):
        n = int(g["n"][b])
        # after step n - 1 + j (j Shifts done) the top is the state pushed at step n - 1 - j
        p = oracle.pointers(bf.ops)["p_traj"][:, b]
        for t in range(n - 1, bf.T):
            assert p[t + 1] >= 0
        j = 0
        for t in range(n, bf.T):
            if bf.ops[t, b] == -1:
                j += 1
                if j < n:
                    np.testing.assert_array_equal(hom["y"][t, b], hom["y"][n - 1 - j, b])


@pytest.mark.gpu
def test_arc_hybrid_three_stacklstms_at_once_match_oracle():
    import torch
    from paper_1904_03409_gb300 import runner
    g = wl.make_arc_hybrid(**wl.GROUPS["arc_hybrid64"])
    got = runner.run_group(g)
    for k in runner.GROUP_MEMBERS:
        w = g[k]
        ref = oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h)
        compare(got[k], ref, "bf16")
    # the same results as one member at a time on one stream (bit for bit)
    for k in runner.GROUP_MEMBERS:
        alone = runner.run(g[k])
        for name in ("dx", "dW", "dbias", "dh0", "y", "h_stack", "p_traj"):
            assert np.array_equal(got[k][name], alone[name], equal_nan=True), (k, name)
    torch.cuda.empty_cache()


@pytest.mark.gpu
def test_grouped_calls_run_one_step_launch_and_match_oracle():
    """The three StackLSTMs through stacklstm_forward_group / stacklstm_backward_group: their
    step kernels run as one launch each way (counted in the first handle's forward and
    backward phases, none in the others'), and the results equal the oracle's and, bit for
    bit, those of separate calls."""
    import torch
    from paper_1904_03409_gb300 import binding as bd
    from paper_1904_03409_gb300 import runner
    g = wl.make_arc_hybrid(**wl.GROUPS["arc_hybrid64"])
    got = runner.run_group(g, one_call=True)
    sep = runner.run_group(g)
    for k in runner.GROUP_MEMBERS:
        w = g[k]
        compare(got[k], oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=w.d_top_h), "bf16")
        for name in ("dx", "dW", "dbias", "dh0", "dc0", "y", "h_stack", "c_stack", "p_traj", "src"):
            assert np.array_equal(got[k][name], sep[k][name], equal_nan=True), (k, name)
    hds = runner.create_group(g)
    try:
        ins = {k: runner.upload(g[k]) for k in runner.GROUP_MEMBERS}
        outs = {k: runner.alloc_outputs(g[k], forward_outputs=False) for k in runner.GROUP_MEMBERS}
        for hd, _ in hds.values():
            bd.stacklstm_set_timing(hd, True)
        runner.group_forward_backward_one_call(hds, ins, outs)
        torch.cuda.synchronize()
        steps = [(bd.stacklstm_get_timing(hds[k][0])["forward"][1], bd.stacklstm_get_timing(hds[k][0])["backward"][1])
                 for k in runner.GROUP_MEMBERS]
        assert steps == [(1, 1), (0, 0), (0, 0)], steps
    finally:
        for hd, _ in hds.values():
            hd.destroy()
    torch.cuda.empty_cache()


@pytest.mark.gpu
def test_grouped_calls_fall_back_when_the_members_differ():
    """Handles that cannot share one launch (different hidden widths, several row tiles)
    still give the results of separate calls."""
    import torch
    from paper_1904_03409_gb300 import binding as bd
    from paper_1904_03409_gb300 import runner
    ws = [wl.make_workload("m%d" % i, T=T, B=B, I=I, H=H, dtype="bf16", seed=60 + i, ops_kind="random_walk",
                           probs=(0.5, 0.3, 0.2), dy_scale=0.5)
          for i, (T, B, I, H) in enumerate([(12, 40, 24, 48), (9, 40, 16, 32), (10, 130, 16, 48)])]
    hds = [bd.stacklstm_create(w.T, w.B, w.I, w.H, bd.SL_BF16, 0) for w in ws]
    try:
        ins = [runner.upload(w) for w in ws]
        outs = [runner.alloc_outputs(w) for w in ws]
        for o in outs:
            for v in o.values():
                if v.is_floating_point():
                    v.fill_(float("nan"))
        fwd = [dict(x=i["x"], ops=i["ops"], h0=i["h0"], c0=i["c0"], W=i["W"], bias=i["bias"], h_stack=o["h_stack"],
                    c_stack=o["c_stack"], p_final=o["p_final"], p_traj=o["p_traj"], src=o["src"], y=o["y"])
               for i, o in zip(ins, outs)]
        bwd = [dict(d_top_h=i["d_top_h"], dy=i["dy"], dx=o["dx"], dh0=o["dh0"], dc0=o["dc0"], dW=o["dW"],
                    dbias=o["dbias"]) for i, o in zip(ins, outs)]
        bd.stacklstm_forward_group(hds, fwd)
        bd.stacklstm_backward_group(hds, bwd)
        torch.cuda.synchronize()
        for w, o in zip(ws, outs):
            got = runner.to_numpy(o)
            alone = runner.run(w)
            for name in ("dx", "dW", "dbias", "dh0", "dc0", "y", "h_stack", "p_traj"):
                assert np.array_equal(got[name], alone[name], equal_nan=True), (w.name, name)
        with pytest.raises(bd.StackLSTMError) as e:
            bd.stacklstm_forward_group([hds[0], hds[0]], fwd[:1] * 2)
        assert e.value.status == 1
    finally:
        for hd in hds:
            hd.destroy()


def parser_oracle(g, got):
    """The oracle of one parser step, stage by stage on the inputs the GPU stage saw:
    each StackLSTM's forward; the head on the GPU's StackLSTM outputs; each StackLSTM's
    backward seeded by the GPU head's output gradients. Also the head on the oracle's own
    (fp64) outputs, for the end-to-end loss."""
    from oracle import parser_head as ph
    import os
    nt = max(1, len(os.sched_getaffinity(0)))
    hp = g["head"]
    fw = {}
    for k in ("stack", "buffer", "action"):
        w = g[k]
        fw[k] = oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=np.zeros_like(w.h0), nthreads=nt,
                           outputs=("p_traj", "src", "y", "h_stack", "c_stack"))
    args = (g["action"].h0, g["n"], g["L"], g["transitions"], hp["Wp"], hp["dp"], hp["Wz"], hp["q"])
    head = ph.forward_backward(got["stack"]["y"], g["stack"].h0, got["buffer"]["y"], got["action"]["y"], *args)
    head64 = ph.forward_backward(fw["stack"]["y"], g["stack"].h0, fw["buffer"]["y"], fw["action"]["y"], *args)
    bw = {}
    for k in ("stack", "buffer", "action"):
        w = g[k]
        bw[k] = oracle.run(w.x, w.ops, w.h0, w.c0, w.W, w.bias, d_top_h=np.zeros_like(w.h0),
                           dy=got["head"]["dy_" + k], nthreads=nt, outputs=("dx", "dh0", "dc0", "dW", "dbias"))
    bw["stack"]["dh0"] = bw["stack"]["dh0"] + head["dh0_stack"]
    bw["action"]["dh0"] = bw["action"]["dh0"] + head["dh0_action"]
    return fw, head, bw, head64


@pytest.mark.gpu
def test_parser_step_three_stacklstms_and_head_match_oracle():
    """A whole parser step through the C ABI (the three StackLSTMs at the same time, the
    head, the three backwards seeded by the head), each stage against the oracle on the
    inputs that stage received; the total loss against the all-fp64 chain."""
    import torch
    from paper_1904_03409_gb300 import runner
    from parity import BF16_REL
    g = wl.make_arc_hybrid(**wl.GROUPS["arc_hybrid64"])
    got = runner.run_parser(g)
    fw, head, bw, head64 = parser_oracle(g, got)
    for k in runner.GROUP_MEMBERS:
        compare(got[k], fw[k], "bf16", keys=("p_traj", "src", "p_final", "y", "h_stack", "c_stack"))
        compare(got[k], bw[k], "bf16", keys=("dx", "dh0", "dc0", "dW", "dbias"))
    gh = got["head"]
    for name in ("loss_rows", "dy_stack", "dy_buffer", "dy_action", "dWp", "ddp", "dWz", "dq"):
        err = float(np.abs(gh[name].astype(np.float64) - head[name]).max())
        tol = BF16_REL * float(np.abs(head[name]).max())
        assert np.isfinite(err) and err <= tol, (name, err, tol)
    # padding transitions carry no loss; the total loss is close to the all-fp64 chain's
    assert np.all(gh["loss_rows"][g["transitions"] < 0] == 0.0)
    assert abs(gh["loss_rows"].sum() - head64["loss"]) <= 1e-2 * abs(head64["loss"])
    # reproducible bit for bit
    again = runner.run_parser(g)
    for name in ("dWp", "ddp", "dWz", "dq", "dy_buffer"):
        assert np.array_equal(gh[name], again["head"][name]), name
    assert np.array_equal(got["stack"]["dW"], again["stack"]["dW"])
    torch.cuda.empty_cache()


@pytest.mark.gpu
@pytest.mark.parametrize("B,H,P,A,n_hi,seed", [(5, 16, 24, 3, 6, 1), (3, 200, 200, 3, 30, 2), (37, 8, 8, 5, 9, 3)])
def test_parser_head_alone_matches_oracle(B, H, P, A, n_hi, seed):
    """The head on random bf16 StackLSTM outputs (ragged lengths, row tiles with a
    ragged tail, several widths) against the head oracle."""
    import torch
    from oracle import parser_head as ph
    from paper_1904_03409_gb300 import binding as bd
    from parity import BF16_REL
    rng = np.random.default_rng(seed)
    n = rng.integers(1, n_hi + 1, size=B).astype(np.int32)
    L = (2 * n - 1).astype(np.int32)
    T, Tb = int(L.max()), int((n + L).max())
    r = lambda *s: wl.round_to_bf16(rng.standard_normal(s).astype(np.float32))
    ys, yb, ya, h0s, h0a = r(T, B, H), r(Tb, B, H), r(T, B, H), r(B, H), r(B, H)
    gold = np.where(np.arange(T)[:, None] < L[None, :], rng.integers(0, A, (T, B)), -1).astype(np.int8)
    Wp = wl.round_to_bf16((rng.standard_normal((P, 3 * H)) / np.sqrt(3 * H)).astype(np.float32))
    dp = (0.1 * rng.standard_normal(P)).astype(np.float32)
    Wz = (rng.standard_normal((A, P)) / np.sqrt(P)).astype(np.float32)
    q = (0.1 * rng.standard_normal(A)).astype(np.float32)
    want = ph.forward_backward(ys, h0s, yb, ya, h0a, n, L, gold, Wp, dp, Wz, q)
    dev = torch.device("cuda", 0)
    bf = lambda a: torch.from_numpy(a).to(dev).to(torch.bfloat16)
    f = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(dev)
    e = lambda *s: torch.full(s, float("nan"), dtype=torch.float32, device=dev)
    out = dict(loss_rows=e(T, B), dy_stack=e(T, B, H), dy_buffer=e(Tb, B, H), dy_action=e(T, B, H),
               dWp=e(P, 3 * H), ddp=e(P), dWz=e(A, P), dq=e(A))
    hh = bd.stacklstm_head_create(T, Tb, B, H, P, A, 0)
    try:
        bd.stacklstm_head_run(hh, bf(ys), bf(h0s), bf(yb), bf(ya), bf(h0a), torch.from_numpy(n).to(dev),
                              torch.from_numpy(L).to(dev), torch.from_numpy(gold).to(dev), bf(Wp), f(dp), f(Wz), f(q),
                              *out.values())
        dh0s, dh0a = torch.zeros(B, H, device=dev), torch.zeros(B, H, device=dev)
        bd.stacklstm_head_add_h0_grads(hh, dh0s, dh0a)
        bd.stacklstm_head_status(hh)
    finally:
        hh.destroy()
    got = {k: v.cpu().numpy() for k, v in out.items()}
    got["dh0_stack"], got["dh0_action"] = dh0s.cpu().numpy(), dh0a.cpu().numpy()
    for name in got:
        err = float(np.abs(got[name].astype(np.float64) - want[name]).max())
        tol = BF16_REL * max(float(np.abs(want[name]).max()), 1e-30)
        assert np.isfinite(err) and err <= tol, (name, err, tol)
    # rows the head does not read get exactly zero gradient
    assert np.all(got["dy_buffer"][want["dy_buffer"] == 0] == 0)
    assert np.all(got["dy_stack"][want["dy_stack"] == 0] == 0)
