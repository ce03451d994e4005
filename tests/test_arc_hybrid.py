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
