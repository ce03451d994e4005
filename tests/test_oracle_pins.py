"""Pins of the fp64 oracle to things other than itself.

Each test fixes part of the oracle against what the paper or mathematics fixes:
 - the all-push stream reduces to a standard LSTM (torch.nn.LSTMCell, fp64, autograd);
 - pointer trajectories and read provenance equal a brute-force list-stack replay and a
   hand-derived trace of a Table 1 transition sequence;
 - a pop followed by a push with the same input rewrites the same state (Sec. 2, Obs. 2);
 - Observation 2: the homogenized mode (Algorithm 1) and the original push/pop
   semantics give identical live results, forward and backward;
 - the analytic backward equals central finite differences and a PyTorch-autograd
   restatement of Algorithm 1 over a batched stack tensor (the paper's own route, Sec. 4.1
   and Sec. 5);
 - dead writes (every pop and hold step) get exactly zero input gradient;
 - with W = 0 every written slot holds a closed-form function of its depth.
"""
import os

import numpy as np
import pytest
import torch

import oracle
from paper_1904_03409_gb300 import workloads as wl

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def rand_case(T, B, I, H, seed, probs=(0.45, 0.35, 0.2), scale=0.6):
    rng = np.random.default_rng(seed)
    ops = wl.ops_random_walk(rng, B, T, probs)
    x = rng.standard_normal((T, B, I))
    W = rng.uniform(-scale, scale, (I + H, 4 * H))
    bias = rng.uniform(-0.3, 0.3, 4 * H)
    h0 = rng.uniform(-0.5, 0.5, (B, H))
    c0 = rng.uniform(-0.5, 0.5, (B, H))
    d_top = rng.standard_normal((B, H))
    dy = rng.standard_normal((T, B, H))
    return dict(x=x, ops=ops, h0=h0, c0=c0, W=W, bias=bias, d_top_h=d_top, dy=dy)


def loss_of(case, out):
    T = case["ops"].shape[0]
    L = float(np.sum(case["d_top_h"] * out["y"][T - 1]))
    if case.get("dy") is not None:
        L += float(np.sum(case["dy"] * out["y"]))
    return L


# --------------------------------------------------------------- standard LSTM (A1)
def torch_cell(W, bias, I, H):
    cell = torch.nn.LSTMCell(I, H).double()
    with torch.no_grad():
        cell.weight_ih.copy_(torch.tensor(W[:I].T))
        cell.weight_hh.copy_(torch.tensor(W[I:].T))
        cell.bias_ih.copy_(torch.tensor(bias))
        cell.bias_hh.zero_()
    return cell


@pytest.mark.parametrize("seed", [0, 1])
def test_all_push_is_standard_lstm(seed):
    T, B, I, H = 9, 3, 5, 4
    c = rand_case(T, B, I, H, seed)
    c["ops"] = np.ones((T, B), np.int8)
    r = oracle.run(**c)
    cell = torch_cell(c["W"], c["bias"], I, H)
    x = torch.tensor(c["x"], requires_grad=True)
    h0 = torch.tensor(c["h0"], requires_grad=True)
    c0 = torch.tensor(c["c0"], requires_grad=True)
    h, cs, ys = h0, c0, []
    for t in range(T):
        h, cs = cell(x[t], (h, cs))
        ys.append(h)
    y = torch.stack(ys)
    L = (y[-1] * torch.tensor(c["d_top_h"])).sum() + (y * torch.tensor(c["dy"])).sum()
    L.backward()
    tol = 1e-12
    assert np.abs(y.detach().numpy() - r["y"]).max() < tol
    # all-push: p_t = t, step t reads slot t (the state written at step t-1)
    assert np.array_equal(r["p_traj"], np.tile(np.arange(T + 1)[:, None], (1, B)))
    assert np.array_equal(r["src"], np.tile(np.arange(T + 1)[:, None], (1, B)))
    assert np.abs(x.grad.numpy() - r["dx"]).max() < tol
    assert np.abs(h0.grad.numpy() - r["dh0"]).max() < tol
    assert np.abs(c0.grad.numpy() - r["dc0"]).max() < tol
    dW = np.concatenate([cell.weight_ih.grad.numpy().T, cell.weight_hh.grad.numpy().T])
    assert np.abs(dW - r["dW"]).max() < tol
    assert np.abs(cell.bias_ih.grad.numpy() - r["dbias"]).max() < tol


# ------------------------------------------------------------------ pointers (Sec. 3)
def replay(ops_col):
    """Brute-force list stack: entries are provenance tags; slot writes per Algorithm 1."""
    slots, p, ps, tops = [0], 0, [0], []
    for t, op in enumerate(ops_col):
        tops.append(slots[p])
        if p + 1 < len(slots):
            slots[p + 1] = t + 1
        else:
            slots.append(t + 1)
        p += int(op)
        assert p >= 0
        ps.append(p)
    tops.append(slots[p])
    return ps, tops


@pytest.mark.parametrize("seed", range(4))
def test_pointers_match_list_stack_replay(seed):
    T, B = 40, 6
    c = rand_case(T, B, 3, 2, seed, probs=(0.4, 0.4, 0.2))
    r = oracle.run(**c, outputs=("p_traj", "src"))
    for b in range(B):
        ps, tops = replay(c["ops"][:, b])
        assert list(r["p_traj"][:, b]) == ps
        assert list(r["src"][:, b]) == tops


def read_golden(name):
    rows = {}
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            k, v = line.split(":", 1)
            rows[k.strip()] = v.split()
    return rows


def test_golden_arc_standard_trace():
    g = read_golden("arc_standard_trace.txt")
    flat = []
    for tr in g["transitions"]:
        flat.extend(wl.ARC_STANDARD_OPS[tr])
    ops = np.array(flat, np.int8)
    assert list(ops) == [int(v) for v in g["ops"]]
    T, I, H = len(ops), 3, 2
    c = rand_case(T, 1, I, H, 7)
    c["ops"] = ops[:, None]
    r = oracle.run(**c)
    assert list(r["p_traj"][:, 0]) == [int(v) for v in g["p"]]
    assert list(r["p_traj"][:-1, 0] + 1) == [int(v) for v in g["written"]]
    assert list(r["src"][:, 0]) == [int(v) for v in g["src"]]
    # final slot-indexed stack: slot s holds the state written at step tag-1 (tag 0 = h0)
    tags = [int(v) for v in g["final_tags"]]
    assert tags[0] == 0 and np.array_equal(r["h_stack"][0, 0], c["h0"][0])
    for s, tag in enumerate(tags[1:], start=1):
        t = tag - 1
        # a live state written at step t is the top after step t, hence y_t
        if r["p_traj"][t + 1, 0] == s:
            assert np.array_equal(r["h_stack"][s, 0], r["y"][t, 0])
    live = dict(kv.split(":") for kv in g["live_slots"])
    assert sorted(int(k) for k in live) == list(range(r["p_traj"][-1, 0] + 1))


# --------------------------------------------------------------- addressing (Obs. 2)
def test_pop_then_push_rewrites_same_state():
    T, B, I, H = 5, 2, 4, 3
    c = rand_case(T, B, I, H, 3)
    c["ops"] = np.array([[1, 1], [1, 0], [-1, -1], [0, 0], [1, 1]], np.int8)
    # the input of step 4 repeats the input of the step that last wrote the slot it rewrites
    c["x"][4, 0] = c["x"][1, 0]  # b=0: slot 2 written at step 1, popped, rewritten at step 4
    c["x"][4, 1] = c["x"][0, 1]  # b=1: step 1 holds (writes slot 2 dead), pop at 2 -> p=0
    r = oracle.run(**c)
    # b=0: p = 0 1 2 1 1 2 ; step 4 reads slot 1 (state of step 0) as step 1 did
    assert list(r["p_traj"][:, 0]) == [0, 1, 2, 1, 1, 2]
    assert np.array_equal(r["y"][4, 0], r["y"][1, 0])
    assert np.array_equal(r["h_stack"][2, 0], r["y"][1, 0])
    # b=1: p = 0 1 1 0 0 1 ; step 4 reads slot 0 (h0) as step 0 did
    assert list(r["p_traj"][:, 1]) == [0, 1, 1, 0, 0, 1]
    assert np.array_equal(r["y"][4, 1], r["y"][0, 1])


@pytest.mark.parametrize("seed", range(3))
def test_definition_equals_homogenized_live(seed):
    T, B, I, H = 30, 5, 4, 3
    c = rand_case(T, B, I, H, seed, probs=(0.4, 0.4, 0.2))
    rh = oracle.run(**c, mode="homogenized")
    rd = oracle.run(**c, mode="definition")
    for k in ("p_traj", "src", "y", "dx", "dh0", "dc0", "dW", "dbias"):
        assert np.array_equal(rh[k], rd[k]), k
    for b in range(B):
        live = rh["p_traj"][-1, b] + 1
        assert np.array_equal(rh["h_stack"][:live, b], rd["h_stack"][:live, b])
        assert np.array_equal(rh["c_stack"][:live, b], rd["c_stack"][:live, b])


@pytest.mark.parametrize("seed", range(4))
def test_only_push_writes_are_ever_read(seed):
    """Observation 2: a state written by a pop or a hold step (to slot p + 1, above the
    top) is overwritten by the next push before the pointer reaches it, so the history
    rows that are ever a top are exactly the initial state and the push steps' writes;
    a brute-force list-stack replay of the slot contents agrees."""
    rng = np.random.default_rng(100 + seed)
    T, B = 60, 7
    ops = wl.ops_random_walk(rng, B, T, (0.4, 0.35, 0.25))
    src = oracle.pointers(ops)["src"]
    for b in range(B):
        read = set(src[:, b].tolist())
        want = {0} | {t + 1 for t in range(T) if ops[t, b] == 1}
        assert read == want
        # replay: slots hold history rows; every step writes slot p + 1, then moves p
        slots, p, tops = [0], 0, [0]
        for t in range(T):
            if len(slots) <= p + 1:
                slots.append(None)
            slots[p + 1] = t + 1
            p += int(ops[t, b])
            tops.append(slots[p])
        assert tops == src[:, b].tolist()


def test_dead_writes_get_zero_input_gradient():
    T, B, I, H = 40, 4, 5, 3
    c = rand_case(T, B, I, H, 11, probs=(0.4, 0.4, 0.2))
    r = oracle.run(**c)
    non_push = c["ops"] != 1
    assert non_push.sum() > 10
    assert np.all(r["dx"][non_push] == 0.0)
    assert np.all(np.abs(r["dx"][~non_push]).sum(-1) > 0)


# ------------------------------------------------------------------------- backward
@pytest.mark.parametrize("seed", [0, 5])
def test_backward_matches_central_differences(seed):
    T, B, I, H = 10, 2, 3, 2
    c = rand_case(T, B, I, H, seed, probs=(0.45, 0.35, 0.2))
    r = oracle.run(**c)
    eps = 1e-6
    worst = 0.0
    for name, grad in (("W", r["dW"]), ("bias", r["dbias"]), ("x", r["dx"]),
                       ("h0", r["dh0"]), ("c0", r["dc0"])):
        base = c[name]
        fd = np.zeros_like(base)
        it = np.nditer(base, flags=["multi_index"])
        for _ in it:
            idx = it.multi_index
            cp = dict(c)
            arr = base.copy()
            arr[idx] += eps
            cp[name] = arr
            lp = loss_of(c, oracle.run(**cp, outputs=("y",)))
            arr[idx] -= 2 * eps
            lm = loss_of(c, oracle.run(**cp, outputs=("y",)))
            fd[idx] = (lp - lm) / (2 * eps)
        scale = max(1.0, np.abs(grad).max())
        err = np.abs(fd - grad).max() / scale
        worst = max(worst, err)
        assert err < 1e-6, (name, err)
    assert worst > 0.0  # the comparison ran on non-trivial numbers


def autograd_algorithm1(c):
    """Algorithm 1 over a batched stack tensor with gather/scatter, gradients by autograd."""
    x = torch.tensor(c["x"], requires_grad=True)
    W = torch.tensor(c["W"], requires_grad=True)
    bias = torch.tensor(c["bias"], requires_grad=True)
    h0 = torch.tensor(c["h0"], requires_grad=True)
    c0 = torch.tensor(c["c0"], requires_grad=True)
    ops = torch.tensor(c["ops"].astype(np.int64))
    T, B = ops.shape
    H = h0.shape[1]
    ar = torch.arange(B)
    Sh = torch.zeros(T + 1, B, H, dtype=torch.float64).index_put((torch.zeros(B, dtype=torch.long), ar), h0)
    Sc = torch.zeros(T + 1, B, H, dtype=torch.float64).index_put((torch.zeros(B, dtype=torch.long), ar), c0)
    p = torch.zeros(B, dtype=torch.long)
    ys = []
    for t in range(T):
        hp, cp = Sh[p, ar], Sc[p, ar]
        z = torch.cat([x[t], hp], 1) @ W + bias
        i, f, g, o = z.split(H, 1)
        i, f, g, o = torch.sigmoid(i), torch.sigmoid(f), torch.tanh(g), torch.sigmoid(o)
        cn = f * cp + i * g
        hn = o * torch.tanh(cn)
        Sh = Sh.index_put((p + 1, ar), hn)
        Sc = Sc.index_put((p + 1, ar), cn)
        p = p + ops[t]
        ys.append(Sh[p, ar])
    y = torch.stack(ys)
    L = (y[-1] * torch.tensor(c["d_top_h"])).sum() + (y * torch.tensor(c["dy"])).sum()
    L.backward()
    return dict(y=y.detach().numpy(), dx=x.grad.numpy(), dW=W.grad.numpy(), dbias=bias.grad.numpy(),
                dh0=h0.grad.numpy(), dc0=c0.grad.numpy())


@pytest.mark.parametrize("seed", [2, 3])
def test_backward_matches_autograd_restatement(seed):
    c = rand_case(24, 4, 5, 3, seed, probs=(0.45, 0.35, 0.2))
    r = oracle.run(**c)
    a = autograd_algorithm1(c)
    for k in ("y", "dx", "dW", "dbias", "dh0", "dc0"):
        assert np.abs(a[k] - r[k]).max() < 1e-10, k


# ----------------------------------------------------------------------- invariants
def test_trailing_holds_and_unbatched_equivalence():
    T, B, I, H = 20, 4, 4, 3
    c = rand_case(T, B, I, H, 9)
    lengths = [20, 13, 7, 1]
    for b, n in enumerate(lengths):
        c["ops"][n:, b] = 0
    c["dy"] = None
    r = oracle.run(**c)
    for b, n in enumerate(lengths):
        one = {k: (v[:, b:b + 1] if k in ("x", "ops") else v[b:b + 1] if k in ("h0", "c0", "d_top_h") else v)
               for k, v in c.items() if v is not None}
        one["x"], one["ops"] = one["x"][:n], one["ops"][:n]
        r1 = oracle.run(**one)
        assert r["p_traj"][-1, b] == r1["p_traj"][-1, 0]
        assert np.array_equal(r["y"][n - 1:, b], np.repeat(r1["y"][n - 1:n, 0], T - n + 1, 0))
        live = r1["p_traj"][-1, 0] + 1
        assert np.array_equal(r["h_stack"][:live, b], r1["h_stack"][:live, 0])
        assert np.array_equal(r["dx"][:n, b], r1["dx"][:, 0])
        assert np.all(r["dx"][n:, b] == 0.0)
        assert np.array_equal(r["dh0"][b], r1["dh0"][0])
        assert np.array_equal(r["dc0"][b], r1["dc0"][0])


def test_batch_permutation():
    c = rand_case(16, 5, 3, 4, 4)
    r = oracle.run(**c)
    perm = np.array([3, 0, 4, 1, 2])
    cp = {k: (v[:, perm] if k in ("x", "ops", "dy") else v[perm] if k in ("h0", "c0", "d_top_h") else v)
          for k, v in c.items()}
    rp = oracle.run(**cp)
    for k in ("p_traj", "src", "y", "dx", "h_stack"):
        assert np.array_equal(rp[k], r[k][:, perm]), k
    for k in ("dh0", "dc0"):
        assert np.array_equal(rp[k], r[k][perm]), k
    assert np.allclose(rp["dW"], r["dW"], rtol=1e-12, atol=1e-14)


def test_holds_only_stream():
    T, B, I, H = 7, 3, 4, 5
    c = rand_case(T, B, I, H, 1)
    c["ops"][:] = 0
    r = oracle.run(**c)
    assert np.all(r["p_traj"] == 0) and np.all(r["src"] == 0)
    assert np.array_equal(r["y"], np.repeat(c["h0"][None], T, 0))
    assert np.allclose(r["dh0"], c["d_top_h"] + c["dy"].sum(0), rtol=0, atol=1e-12)
    assert np.all(r["dc0"] == 0) and np.all(r["dx"] == 0)
    assert np.all(r["dW"] == 0) and np.all(r["dbias"] == 0)


def test_closed_form_with_zero_weights():
    """W = 0 makes every gate a constant, so a state built through j cell applications
    from c0 = 0 has c_j = i g (1 - f^j) / (1 - f) and h_j = o tanh(c_j). Under
    Algorithm 1 every write to slot j comes from slot j-1, so every written slot j holds
    exactly that value."""
    T, B, I, H = 60, 3, 3, 4
    c = rand_case(T, B, I, H, 6, probs=(0.5, 0.3, 0.2))
    c["W"][:] = 0.0
    c["c0"][:] = 0.0
    c["h0"][:] = 0.3
    r = oracle.run(**c)
    b_i, b_f, b_g, b_o = np.split(c["bias"], 4)
    sg = lambda v: 1 / (1 + np.exp(-v))
    i, f, g, o = sg(b_i), sg(b_f), np.tanh(b_g), sg(b_o)
    for b in range(B):
        depth_max = int(r["p_traj"][:-1, b].max()) + 1  # highest slot any step wrote
        for j in range(1, min(depth_max, T) + 1):
            cj = i * g * (1 - f ** j) / (1 - f)
            assert np.allclose(r["c_stack"][j, b], cj, rtol=1e-13, atol=1e-15)
            assert np.allclose(r["h_stack"][j, b], o * np.tanh(cj), rtol=1e-13, atol=1e-15)
    for t in range(T):
        for b in range(B):
            j = r["p_traj"][t + 1, b]
            want = c["h0"][b] if j == 0 else o * np.tanh(i * g * (1 - f ** j) / (1 - f))
            assert np.allclose(r["y"][t, b], want, rtol=1e-13, atol=1e-15)


def test_errors():
    c = rand_case(4, 2, 3, 2, 0)
    c["ops"] = np.array([[1, 1], [-1, -1], [-1, 1], [0, 0]], np.int8)
    with pytest.raises(oracle.OracleError) as e:
        oracle.run(**c)
    assert e.value.code == 2
    c["ops"] = np.array([[1, 2], [0, 0], [0, 0], [0, 0]], np.int8)
    with pytest.raises(oracle.OracleError) as e:
        oracle.run(**c)
    assert e.value.code == 1


def test_pointer_only_entry_matches_full_oracle():
    c = rand_case(60, 9, 3, 2, 12, probs=(0.4, 0.4, 0.2))
    r = oracle.run(**c, outputs=("p_traj", "src"))
    q = oracle.pointers(c["ops"])
    assert np.array_equal(r["p_traj"], q["p_traj"]) and np.array_equal(r["src"], q["src"])
    for b in range(9):
        ps, tops = replay(c["ops"][:, b])
        assert list(q["p_traj"][:, b]) == ps and list(q["src"][:, b]) == tops
