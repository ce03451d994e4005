"""Pins of the parser-head oracle (oracle/parser_head.py) against what the mathematics
fixes: central finite differences, library restatements (torch Linear, relu and
cross_entropy in fp64 over the rows the head reads), a closed form with zero weights, and
which StackLSTM output rows receive gradient."""
import numpy as np
import pytest
import torch

from oracle import parser_head as ph


def case(seed, B=3, H=4, P=5, A=3, n=(2, 4, 3)):
    rng = np.random.default_rng(seed)
    n = np.array(n[:B], np.int32)
    L = 2 * n - 1
    T, Tb = int(L.max()), int((n + L).max())
    d = dict(y_stack=rng.standard_normal((T, B, H)), h0_stack=rng.standard_normal((B, H)),
             y_buffer=rng.standard_normal((Tb, B, H)), y_action=rng.standard_normal((T, B, H)),
             h0_action=rng.standard_normal((B, H)), n=n, L=L,
             gold=np.where(np.arange(T)[:, None] < L[None, :], rng.integers(0, A, (T, B)), -1).astype(np.int8),
             Wp=rng.standard_normal((P, 3 * H)) * 0.7, dp=rng.standard_normal(P) * 0.3,
             Wz=rng.standard_normal((A, P)), q=rng.standard_normal(A) * 0.2)
    return d


def loss_of(d):
    return ph.forward_backward(**d)["loss"]


@pytest.mark.parametrize("seed", [0, 1])
def test_head_gradients_match_central_differences(seed):
    d = case(seed)
    g = ph.forward_backward(**d)
    grads = dict(y_stack="dy_stack", y_buffer="dy_buffer", y_action="dy_action", h0_stack="dh0_stack",
                 h0_action="dh0_action", Wp="dWp", dp="ddp", Wz="dWz", q="dq")
    eps = 1e-6
    for name, gname in grads.items():
        a = d[name]
        num = np.zeros_like(a)
        for idx in np.ndindex(a.shape):
            old = a[idx]
            a[idx] = old + eps
            lp = loss_of(d)
            a[idx] = old - eps
            lm = loss_of(d)
            a[idx] = old
            num[idx] = (lp - lm) / (2 * eps)
        np.testing.assert_allclose(g[gname], num, rtol=1e-5, atol=1e-7, err_msg=name)


def test_head_equals_torch_layers_on_the_rows_it_reads():
    d = case(3, B=3, H=6, P=7, A=4, n=(5, 2, 4))
    g = ph.forward_backward(**d)
    T, B, H = d["y_stack"].shape
    rows, gold = [], []
    for b in range(B):
        for k in range(int(d["L"][b])):
            s = d["y_stack"][k - 1, b] if k else d["h0_stack"][b]
            a = d["y_action"][k - 1, b] if k else d["h0_action"][b]
            rows.append(np.concatenate([s, d["y_buffer"][d["n"][b] - 1 + k, b], a]))
            gold.append(int(d["gold"][k, b]))
    u = torch.tensor(np.stack(rows), dtype=torch.float64)
    lin1 = torch.nn.Linear(3 * H, d["Wp"].shape[0]).double()
    lin2 = torch.nn.Linear(d["Wp"].shape[0], d["Wz"].shape[0]).double()
    with torch.no_grad():
        lin1.weight.copy_(torch.tensor(d["Wp"]))
        lin1.bias.copy_(torch.tensor(d["dp"]))
        lin2.weight.copy_(torch.tensor(d["Wz"]))
        lin2.bias.copy_(torch.tensor(d["q"]))
    loss = torch.nn.functional.cross_entropy(lin2(torch.relu(lin1(u))), torch.tensor(gold), reduction="sum")
    loss.backward()
    np.testing.assert_allclose(g["loss"], loss.item(), rtol=1e-12)
    np.testing.assert_allclose(g["dWp"], lin1.weight.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(g["ddp"], lin1.bias.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(g["dWz"], lin2.weight.grad.numpy(), rtol=1e-10, atol=1e-12)
    np.testing.assert_allclose(g["dq"], lin2.bias.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_head_with_zero_weights_is_the_prior_of_q():
    d = case(4)
    d["Wp"][:] = 0.0
    d["dp"][:] = 0.0
    g = ph.forward_backward(**d)
    q = d["q"]
    lse = np.log(np.exp(q).sum())
    sm = np.exp(q - lse)
    valid = [(k, b) for b in range(len(d["n"])) for k in range(int(d["L"][b]))]
    assert np.isclose(g["loss"], sum(lse - q[d["gold"][k, b]] for k, b in valid))
    want_dq = sum(sm - np.eye(len(q))[d["gold"][k, b]] for k, b in valid)
    np.testing.assert_allclose(g["dq"], want_dq, rtol=1e-12, atol=1e-12)
    for name in ("dWp", "ddp", "dWz", "dy_stack", "dy_buffer", "dy_action", "dh0_stack", "dh0_action"):
        assert np.all(g[name] == 0.0), name


def test_head_reads_exactly_the_tops_before_each_transition():
    d = case(5, B=3, H=4, P=6, A=3, n=(4, 2, 3))
    g = ph.forward_backward(**d)
    T, B, _ = d["y_stack"].shape
    Tb = d["y_buffer"].shape[0]
    for b in range(B):
        n, L = int(d["n"][b]), int(d["L"][b])
        live_s = set(range(L - 1))                    # y_stack[k - 1] for k = 1 .. L - 1
        live_b = set(range(n - 1, n - 1 + L))          # y_buffer[n - 1 + k]
        for t in range(T):
            assert np.any(g["dy_stack"][t, b] != 0) == (t in live_s)
            assert np.any(g["dy_action"][t, b] != 0) == (t in live_s)
        for t in range(Tb):
            assert np.any(g["dy_buffer"][t, b] != 0) == (t in live_b)
        assert np.any(g["dh0_stack"][b] != 0) and np.any(g["dh0_action"][b] != 0)
        assert np.all(g["loss_rows"][L:, b] == 0) and np.all(g["loss_rows"][:L, b] > 0)
    # values in rows the head does not read change nothing
    d2 = {k: (v.copy() if isinstance(v, np.ndarray) else v) for k, v in d.items()}
    d2["y_stack"][int(d["L"][0]) - 1:, 0] = 1e3
    d2["y_buffer"][: int(d["n"][0]) - 1, 0] = -1e3
    assert ph.forward_backward(**d2)["loss"] == g["loss"]
