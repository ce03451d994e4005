"""fp64 CPU oracle of the parser head after the three StackLSTMs (test infrastructure).

TEST INFRASTRUCTURE ONLY: used by the test suite, the smoke check and the benchmark's
CPU-baseline leg; the product library never imports it, and it imports nothing from the
product package.

The head follows the parser architecture the experiments of Sec. 4.1 use: before each
transition the parser state is built from the tops of the stack, buffer and action-history
StackLSTMs (the output of Algorithm 1), p = ReLU(W_p [s; b; a] + d_p) with a 200-wide
state (Sec. 4.1), then a softmax over the transitions, and the loss is the negative log
probability of the transition taken, summed over transitions and instances.

Which top each transition k of instance b reads (the tops *before* transition k):
- stack:  y_stack[k - 1, b], or the stack's initial state h0_stack[b] when k = 0;
- buffer: y_buffer[n_b - 1 + k, b] (the buffer was filled by n_b pushes first);
- action: y_action[k - 1, b], or h0_action[b] when k = 0.
Transitions k >= L_b (hold padding) contribute nothing.

Written as plain loops over instances and transitions with numpy matrix-vector products,
in the order above; no batching or fusion.
"""
from __future__ import annotations

import numpy as np


def _tops(k, b, n, y_stack, h0_stack, y_buffer, y_action, h0_action):
    s = y_stack[k - 1, b] if k >= 1 else h0_stack[b]
    bu = y_buffer[n[b] - 1 + k, b]
    a = y_action[k - 1, b] if k >= 1 else h0_action[b]
    return np.concatenate([s, bu, a])


def forward_backward(y_stack, h0_stack, y_buffer, y_action, h0_action, n, L, gold, Wp, dp, Wz, q):
    """Loss and gradients of the parser head, fp64.

    Shapes: y_stack, y_action [T, B, H]; y_buffer [Tb, B, H]; h0_* [B, H]; n, L [B];
    gold [T, B] transition ids; Wp [P, 3H]; dp [P]; Wz [A, P]; q [A].
    Returns a dict: loss (scalar), loss_rows [T, B] (0 past L), dy_stack, dy_action
    [T, B, H], dy_buffer [Tb, B, H] (gradients w.r.t. the StackLSTM outputs), dh0_stack,
    dh0_action [B, H] (w.r.t. the initial states read at k = 0), dWp, ddp, dWz, dq.
    """
    f = lambda a: np.asarray(a, dtype=np.float64)
    y_stack, h0_stack, y_buffer, y_action, h0_action = map(f, (y_stack, h0_stack, y_buffer, y_action, h0_action))
    Wp, dp, Wz, q = map(f, (Wp, dp, Wz, q))
    T, B, H = y_stack.shape
    P, A = Wp.shape[0], Wz.shape[0]
    out = dict(loss=0.0, loss_rows=np.zeros((T, B)), dy_stack=np.zeros_like(y_stack),
               dy_buffer=np.zeros_like(y_buffer), dy_action=np.zeros_like(y_action),
               dh0_stack=np.zeros((B, H)), dh0_action=np.zeros((B, H)), dWp=np.zeros_like(Wp),
               ddp=np.zeros(P), dWz=np.zeros_like(Wz), dq=np.zeros(A))
    for b in range(B):
        for k in range(int(L[b])):
            u = _tops(k, b, n, y_stack, h0_stack, y_buffer, y_action, h0_action)
            pre = Wp @ u + dp
            p = np.maximum(pre, 0.0)
            z = Wz @ p + q
            m = z.max()
            lse = m + np.log(np.exp(z - m).sum())
            g = int(gold[k, b])
            out["loss_rows"][k, b] = lse - z[g]
            # backward of the row's loss
            dz = np.exp(z - lse)
            dz[g] -= 1.0
            out["dWz"] += np.outer(dz, p)
            out["dq"] += dz
            dpv = (Wz.T @ dz) * (pre > 0)
            out["dWp"] += np.outer(dpv, u)
            out["ddp"] += dpv
            du = Wp.T @ dpv
            if k >= 1:
                out["dy_stack"][k - 1, b] += du[:H]
                out["dy_action"][k - 1, b] += du[2 * H:]
            else:
                out["dh0_stack"][b] += du[:H]
                out["dh0_action"][b] += du[2 * H:]
            out["dy_buffer"][n[b] - 1 + k, b] += du[H:2 * H]
    out["loss"] = float(out["loss_rows"].sum())
    return out
