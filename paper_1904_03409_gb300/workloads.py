"""Seeded synthetic workloads for the homogenized StackLSTM step.

This module draws the inputs that both the CUDA path and the fp64 oracle consume:
the discrete op streams, x, W, bias and the initial state. It holds none of the
StackLSTM arithmetic -- only random draws, the op-stream generators (which track the
stack depth solely to keep every stream valid) and the round-to-nearest-even
rounding of inputs to bf16, so that both sides see bit-identical input values.

Op encoding follows the unified pointer update of Sec. 3 (p <- p + op): push = +1,
pop = -1, hold = 0 (the hold op is introduced for arc-eager / arc-hybrid, Sec. 3,
last paragraph). The arc-standard stream generator flattens each transition of
Table 1 into primitive stack ops: Shift -> push, Left-Arc -> pop, pop, push,
Right-Arc -> pop.

Random draws use numpy's PCG64 (``numpy.random.default_rng(seed)``) in this fixed
order: (1) per-instance lengths and op choices, instance-major then time;
(2) x in [T, B, I] C order; (3) W; (4) bias, h0 and c0 when a variant asks for them
(zeros otherwise).
"""
from __future__ import annotations

import dataclasses
import math
from typing import Optional, Sequence

import numpy as np

PUSH, POP, HOLD = 1, -1, 0


# ----------------------------------------------------------------------------- bf16
def to_bf16_bits(a: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round to nearest, ties to even); return the bits."""
    u = np.ascontiguousarray(a, dtype=np.float32).view(np.uint32)
    bias = ((u >> np.uint32(16)) & np.uint32(1)) + np.uint32(0x7FFF)
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns exactly to float32."""
    return (np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def round_to_bf16(a: np.ndarray) -> np.ndarray:
    """float32 array holding the bf16-rounded values of ``a``."""
    return bf16_bits_to_f32(to_bf16_bits(a))


# ------------------------------------------------------------------------ op streams
def ops_random_walk(rng: np.random.Generator, B: int, T: int,
                    probs: Sequence[float], lengths: Optional[np.ndarray] = None) -> np.ndarray:
    """Ops [T, B] int8 drawn per step with probabilities (push, pop, hold).

    A pop is never drawn at depth 0: there the pop weight is dropped and the push and
    hold weights are renormalised. Steps at or beyond an instance's length are holds.
    One uniform per (instance, step) is drawn, instance-major.
    """
    w_push, w_pop, w_hold = (float(v) for v in probs)
    u = rng.random((B, T))  # instance-major draw order
    ops = np.zeros((T, B), dtype=np.int8)
    depth = np.zeros(B, dtype=np.int64)
    lim = np.full(B, T, dtype=np.int64) if lengths is None else np.asarray(lengths, dtype=np.int64)
    tot = w_push + w_pop + w_hold
    t_push, t_pop = w_push / tot, (w_push + w_pop) / tot
    t_push0 = w_push / (w_push + w_hold)
    for t in range(T):
        ut = u[:, t]
        at_bottom = depth == 0
        op = np.where(ut < t_push, PUSH, np.where(ut < t_pop, POP, HOLD))
        op0 = np.where(ut < t_push0, PUSH, HOLD)
        op = np.where(at_bottom, op0, op)
        op = np.where(t < lim, op, HOLD)
        ops[t] = op
        depth += op
    return ops


def arc_standard_transitions(rng: np.random.Generator, n: int) -> list:
    """One uniformly random valid arc-standard transition sequence over n tokens.

    At each parser state the next transition is chosen uniformly among the valid ones:
    Shift while the buffer is non-empty, Left-Arc and Right-Arc while the token stack
    holds at least two tokens. The sequence ends with an empty buffer and one token on
    the stack, so it has 2n - 1 transitions.
    """
    buf, stack, seq = n, 0, []
    while buf > 0 or stack > 1:
        valid = []
        if buf > 0:
            valid.append("S")
        if stack >= 2:
            valid += ["LA", "RA"]
        tr = valid[int(rng.integers(len(valid)))]
        seq.append(tr)
        if tr == "S":
            buf -= 1
            stack += 1
        else:
            stack -= 1
    return seq


ARC_STANDARD_OPS = {"S": (PUSH,), "LA": (POP, POP, PUSH), "RA": (POP,)}


def ops_arc_standard(rng: np.random.Generator, B: int, n_range=(10, 60)):
    """Per instance: n ~ U{n_lo..n_hi}, a random valid arc-standard sequence, flattened
    to primitive ops (Table 1) and padded with holds to the batch maximum.
    Returns (ops [T, B] int8, lengths [B] int32)."""
    streams = []
    for _ in range(B):
        n = int(rng.integers(n_range[0], n_range[1] + 1))
        flat = []
        for tr in arc_standard_transitions(rng, n):
            flat.extend(ARC_STANDARD_OPS[tr])
        streams.append(flat)
    T = max(len(s) for s in streams)
    ops = np.zeros((T, B), dtype=np.int8)
    for b, s in enumerate(streams):
        ops[: len(s), b] = s
    return ops, np.array([len(s) for s in streams], dtype=np.int32)


def arc_hybrid_transitions(rng: np.random.Generator, n: int) -> list:
    """One uniformly random valid arc-hybrid transition sequence over n tokens.

    Parser state: a token stack and a buffer holding the tokens not yet shifted. Shift
    (move the buffer front onto the stack) is valid while the buffer is non-empty,
    Left-Arc (the stack top becomes a dependent of the buffer front; pop the stack) while
    both are non-empty, Right-Arc (the stack top becomes a dependent of the token below it;
    pop the stack) while the stack holds at least two tokens. The next transition is chosen
    uniformly among the valid ones; the sequence ends with an empty buffer and one token
    on the stack (the root), after n shifts and n - 1 arcs: 2n - 1 transitions.
    """
    buf, stack, seq = n, 0, []
    while buf > 0 or stack > 1:
        valid = []
        if buf > 0:
            valid.append("S")
        if stack >= 1 and buf > 0:
            valid.append("LA")
        if stack >= 2:
            valid.append("RA")
        tr = valid[int(rng.integers(len(valid)))]
        seq.append(tr)
        if tr == "S":
            buf -= 1
            stack += 1
        else:
            stack -= 1
    return seq


# Table 1, arc-hybrid rows: (stack op, buffer op) of each transition; the action history
# pushes every transition.
ARC_HYBRID_OPS = {"S": (PUSH, POP), "LA": (POP, HOLD), "RA": (POP, HOLD)}
ARC_HYBRID_ACTIONS = ("S", "LA", "RA")


def arc_hybrid_op_streams(seq, n: int) -> dict:
    """The op streams of one sentence's transitions for the three StackLSTMs, and which
    token each step's input is (-1: a zero input).

    buffer: n pushes of tokens n - 1 .. 0 (token 0 ends on top), then per transition its
    buffer op (input zero); stack: per transition its stack op, input the buffer-front
    token (-1 once the buffer is empty); action: a push per transition."""
    out = dict(stack_ops=[], stack_tok=[], buffer_ops=[PUSH] * n, buffer_tok=list(range(n - 1, -1, -1)),
               action_ops=[])
    front = 0
    for tr in seq:
        so, bo = ARC_HYBRID_OPS[tr]
        out["stack_ops"].append(so)
        out["stack_tok"].append(front if front < n else -1)
        out["buffer_ops"].append(bo)
        out["buffer_tok"].append(-1)
        out["action_ops"].append(PUSH)
        if tr == "S":
            front += 1
    return out


# ------------------------------------------------------------------------- workload
@dataclasses.dataclass
class Workload:
    """One batch of synthetic input. Float arrays are float32; for the bf16 path they
    already hold bf16-representable values (x, W, h0), so the oracle and the kernels
    consume bit-identical inputs. c0, bias and the loss seed stay float32."""

    name: str
    T: int
    B: int
    I: int
    H: int
    dtype: str  # "fp32" or "bf16"
    seed: int
    ops: np.ndarray  # [T, B] int8 in {-1, 0, 1}
    lengths: np.ndarray  # [B] int32, real (non-padding) steps per instance
    x: np.ndarray  # [T, B, I]
    W: np.ndarray  # [I + H, 4H], gate column blocks i, f, g, o
    bias: np.ndarray  # [4H]
    h0: np.ndarray  # [B, H]
    c0: np.ndarray  # [B, H]
    d_top_h: np.ndarray  # [B, H] gradient of the loss w.r.t. the final top h
    dy: Optional[np.ndarray] = None  # [T, B, H] gradient w.r.t. y_t, or None

    @property
    def real_step_share(self) -> float:
        return float(self.lengths.sum()) / float(self.T * self.B)

    def bits(self, name: str) -> np.ndarray:
        """bf16 bit pattern of x, W or h0 (bf16 workloads only)."""
        assert self.dtype == "bf16"
        return to_bf16_bits(getattr(self, name))


def make_workload(name: str, T: Optional[int], B: int, I: int, H: int, dtype: str, seed: int,
                  ops_kind: str, probs=(1 / 3, 1 / 3, 1 / 3), len_range=None,
                  bias_scale: float = 0.0, h0_scale: float = 0.0, c0_scale: float = 0.0,
                  dy_scale: float = 0.0, n_range=(10, 60)) -> Workload:
    """Draw one workload. ``ops_kind`` is "random_walk" (needs T and probs, optional
    len_range for ragged hold-padded lengths) or "arc_standard" (T = batch maximum)."""
    rng = np.random.default_rng(seed)
    if ops_kind == "arc_standard":
        ops, lengths = ops_arc_standard(rng, B, n_range)
        T = ops.shape[0]
    elif ops_kind == "random_walk":
        if len_range is not None:
            lengths = rng.integers(len_range[0], len_range[1] + 1, size=B).astype(np.int32)
        else:
            lengths = np.full(B, T, dtype=np.int32)
        ops = ops_random_walk(rng, B, T, probs, lengths)
    else:
        raise ValueError(ops_kind)
    x = rng.standard_normal((T, B, I), dtype=np.float32)
    r = 1.0 / math.sqrt(H)
    W = rng.uniform(-r, r, size=(I + H, 4 * H)).astype(np.float32)
    bias = (rng.uniform(-bias_scale, bias_scale, size=4 * H) if bias_scale else np.zeros(4 * H)).astype(np.float32)
    h0 = (rng.uniform(-h0_scale, h0_scale, size=(B, H)) if h0_scale else np.zeros((B, H))).astype(np.float32)
    c0 = (rng.uniform(-c0_scale, c0_scale, size=(B, H)) if c0_scale else np.zeros((B, H))).astype(np.float32)
    dy = rng.standard_normal((T, B, H), dtype=np.float32) * np.float32(dy_scale) if dy_scale else None
    if dtype == "bf16":
        x, W, h0 = round_to_bf16(x), round_to_bf16(W), round_to_bf16(h0)
    elif dtype != "fp32":
        raise ValueError(dtype)
    return Workload(name=name, T=int(T), B=B, I=I, H=H, dtype=dtype, seed=seed, ops=ops,
                    lengths=lengths, x=x, W=W, bias=bias, h0=h0, c0=c0,
                    d_top_h=np.ones((B, H), dtype=np.float32), dy=dy)


# The five synthetic workloads, shaped like the parsing workloads of Sec. 4.1
# (hidden size 200) and like larger string-to-tree decoders.
CONFIGS = {
    "tiny": dict(T=12, B=4, I=16, H=16, dtype="fp32", seed=0, ops_kind="random_walk",
                 probs=(1 / 3, 1 / 3, 1 / 3)),
    "parser64": dict(T=None, B=64, I=200, H=200, dtype="bf16", seed=1, ops_kind="arc_standard"),
    "sweep": dict(T=None, B=(1, 8, 32, 128, 512, 1024), I=200, H=200, dtype="bf16", seed=2,
                  ops_kind="arc_standard"),
    "large": dict(T=256, B=256, I=512, H=1024, dtype="bf16", seed=3, ops_kind="random_walk",
                  probs=(0.5, 0.3, 0.2), len_range=(64, 256)),
    "stress": dict(T=512, B=4096, I=256, H=256, dtype="bf16", seed=4, ops_kind="random_walk",
                   probs=(0.6, 0.3, 0.1)),
}


def make_arc_hybrid(B: int, seed: int, H: int = 200, I_tok: int = 200, I_act: int = 48, dtype: str = "bf16",
                    n_range=(10, 60), P: int = 200) -> dict:
    """The three StackLSTMs of an arc-hybrid parser over one batch (Table 1), as three
    workloads driven by one transition sequence per instance.

    - ``stack``: per transition, Shift pushes, Left-Arc and Right-Arc pop; its input at
      every step is the representation of the token at the buffer front (zeros once the
      buffer is empty), which is the token a Shift moves onto the stack.
    - ``buffer``: filled first by n pushes of the sentence's token representations, last
      token first, so the first token is on top; then per transition, Shift pops and the
      arcs hold (input zeros).
    - ``action``: the transition history, pushed every transition, input the embedding of
      the transition taken.

    Each is hold-padded to its batch maximum (stack and action 2n - 1 steps, buffer
    3n - 1). Draws, in order: (1) per instance n ~ U{n_lo..n_hi} and its transitions,
    instance-major; (2) token representations [n_hi, B, I_tok]; (3) action embeddings
    [3, I_act]; (4) W of the stack, buffer and action LSTMs, each U(-1/sqrt(H), 1/sqrt(H));
    (5) the parser head's Wp [P, 3H] ~ U(-1/sqrt(3H), 1/sqrt(3H)) and Wz [3, P] ~
    U(-1/sqrt(P), 1/sqrt(P)) (its biases dp, q zero). Biases, h0 and c0 of the StackLSTMs
    are zero; each workload's own loss seed is d(final top h) = 1. Returns a dict with the
    three workloads, ``transitions`` ([T_s, B] int8 action ids, -1 past the end), ``n``
    ([B] sentence lengths), ``L`` ([B] transitions) and ``head`` (Wp, dp, Wz, q).
    """
    rng = np.random.default_rng(seed)
    seqs, ns = [], []
    for _ in range(B):
        n = int(rng.integers(n_range[0], n_range[1] + 1))
        ns.append(n)
        seqs.append(arc_hybrid_transitions(rng, n))
    rep = rng.standard_normal((n_range[1], B, I_tok), dtype=np.float32)
    emb = rng.standard_normal((len(ARC_HYBRID_ACTIONS), I_act), dtype=np.float32)
    r = 1.0 / math.sqrt(H)
    Ws = [rng.uniform(-r, r, size=(I + H, 4 * H)).astype(np.float32) for I in (I_tok, I_tok, I_act)]
    A = len(ARC_HYBRID_ACTIONS)
    Wp = rng.uniform(-1.0 / math.sqrt(3 * H), 1.0 / math.sqrt(3 * H), size=(P, 3 * H)).astype(np.float32)
    Wz = rng.uniform(-1.0 / math.sqrt(P), 1.0 / math.sqrt(P), size=(A, P)).astype(np.float32)
    Ts = max(len(q) for q in seqs)
    Tb = max(n + len(q) for n, q in zip(ns, seqs))
    ops_s, ops_a = np.zeros((Ts, B), np.int8), np.zeros((Ts, B), np.int8)
    ops_b = np.zeros((Tb, B), np.int8)
    x_s, x_a = np.zeros((Ts, B, I_tok), np.float32), np.zeros((Ts, B, I_act), np.float32)
    x_b = np.zeros((Tb, B, I_tok), np.float32)
    trans = np.full((Ts, B), -1, np.int8)
    for b, (n, q) in enumerate(zip(ns, seqs)):
        st = arc_hybrid_op_streams(q, n)
        ops_b[: len(st["buffer_ops"]), b] = st["buffer_ops"]
        ops_s[: len(q), b] = st["stack_ops"]
        ops_a[: len(q), b] = st["action_ops"]
        for t, tok in enumerate(st["buffer_tok"]):
            if tok >= 0:
                x_b[t, b] = rep[tok, b]
        for k, tr in enumerate(q):
            if st["stack_tok"][k] >= 0:
                x_s[k, b] = rep[st["stack_tok"][k], b]
            x_a[k, b] = emb[ARC_HYBRID_ACTIONS.index(tr)]
            trans[k, b] = ARC_HYBRID_ACTIONS.index(tr)
    lens_s = np.array([len(q) for q in seqs], np.int32)
    lens_b = np.array([n + len(q) for n, q in zip(ns, seqs)], np.int32)
    if dtype == "bf16":
        x_s, x_b, x_a = round_to_bf16(x_s), round_to_bf16(x_b), round_to_bf16(x_a)
        Ws = [round_to_bf16(W) for W in Ws]
        Wp = round_to_bf16(Wp)
    elif dtype != "fp32":
        raise ValueError(dtype)
    out = {}
    for name, ops, x, W, lens in (("stack", ops_s, x_s, Ws[0], lens_s), ("buffer", ops_b, x_b, Ws[1], lens_b),
                                  ("action", ops_a, x_a, Ws[2], lens_s)):
        T, I = ops.shape[0], x.shape[2]
        out[name] = Workload(name="arc_hybrid_" + name, T=int(T), B=B, I=I, H=H, dtype=dtype, seed=seed, ops=ops,
                             lengths=lens, x=x, W=W, bias=np.zeros(4 * H, np.float32),
                             h0=np.zeros((B, H), np.float32), c0=np.zeros((B, H), np.float32),
                             d_top_h=np.ones((B, H), dtype=np.float32))
    out["transitions"] = trans
    out["n"] = np.array(ns, np.int32)
    out["L"] = lens_s
    out["head"] = dict(Wp=Wp, dp=np.zeros(P, np.float32), Wz=Wz, q=np.zeros(A, np.float32), P=P, A=A)
    return out


# Parser workloads of three StackLSTMs (stack, buffer, action history) per batch.
GROUPS = {"arc_hybrid64": dict(B=64, seed=5, H=200, I_tok=200, I_act=48, dtype="bf16")}


def config_workload(name: str, B: Optional[int] = None, T: Optional[int] = None) -> Workload:
    """The named workload. ``sweep`` needs B (one of its batch sizes). T, for the workloads
    with a fixed step count (tiny, large, stress), generates the same recipe with fewer
    steps (a smaller case of the same shape, e.g. for profiling)."""
    cfg = dict(CONFIGS[name])
    if T is not None:
        if "T" not in cfg:
            raise ValueError("%s has no fixed step count to change" % name)
        cfg["T"] = T
    if name == "sweep":
        if B is None or B not in cfg["B"]:
            raise ValueError("sweep needs B in %s" % (cfg["B"],))
        cfg["B"] = B
    elif B is not None and B != cfg["B"]:
        raise ValueError("%s has fixed B=%d" % (name, cfg["B"]))
    return make_workload(name=name, **cfg)
