"""Reference attention in float64 -- test infrastructure only.

The paper has no attention formula of its own (it reaches its models through
a serving API, Section 4.1).  What it fixes is where each query looks:

* Section 3.3 (forking): every branch receives the same snapshot H_t + R_t,
  so branch b's context is the shared prefix followed by its own rows.
* Section 3.5 (harvesting): the harvested thoughts are appended after the
  existing context and read in order on the next turn, so thought row i of a
  merge sees the main context plus thought rows 0..i (causal).

Each query attends with the standard scaled softmax, in this project's
reading: scores s_j = (q . k_j) / sqrt(D); lse = log sum_j exp(s_j) (natural
log, scale included); o = sum_j exp(s_j - lse) v_j.  Query head h reads KV
head floor(h / G) with G = Hq / Hkv (contiguous grouping).

Inputs are the exact bf16 values widened to float64; nothing is blocked,
fused, split or reordered beyond one matrix product per head.
"""
import math

import numpy as np


def _f64(x):
    """bf16/fp32 torch tensor or array -> float64 numpy array (exact widening)."""
    try:
        import torch
        if isinstance(x, torch.Tensor):
            return x.detach().to("cpu", torch.float64).numpy()
    except ImportError:  # pragma: no cover
        pass
    return np.asarray(x, dtype=np.float64)


def decode(q, k_ctx, v_ctx):
    """One decode query per head over a materialised context.

    q      [Hq, D]       the branch's query
    k_ctx  [n, Hkv, D]   the branch's keys, logical order (prefix ++ suffix)
    v_ctx  [n, Hkv, D]
    returns o [Hq, D] float64, lse [Hq] float64
    """
    q = _f64(q)
    Hq, D = q.shape
    n, Hkv = k_ctx.shape[0], k_ctx.shape[1]
    if n == 0:
        raise ValueError("decode over an empty context")
    G = Hq // Hkv
    o = np.empty((Hq, D))
    lse = np.empty(Hq)
    for g in range(Hkv):
        # one KV head at a time, widened exactly to float64
        kg, vg = _f64(k_ctx[:, g, :]), _f64(v_ctx[:, g, :])
        for h in range(g * G, (g + 1) * G):
            s = (kg @ q[h]) / math.sqrt(D)
            m = s.max()
            lse[h] = m + math.log(np.exp(s - m).sum())
            o[h] = np.exp(s - lse[h]) @ vg
    return o, lse


def decode_branches(q, contexts):
    """q [n_br, Hq, D]; contexts = list of (k_ctx, v_ctx) per branch."""
    outs = [decode(q[b], *contexts[b]) for b in range(len(contexts))]
    return np.stack([o for o, _ in outs]), np.stack([l for _, l in outs])


def merge_prefill(q, k_all, v_all, L0, rows=None):
    """The merge: thought row i attends over main rows [0, L0 + i] inclusive.

    q      [T, Hq, D]           queries of the appended thought rows
    k_all  [L0 + T, Hkv, D]     main's keys after the append
    v_all  [L0 + T, Hkv, D]
    rows   which thought rows to evaluate (default: all T)
    returns o [len(rows), Hq, D], lse [len(rows), Hq]
    """
    q = _f64(q)
    k, v = k_all, v_all
    T = q.shape[0]
    rows = range(T) if rows is None else rows
    outs = [decode(q[i], k[: L0 + i + 1], v[: L0 + i + 1]) for i in rows]
    return np.stack([o for o, _ in outs]), np.stack([l for _, l in outs])


def combine(partials):
    """Log-sum-exp combine of attention partials over disjoint key sets.

    partials: list of (o_i [.., D], lse_i [..]) each normalised over its own
    keys.  lse = log sum_i exp(lse_i); o = sum_i exp(lse_i - lse) o_i.
    A partial over no keys has lse = -inf and contributes nothing.
    """
    lses = np.stack([_f64(l) for _, l in partials])
    m = lses.max(axis=0)
    lse = m + np.log(np.exp(lses - m).sum(axis=0))
    o = sum(np.exp(_f64(l) - lse)[..., None] * _f64(oi) for oi, l in partials)
    return o, lse
