"""Seeded value generators (torch) and length generators (numpy PCG64)."""
import hashlib

import numpy as np
import torch


def seed_for(*key) -> int:
    """A stable 63-bit seed from a tuple of ints/strings (same on every host)."""
    h = hashlib.blake2b(repr(tuple(key)).encode(), digest_size=8).digest()
    return int.from_bytes(h, "little") & ((1 << 63) - 1)


def lengths_rng(*key) -> np.random.Generator:
    return np.random.default_rng(seed_for("lengths", *key))


def _normal_bf16(shape, seed, scale, device):
    g = torch.Generator(device=device)
    g.manual_seed(seed)
    x = torch.randn(shape, generator=g, device=device, dtype=torch.float32)
    if scale != 1.0:
        x.mul_(scale)
    return x.to(torch.bfloat16)


def kv_rows(w, tag, n_tok, device="cpu", layers=None, out=None):
    """K and V rows for one append, bf16 [L][n_tok][Hkv][D] each.

    Every layer is drawn from its own seed (tag, layer, 'k'|'v'), so one layer
    can be regenerated on its own.  ``layers`` restricts the draw to a subset
    (the result then has len(layers) rows in its first dimension).
    """
    layers = list(range(w.n_layers)) if layers is None else list(layers)
    shape = (n_tok, w.n_kv_heads, w.head_dim)
    if out is None:
        k = torch.empty((len(layers),) + shape, dtype=torch.bfloat16, device=device)
        v = torch.empty_like(k)
    else:
        k, v = out
    for i, l in enumerate(layers):
        k[i] = _normal_bf16(shape, seed_for(w.name, w.seed, tag, l, "k"), w.value_scale, device)
        v[i] = _normal_bf16(shape, seed_for(w.name, w.seed, tag, l, "v"), w.value_scale, device)
    return k, v


def queries(w, tag, n_rows, device="cpu", layers=None):
    """Query rows, bf16 [L][n_rows][Hq][D] (one row per branch for decode,
    one per appended token for a merge)."""
    layers = list(range(w.n_layers)) if layers is None else list(layers)
    shape = (n_rows, w.n_q_heads, w.head_dim)
    q = torch.empty((len(layers),) + shape, dtype=torch.bfloat16, device=device)
    for i, l in enumerate(layers):
        q[i] = _normal_bf16(shape, seed_for(w.name, w.seed, tag, l, "q"), w.value_scale, device)
    return q
