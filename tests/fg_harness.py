"""Drives the library and the reference pool with the same fork-group
operations, and materialises any branch's context for the oracle.

Each append draws its rows from workloads.kv_rows under a tag; the harness
records, per sequence, which (tag, row range) pieces make up its logical
context (inherited at fork), so the oracle's context for (sequence, layer)
is rebuilt by re-drawing those pieces -- never read back from the GPU pool.
"""
import json
import os
from collections import OrderedDict

import numpy as np
import torch

import paper_2608_13667_gb300 as stpkg
from oracle import attention as A
from oracle import pool as R
from workloads import kv_rows, queries

# Tolerances of the parity target: O within max-abs 2e-3 and max-rel 1e-2 (the
# relative bound over |oracle| >= REL_FLOOR), the log-sum-exp within 1e-4.
O_ABS, O_REL, LSE_ABS = 2e-3, 1e-2, 1e-4
REL_FLOOR = 1e-2


class Run:
    def __init__(self, w, device="cuda", max_seqs=64, max_decode_branches=16, max_splits=16,
                 max_pages=None, pool_seed=None, cache_layers=64):
        self.w = w
        self.device = device
        seed = w.seed if pool_seed is None else pool_seed
        self.pool = stpkg.Pool(n_layers=w.n_layers, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads,
                               head_dim=w.head_dim, n_blocks=w.n_blocks, seed=seed, max_seqs=max_seqs,
                               max_pages=max_pages or min(w.n_blocks, 1 << 16),
                               max_decode_branches=max_decode_branches, max_splits=max_splits,
                               device=device)
        self.ref = R.RefPool(w.n_blocks, seed, max_seqs=max_seqs)
        self.hist = {}
        self.handle = {}
        self.sizes = {}
        self._cache = OrderedDict()
        self._cache_cap = cache_layers

    # -- operations (library and reference in lock-step) ---------------------
    def create(self):
        rid = self.ref.create()
        self.handle[rid] = self.pool.seq_create()
        self.hist[rid] = []
        return rid

    def fork(self, rid, n_aux=4):
        kids = self.ref.fork(rid, n_aux)
        for k, h in zip(kids, self.pool.fork(self.handle[rid], n_aux)):
            self.handle[k] = h
            self.hist[k] = list(self.hist[rid])
        return kids

    def fork_at(self, rid, length, n_aux=4):
        kids = self.ref.fork_at(rid, length, n_aux)
        cut, left = [], length
        for tag, off, cnt in self.hist[rid]:
            if left <= 0:
                break
            take = min(cnt, left)
            cut.append((tag, off, take))
            left -= take
        for k, h in zip(kids, self.pool.fork_at(self.handle[rid], length, n_aux)):
            self.handle[k] = h
            self.hist[k] = list(cut)
        return kids

    def append(self, rids, n_tok, tag):
        w = self.w
        n = len(rids)
        k, v = kv_rows(w, tag, n * n_tok, device=self.device)
        shape = (w.n_layers, n, n_tok, w.n_kv_heads, w.head_dim)
        self.pool.append_kv([self.handle[r] for r in rids], k.view(shape), v.view(shape))
        self.ref.append(rids, n_tok)  # the library accepted it, so the reference must too
        self.sizes[tag] = n * n_tok
        for i, r in enumerate(rids):
            self.hist[r].append((tag, i * n_tok, n_tok))

    def decode(self, rids, tag):
        w = self.w
        q = queries(w, tag, len(rids), device=self.device)
        o, lse = self.pool.decode_attn([self.handle[r] for r in rids], q)
        return q, o, lse

    def merge(self, rid, T, tag):
        w = self.w
        k, v = kv_rows(w, tag, T, device=self.device)
        q = queries(w, ("merge_q",) + tuple(tag), T, device=self.device)
        L0 = self.ref.seqs[rid].length
        o, lse = self.pool.merge(self.handle[rid], q, k, v)
        self.ref.merge(rid, T)
        self.sizes[tag] = T
        self.hist[rid].append((tag, 0, T))
        return q, o, lse, L0

    def prefill_batch(self, rids, counts, tag):
        """Batched prefill: counts[i] rows onto rids[i], packed in that order."""
        w = self.w
        R = sum(counts)
        k, v = kv_rows(w, tag, R, device=self.device)
        q = queries(w, ("prefill_q",) + tuple(tag), R, device=self.device)
        L0 = [self.ref.seqs[r].length for r in rids]
        o, lse = self.pool.prefill_batch([self.handle[r] for r in rids], counts, q, k, v)
        self.ref.prefill_batch(rids, counts)
        self.sizes[tag] = R
        off = 0
        for r, n in zip(rids, counts):
            if n:
                self.hist[r].append((tag, off, n))
            off += n
        return q, o, lse, L0

    def release(self, rid):
        self.ref.release(rid)
        self.pool.release(self.handle[rid])

    # -- oracle side ----------------------------------------------------------
    def _rows(self, tag, layer):
        key = (tag, layer)
        if key in self._cache:
            self._cache.move_to_end(key)
            return self._cache[key]
        k, v = kv_rows(self.w, tag, self.sizes[tag], device=self.device, layers=[layer])
        val = (k[0].cpu(), v[0].cpu())
        self._cache[key] = val
        if len(self._cache) > self._cache_cap:
            self._cache.popitem(last=False)
        return val

    def context(self, rid, layer):
        """(K, V) bf16 [n, Hkv, D] of sequence rid at `layer`, in logical order."""
        ks, vs = [], []
        for tag, off, cnt in self.hist[rid]:
            k, v = self._rows(tag, layer)
            ks.append(k[off:off + cnt])
            vs.append(v[off:off + cnt])
        return torch.cat(ks), torch.cat(vs)

    def oracle_decode(self, rids, q, layer):
        """float64 O [n_br, Hq, D], LSE [n_br, Hq] for one layer."""
        outs = [A.decode(q[layer, i].cpu(), *self.context(r, layer)) for i, r in enumerate(rids)]
        return np.stack([o for o, _ in outs]), np.stack([l for _, l in outs])

    def check_tables(self):
        assert self.pool.refcounts() == self.ref.ref
        assert self.pool.free_list() == list(self.ref.free)
        for rid in self.ref.live():
            table, n = self.pool.block_table(self.handle[rid])
            assert table == self.ref.seqs[rid].table, rid
            assert n == self.ref.seqs[rid].length


def _log(what, n, max_abs, max_rel, max_lse):
    """One JSON line per comparison into $ST_PARITY_LOG, when it is set (the
    achieved-error figures)."""
    path = os.environ.get("ST_PARITY_LOG")
    if not path:
        return
    test = os.environ.get("PYTEST_CURRENT_TEST", "").split(" ")[0]
    with open(path, "a") as f:
        f.write(json.dumps({"test": test, "what": what, "n": int(n), "max_abs": max_abs,
                            "max_rel": max_rel, "max_lse": max_lse}) + "\n")


def compare(o_gpu, lse_gpu, o_ref, lse_ref, what=""):
    """Element-wise check against the oracle, in two forms:
    * the stated target read literally: max |gpu - oracle| <= 2e-3 over all
      O elements, and max |gpu - oracle| / |oracle| <= 1e-2 over the elements
      with |oracle| >= REL_FLOOR (below it a relative error measures nothing
      but the rounding of a value near zero);
    * the allclose reading, |gpu - oracle| <= 2e-3 + 1e-2 |oracle| per
      element (implied by the first; the per-element form of the same bound);
    and |LSE gpu - LSE oracle| <= 1e-4.  Returns (max_abs, max_rel, max_lse)."""
    o = o_gpu.double().cpu().numpy() if isinstance(o_gpu, torch.Tensor) else np.asarray(o_gpu, np.float64)
    l = lse_gpu.double().cpu().numpy() if isinstance(lse_gpu, torch.Tensor) else np.asarray(lse_gpu, np.float64)
    assert o.shape == o_ref.shape and l.shape == lse_ref.shape, what
    assert np.isfinite(o).all() and np.isfinite(l).all(), what
    err = np.abs(o - o_ref)
    big = np.abs(o_ref) >= REL_FLOOR
    max_abs = float(err.max(initial=0.0))
    max_rel = float((err[big] / np.abs(o_ref[big])).max(initial=0.0))
    max_lse = float(np.abs(l - lse_ref).max(initial=0.0))
    _log(what, o.size, max_abs, max_rel, max_lse)
    bad = err > O_ABS + O_REL * np.abs(o_ref)
    assert not bad.any(), f"{what}: {bad.sum()} O elements out of tolerance, max abs {max_abs:.3e}"
    assert max_abs <= O_ABS, f"{what}: max abs O error {max_abs:.3e} > {O_ABS}"
    assert max_rel <= O_REL, f"{what}: max rel O error {max_rel:.3e} > {O_REL}"
    assert max_lse <= LSE_ABS, f"{what}: max lse err {max_lse:.3e}"
    return max_abs, max_rel, max_lse
