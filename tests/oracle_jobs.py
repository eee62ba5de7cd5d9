"""The float64 oracle in spawned worker processes (test infrastructure).

The full-size parity checks evaluate the oracle over thousands of branch
contexts of up to 131k keys; one process does about one branch-layer of the
long-trajectory workload per 0.3 s, so the checks run in a pool of worker
processes, one per host core.  A job names each context by the row ranges it
is made of -- (tag, offset, count) pieces drawn by workloads.kv_rows, exactly
as the harness records them -- and the worker redraws those rows itself
(on the same seeded CUDA generator the harness and the library's inputs use)
instead of receiving hundreds of megabytes through a pipe.  Nothing is ever
read back from the library's pool.

The pool is started with the spawn method (never fork: the parent has a CUDA
context), and each worker keeps one BLAS / torch thread.
"""
import os
import sys
from collections import OrderedDict

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)

_CACHE = OrderedDict()
_CACHE_BYTES = [0]
_CACHE_CAP = 2 << 30  # bytes of redrawn rows a worker keeps


def _init():
    for p in (ROOT, HERE):
        if p not in sys.path:
            sys.path.insert(0, p)
    import torch
    torch.set_num_threads(1)


def _rows(w, tag, size, layer):
    from workloads import kv_rows
    key = (w.name, w.seed, tag, size, layer)
    hit = _CACHE.get(key)
    if hit is not None:
        _CACHE.move_to_end(key)
        return hit
    k, v = kv_rows(w, tag, size, device="cuda", layers=[layer])
    val = (k[0].cpu(), v[0].cpu())
    _CACHE[key] = val
    _CACHE_BYTES[0] += 2 * val[0].numel() * 2
    while _CACHE_BYTES[0] > _CACHE_CAP and len(_CACHE) > 1:
        _, (ok, _ov) = _CACHE.popitem(last=False)
        _CACHE_BYTES[0] -= 2 * ok.numel() * 2
    return val


def _context(w, layer, pieces, sizes):
    import torch
    ks, vs = [], []
    for tag, off, cnt in pieces:
        k, v = _rows(w, tag, sizes[tag], layer)
        ks.append(k[off:off + cnt])
        vs.append(v[off:off + cnt])
    return torch.cat(ks), torch.cat(vs)


def _decode_job(w, layer, q, contexts, sizes):
    """q: bf16 [n, Hq, D] (CPU); contexts: n piece lists."""
    from oracle import attention as A
    outs = [A.decode(q[i], *_context(w, layer, pieces, sizes)) for i, pieces in enumerate(contexts)]
    return np.stack([o for o, _ in outs]), np.stack([l for _, l in outs])


def _merge_job(w, layer, q, pieces, sizes, L0, rows):
    """q: bf16 [T, Hq, D] (CPU), the merge's queries at `layer`."""
    from oracle import attention as A
    k, v = _context(w, layer, pieces, sizes)
    return A.merge_prefill(q, k, v, L0, rows=rows)


class OracleJobs:
    """A pool of oracle workers; decode() and merge() return async results
    whose .get() gives (o, lse) as float64 arrays."""

    def __init__(self, n_workers=None):
        import multiprocessing as mp
        n = n_workers or max(1, min(16, os.cpu_count() or 1))
        saved = {}
        for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS"):
            saved[var] = os.environ.get(var)
            os.environ[var] = "1"
        try:
            self._pool = mp.get_context("spawn").Pool(n, initializer=_init)
        finally:
            for var, val in saved.items():
                if val is None:
                    os.environ.pop(var, None)
                else:
                    os.environ[var] = val
        self.n_workers = n

    def decode(self, w, layer, q, contexts, sizes):
        return self._pool.apply_async(_decode_job, (w, layer, q, contexts, sizes))

    def merge(self, w, layer, q, pieces, sizes, L0, rows):
        return self._pool.apply_async(_merge_job, (w, layer, q, pieces, sizes, L0, list(rows)))

    def close(self):
        self._pool.terminate()
        self._pool.join()
