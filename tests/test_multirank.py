"""The N > 1 path on CPU with gloo, world size 2.

Fork groups are independent, so ranks run replicas with no data-path
collective; what crosses ranks is (a) the max-over-ranks timing of the
bench and (b), where one long prefix is split across GPUs, the exchange of
split-KV partials that the log-sum-exp combine merges.  Both are exercised
here with processes on CPU (the block pool runs metadata-only)."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from conftest import ROOT


def _port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _env(rank, ws, port):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(ws), LOCAL_RANK=str(rank))


def _replica_worker(rank, ws, port, out):
    import sys
    sys.path.insert(0, ROOT)
    _env(rank, ws, port)
    import torch.distributed as dist
    import bench
    import paper_2608_13667_gb300 as st
    from workloads import get
    r, w_, local = bench._dist(backend="gloo")
    w = get(4)
    # each rank owns a full replica of the long-trajectory pool (metadata only)
    pool = st.Pool(n_layers=w.n_layers, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads,
                   head_dim=w.head_dim, n_blocks=w.n_blocks, seed=w.seed, device=None, **w.limits)
    br = []
    for t in range(w.n_tasks):
        m = pool.seq_create()
        pool.append_kv([m], w.prefix[t], None)
        kids = pool.fork(m, w.n_aux)
        for h, s in zip([m] + kids, w.suffix[t]):
            if s:
                pool.append_kv([h], s, None)
        br += [m] + kids
    pool.append_kv(br, 1, None)
    digest = hash(tuple(pool.refcounts()))
    slowest = bench._allreduce_max(float(10 * (rank + 1)), ws)
    got = [None] * ws
    dist.all_gather_object(got, (rank, digest, len(br)))
    bench._barrier(ws)
    out.put((rank, slowest, got))
    dist.destroy_process_group()


def _split_kv_worker(rank, ws, port, out):
    import sys
    sys.path.insert(0, ROOT)
    _env(rank, ws, port)
    import torch.distributed as dist
    import bench
    from oracle import attention as A
    bench._dist(backend="gloo")
    rng = np.random.default_rng(0)            # same data on both ranks
    n, Hq, Hkv, D = 600, 8, 2, 16
    q = rng.standard_normal((Hq, D)) * 2
    k = rng.standard_normal((n, Hkv, D))
    v = rng.standard_normal((n, Hkv, D))
    # rank r owns pages [r*n/2, (r+1)*n/2) of the prefix: its partial over them
    lo, hi = rank * n // ws, (rank + 1) * n // ws
    part = A.decode(q, k[lo:hi], v[lo:hi])
    parts = [None] * ws
    dist.all_gather_object(parts, part)      # the one exchange step
    o, lse = A.combine(parts)
    o_ref, lse_ref = A.decode(q, k, v)
    out.put((rank, float(np.abs(o - o_ref).max()), float(np.abs(lse - lse_ref).max())))
    dist.destroy_process_group()


def _run(fn, ws=2):
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _port()
    procs = [ctx.Process(target=fn, args=(r, ws, port, q)) for r in range(ws)]
    for p in procs:
        p.start()
    res = [q.get(timeout=240) for _ in procs]
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    return sorted(res)


def test_replicas_are_independent_and_time_is_the_slowest_rank(stlib):
    res = _run(_replica_worker)
    assert [r[1] for r in res] == [20.0, 20.0]
    gathered = res[0][2]
    assert [g[0] for g in gathered] == [0, 1]
    assert gathered[0][1] == gathered[1][1]      # same seeds -> identical replica state
    assert all(g[2] == 20 for g in gathered)     # 4 groups x 5 branches on each rank


def test_split_prefix_partials_exchanged_and_combined():
    for rank, o_err, l_err in _run(_split_kv_worker):
        assert o_err < 1e-12 and l_err < 1e-12
