"""The allocation-free decode entry point (st_decode_attn_noalloc) against the
pool's st_decode_attn on the same KV, on two calls in a row.

That entry point serves callers that cannot allocate device memory (a host
framework that owns all device allocations, a real-time loop that must not
allocate, a plugin handed only input/output pointers): its scratch is a
static device array instead of a caller-provided workspace.  This file is
collected last so that a failure here comes after every other test."""
import pytest
import torch

import paper_2608_13667_gb300 as stpkg
from fg_harness import Run, compare
from workloads import Workload, queries

pytestmark = pytest.mark.gpu


def _noalloc(run, rids, q):
    w = run.w
    tables, lens = [], []
    for r in rids:
        t, n = run.pool.block_table(run.handle[r])
        tables.append(t)
        lens.append(n)
    o = torch.empty((w.n_layers, len(rids), w.n_q_heads, w.head_dim), dtype=torch.float32, device="cuda")
    lse = torch.empty((w.n_layers, len(rids), w.n_q_heads), dtype=torch.float32, device="cuda")
    st = stpkg.st_decode_attn_noalloc(run.pool.cfg, run.pool.k_pool, run.pool.v_pool, tables, lens, q, o, lse)
    assert st == stpkg.ST_OK, stpkg.lib().st_status_str(st)
    return o, lse


def test_noalloc_decode_matches_pool_decode_twice(stlib):
    w = Workload(name="noalloc", n_layers=2, n_q_heads=32, n_kv_heads=8, head_dim=128,
                 n_blocks=1024, seed=21)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=16)
    m = run.create()
    run.append([m], 4100, ("prefix",))
    rids = [m] + run.fork(m, 4)
    for b, r in enumerate(rids):
        run.append([r], 3 + 11 * b, ("suffix", b))
    for call in range(2):
        run.append(rids, 1, ("step", call))
        q = queries(w, ("q", call), len(rids), device="cuda")
        o_ref, lse_ref = run.pool.decode_attn([run.handle[r] for r in rids], q)
        o, lse = _noalloc(run, rids, q)
        torch.cuda.synchronize()
        for layer in range(w.n_layers):
            compare(o[layer], lse[layer], o_ref[layer].double().cpu().numpy(),
                    lse_ref[layer].double().cpu().numpy(), f"call {call} layer {layer}")


def test_noalloc_rejects_what_does_not_fit(stlib):
    w = Workload(name="noalloc_big", n_layers=32, n_q_heads=64, n_kv_heads=8, head_dim=128,
                 n_blocks=64, seed=22)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=16)
    m = run.create()
    run.append([m], 40, ("ctx",))
    rids = [m] + run.fork(m, 4)
    q = queries(w, ("q",), len(rids), device="cuda")
    o = torch.empty((w.n_layers, 5, w.n_q_heads, w.head_dim), dtype=torch.float32, device="cuda")
    lse = torch.empty((w.n_layers, 5, w.n_q_heads), dtype=torch.float32, device="cuda")
    tables = [run.pool.block_table(run.handle[r])[0] for r in rids]
    # 32 layers x 5 branches x 64 heads x 16 slots x 129 floats > 16 MiB
    st = stpkg.st_decode_attn_noalloc(run.pool.cfg, run.pool.k_pool, run.pool.v_pool, tables, [40] * 5, q, o, lse)
    assert st == stpkg.ST_ERR_OOM
    st = stpkg.st_decode_attn_noalloc(run.pool.cfg, run.pool.k_pool, run.pool.v_pool, tables, [0] * 5, q, o, lse)
    assert st == stpkg.ST_ERR_INVALID
