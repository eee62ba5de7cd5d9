"""The allocation-free decode entry point (st_decode_attn_noalloc): against the
pool's st_decode_attn on the same KV on two calls in a row, and against the
float64 oracle on the branch layouts its own planner has to handle.

That entry point serves callers that cannot allocate device memory (a host
framework that owns all device allocations, a real-time loop that must not
allocate, a plugin handed only input/output pointers): its scratch is a
static device array instead of a caller-provided workspace, and its
device-side outcome goes to a status word the caller owns.  This file is
collected last so that a failure here comes after every other test."""
import pytest
import torch

import paper_2608_13667_gb300 as stpkg
from fg_harness import Run, compare
from workloads import Workload, queries

pytestmark = pytest.mark.gpu


def _noalloc(run, rids, q, geom=None):
    w = run.w
    tables, lens = [], []
    for r in rids:
        t, n = run.pool.block_table(run.handle[r])
        tables.append(t)
        lens.append(n)
    o = torch.empty((w.n_layers, len(rids), w.n_q_heads, w.head_dim), dtype=torch.float32, device="cuda")
    lse = torch.empty((w.n_layers, len(rids), w.n_q_heads), dtype=torch.float32, device="cuda")
    st, status = stpkg.st_decode_attn_noalloc(geom or run.pool.cfg, run.pool.k_pool, run.pool.v_pool, tables,
                                              lens, q, o, lse)
    assert st == stpkg.ST_OK, stpkg.lib().st_status_str(st)
    return o, lse, status


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
        o, lse, status = _noalloc(run, rids, q)
        torch.cuda.synchronize()
        assert int(status.item()) == stpkg.ST_OK
        for layer in range(w.n_layers):
            compare(o[layer], lse[layer], o_ref[layer].double().cpu().numpy(),
                    lse_ref[layer].double().cpu().numpy(), f"call {call} layer {layer}")


def _two_groups_and_loners():
    """Two independent fork groups, a lone sequence shorter than a page, a
    lone long one, and a pair whose tables share their first pages and then
    diverge (a fork from an earlier point), listed interleaved."""
    w = Workload(name="noalloc_mix", n_layers=2, n_q_heads=32, n_kv_heads=8, head_dim=128,
                 n_blocks=2048, seed=23)
    run = Run(w, max_seqs=24, max_decode_branches=16, max_splits=16)
    m1 = run.create()
    run.append([m1], 4100, ("p1",))
    g1 = run.fork(m1, 4)
    m2 = run.create()
    run.append([m2], 2000, ("p2",))
    g2 = run.fork(m2, 2)
    for i, r in enumerate(g1 + g2):
        run.append([r], 5 + 17 * i, ("s", i))
    short = run.create()
    run.append([short], 10, ("short",))
    long_ = run.create()
    run.append([long_], 700, ("long",))
    m3 = run.create()
    run.append([m3], 100, ("p3",))
    (c3,) = run.fork_at(m3, 60, 1)
    run.append([c3], 9, ("c3",))
    run.append([m3], 40, ("m3",))
    rids = [m1, m2, short, g1[0], m3, g2[0], c3, g1[1], long_, g1[2], g2[1], g1[3]]
    t_m3, t_c3 = run.pool.block_table(run.handle[m3])[0], run.pool.block_table(run.handle[c3])[0]
    assert t_m3[:3] == t_c3[:3] and t_m3[3] != t_c3[3]
    return run, rids


def _family_split():
    """G = 8: a family of 9 branches exceeds 64 / G = 8 per group and is
    split (a group of 8, and one branch that reads its pages on its own);
    one more sequence is shorter than a page."""
    w = Workload(name="noalloc_split", n_layers=2, n_q_heads=64, n_kv_heads=8, head_dim=128,
                 n_blocks=1024, seed=24)
    run = Run(w, max_seqs=16, max_decode_branches=16, max_splits=16)
    m = run.create()
    run.append([m], 3000, ("p",))
    br = [m] + run.fork(m, 8)
    for i, r in enumerate(br):
        run.append([r], 1 + 7 * i, ("s", i))
    tiny = run.create()
    run.append([tiny], 5, ("tiny",))
    return run, br + [tiny]


def _head_dim_64():
    w = Workload(name="noalloc_d64", n_layers=3, n_q_heads=8, n_kv_heads=2, head_dim=64,
                 n_blocks=512, seed=25)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=16)
    m = run.create()
    run.append([m], 1500, ("p",))
    br = [m] + run.fork(m, 4)
    for i, r in enumerate(br[1:], 1):
        run.append([r], 2 * i, ("s", i))
    lone = run.create()
    run.append([lone], 333, ("lone",))
    return run, br + [lone]


@pytest.mark.parametrize("make", [_two_groups_and_loners, _family_split, _head_dim_64],
                         ids=["two_groups_and_loners", "family_split_G8", "head_dim_64"])
def test_noalloc_matches_oracle_twice(stlib, make):
    run, rids = make()
    w = run.w
    for call in range(2):
        run.append(rids, 1, ("step", call))
        q = queries(w, ("q", call), len(rids), device="cuda")
        o, lse, status = _noalloc(run, rids, q)
        torch.cuda.synchronize()
        assert int(status.item()) == stpkg.ST_OK
        for layer in range(w.n_layers):
            o_ref, l_ref = run.oracle_decode(rids, q, layer)
            compare(o[layer], lse[layer], o_ref, l_ref, f"{w.name} call {call} layer {layer}")


def test_noalloc_reports_a_device_timeout_in_the_status_word(stlib):
    # ST_FLAG_HOLD_LOADS: the decode's loader issues no copies, its bounded
    # waits (2 s) run out, and the kernel records ST_ERR_TIMEOUT and returns.
    run, rids = _head_dim_64()
    w = run.w
    q = queries(w, ("q",), len(rids), device="cuda")
    geom = stpkg.StConfig.from_buffer_copy(run.pool.cfg)
    geom.flags = stpkg.ST_FLAG_HOLD_LOADS
    _, _, status = _noalloc(run, rids, q, geom)
    torch.cuda.synchronize()
    assert int(status.item()) == stpkg.ST_ERR_TIMEOUT
    # the next call clears the word and computes normally on the same context
    o, lse, status = _noalloc(run, rids, q)
    torch.cuda.synchronize()
    assert int(status.item()) == stpkg.ST_OK
    o_ref, l_ref = run.oracle_decode(rids, q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "after a timed-out call")


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
    args = (run.pool.cfg, run.pool.k_pool, run.pool.v_pool)
    # 32 layers x 5 branches x 64 heads x 16 slots x 129 floats > 16 MiB
    assert stpkg.st_decode_attn_noalloc(*args, tables, [40] * 5, q, o, lse)[0] == stpkg.ST_ERR_OOM
    assert stpkg.st_decode_attn_noalloc(*args, tables, [0] * 5, q, o, lse)[0] == stpkg.ST_ERR_INVALID
    bad = [list(t) for t in tables]
    bad[2][1] = w.n_blocks                      # a page id past the pool: refused on the host
    assert stpkg.st_decode_attn_noalloc(*args, bad, [40] * 5, q, o, lse)[0] == stpkg.ST_ERR_INVALID
