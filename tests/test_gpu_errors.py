"""Error paths and limits on a GPU pool: rejected calls change nothing and
leave the pool usable; the smallest split budget and pool exhaustion in the
middle of a decode loop still give oracle-exact results."""
import pytest
import torch

import paper_2608_13667_gb300 as stpkg
from fg_harness import Run, compare
from workloads import Workload, queries

pytestmark = pytest.mark.gpu


def _w(n_blocks=64, L=1):
    return Workload(name="err", n_layers=L, n_q_heads=8, n_kv_heads=2, head_dim=64, n_blocks=n_blocks, seed=51)


def _snap(run):
    return (run.pool.refcounts(), run.pool.free_list(),
            {r: run.pool.block_table(run.handle[r]) for r in run.ref.live()})


def test_rejected_decode_calls_change_nothing(stlib):
    w = _w()
    run = Run(w, max_seqs=8, max_decode_branches=3, max_splits=4)
    m = run.create()
    run.append([m], 50, ("ctx",))
    aux = run.fork(m, 3)
    empty = run.create()
    snap = _snap(run)
    q = queries(w, ("q",), 4, device="cuda")
    cases = [
        ([m] + aux, q, stpkg.ST_ERR_INVALID),                                   # 4 > max_decode_branches
        ([m, m], queries(w, ("q2",), 2, device="cuda"), stpkg.ST_ERR_INVALID),  # listed twice
        ([empty], queries(w, ("q3",), 1, device="cuda"), stpkg.ST_ERR_INVALID),  # empty sequence
    ]
    for br, qq, status in cases:
        with pytest.raises(stpkg.STError) as e:
            run.pool.decode_attn([run.handle[r] for r in br], qq)
        assert e.value.status == status
    stale = run.handle[aux[2]]
    run.release(aux[2])
    with pytest.raises(stpkg.STError) as e:
        run.pool.decode_attn([stale], queries(w, ("q4",), 1, device="cuda"))
    assert e.value.status == stpkg.ST_ERR_INVALID
    snap2 = _snap(run)
    assert snap2[0] != snap[0]  # only the release changed the pool
    # still correct afterwards
    q5, o, lse = run.decode([m] + aux[:2], ("q5",))
    run.pool.sync()
    o_ref, l_ref = run.oracle_decode([m] + aux[:2], q5, 0)
    compare(o[0], lse[0], o_ref, l_ref, "after rejected calls")


def test_smallest_split_budget(stlib):
    w = _w(n_blocks=512, L=2)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=2)
    m = run.create()
    run.append([m], 5000, ("ctx",))
    br = [m] + run.fork(m, 4)
    for b, r in enumerate(br):
        run.append([r], 3 * b + 1, ("s", b))
    q, o, lse = run.decode(br, ("q",))
    for layer in range(2):
        o_ref, l_ref = run.oracle_decode(br, q, layer)
        compare(o[layer], lse[layer], o_ref, l_ref, f"max_splits=2 layer {layer}")


def test_pool_exhaustion_mid_decode_loop(stlib):
    w = _w(n_blocks=40)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=4)
    m = run.create()
    run.append([m], 30 * 16 - 3, ("ctx",))           # 30 pages, the last one partial
    br = [m] + run.fork(m, 4)
    step, failed = 0, False
    while not failed and step < 64:
        before = _snap(run)
        try:
            run.append(br, 1, ("step", step))
        except stpkg.STError as e:
            assert e.status == stpkg.ST_ERR_OOM
            assert _snap(run) == before
            failed = True
            break
        q, o, lse = run.decode(br, ("q", step))
        step += 1
    assert failed
    # the last successful step's state still decodes correctly
    q, o, lse = run.decode(br, ("q_after",))
    run.pool.sync()
    o_ref, l_ref = run.oracle_decode(br, q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "after exhaustion")
    run.check_tables()


def test_failed_launch_after_append_makes_the_pool_unusable(stlib):
    # ST_FLAG_FAIL_LAUNCH reports every launch as failed without making it (a
    # fake of a failing CUDA launch): the append has already changed the host
    # tables when its launch fails, so the pool refuses every later call.
    pool = stpkg.Pool(n_layers=1, n_q_heads=8, n_kv_heads=2, head_dim=64, n_blocks=32, seed=3,
                      max_seqs=4, device="cuda", flags=stpkg.ST_FLAG_FAIL_LAUNCH)
    m = pool.seq_create()
    kv = torch.zeros((1, 1, 20, 2, 64), dtype=torch.bfloat16, device="cuda")
    with pytest.raises(stpkg.STError) as e:
        pool.append_kv([m], kv, kv)
    assert e.value.status == stpkg.ST_ERR_CUDA
    for call in (lambda: pool.append_kv([m], kv, kv), lambda: pool.fork(m, 2), pool.seq_create,
                 lambda: pool.release(m), pool.sync,
                 lambda: pool.decode_attn([m], torch.zeros((1, 1, 8, 64), dtype=torch.bfloat16, device="cuda"))):
        with pytest.raises(stpkg.STError) as e:
            call()
        assert e.value.status == stpkg.ST_ERR_STATE
        assert "unusable" in str(e.value)
    # introspection still reports the host's view: the 20 rows went in
    assert pool.block_table(m)[1] == 20
    pool.close()
    # a pool without the flag on the same device is unaffected
    run = Run(_w(), max_seqs=4, max_decode_branches=2, max_splits=4)
    a = run.create()
    run.append([a], 21, ("ctx",))
    q, o, lse = run.decode([a], ("q",))
    run.pool.sync()
    o_ref, l_ref = run.oracle_decode([a], q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "after a broken pool")
