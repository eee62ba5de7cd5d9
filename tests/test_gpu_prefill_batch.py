"""Batched prefill across sequences (observation and thought rows of several
agents in one launch): every sequence's rows against the float64 oracle's
causal prefill over its own context, tables and refcounts bit-exact."""
import numpy as np
import pytest

from fg_harness import Run, compare
from oracle import attention as A
from workloads import Workload

pytestmark = pytest.mark.gpu


def _w(D, Hq, Hkv, L=2, n_blocks=2048, seed=21):
    return Workload(name=f"prefill_{D}_{Hq}_{Hkv}", n_layers=L, n_q_heads=Hq, n_kv_heads=Hkv,
                    head_dim=D, n_blocks=n_blocks, seed=seed)


def _check(run, rids, counts, q, o, lse, L0, what):
    run.pool.sync()
    run.check_tables()
    off = 0
    for r, n, l0 in zip(rids, counts, L0):
        if n:
            for layer in range(run.w.n_layers):
                k, v = run.context(r, layer)
                o_ref, l_ref = A.merge_prefill(q[layer, off:off + n].cpu(), k, v, l0)
                compare(o[layer, off:off + n], lse[layer, off:off + n], o_ref, l_ref,
                        f"{what}: seq {r} layer {layer}")
        off += n


@pytest.mark.parametrize("D,Hq,Hkv", [(128, 32, 8), (64, 8, 2), (128, 64, 8)])
def test_agents_of_different_lengths(stlib, D, Hq, Hkv):
    w = _w(D, Hq, Hkv)
    run = Run(w, max_seqs=16, max_decode_branches=16, max_splits=8)
    lens = [0, 17, 300, 2100, 16, 999]
    rids = []
    for i, n in enumerate(lens):
        r = run.create()
        if n:
            run.append([r], n, ("ctx", i))
        rids.append(r)
    counts = [37, 1, 64, 129, 0, 300]      # an agent with nothing new is left unchanged
    q, o, lse, L0 = run.prefill_batch(rids, counts, ("obs",))
    _check(run, rids, counts, q, o, lse, L0, "batch")
    # every sequence then decodes over its grown context
    live = [r for r in rids if run.ref.seqs[r].length > 0]
    q2, o2, l2 = run.decode(live, ("q",))
    o_ref, l_ref = run.oracle_decode(live, q2, 1)
    compare(o2[1], l2[1], o_ref, l_ref, "decode after the batch")


def test_siblings_of_one_fork_group(stlib):
    # the aux branches of a group each take an observation: copy-on-write of the
    # shared partial page happens in sequence order, as in separate appends
    w = _w(128, 32, 8)
    run = Run(w, max_seqs=16, max_decode_branches=16, max_splits=8)
    m = run.create()
    run.append([m], 1000, ("prefix",))            # last page holds 8 rows, shared after the fork
    aux = run.fork(m, 4)
    rids = [m] + aux
    counts = [3, 0, 16, 40, 1]
    q, o, lse, L0 = run.prefill_batch(rids, counts, ("obs",))
    _check(run, rids, counts, q, o, lse, L0, "siblings")


def test_batch_equals_one_merge_per_sequence(stlib):
    w = _w(128, 32, 8, L=1)
    runs = [Run(w, max_seqs=8, max_decode_branches=8, max_splits=8) for _ in range(2)]
    counts = [50, 7, 200]
    outs = []
    for batched, run in zip((True, False), runs):
        rids = []
        for i, n in enumerate((100, 3000, 40)):
            r = run.create()
            run.append([r], n, ("ctx", i))
            rids.append(r)
        if batched:
            q, o, lse, _ = run.prefill_batch(rids, counts, ("obs",))
            outs.append((o.cpu(), lse.cpu(), run.pool.refcounts(), run.pool.free_list()))
        else:
            # the same rows, one st_merge per sequence
            from workloads import kv_rows, queries
            k, v = kv_rows(w, ("obs",), sum(counts), device="cuda")
            q = queries(w, ("prefill_q", "obs"), sum(counts), device="cuda")
            os_, ls_ = [], []
            off = 0
            for r, n in zip(rids, counts):
                o1, l1 = run.pool.merge(run.handle[r], q[:, off:off + n].contiguous(),
                                        k[:, off:off + n].contiguous(), v[:, off:off + n].contiguous())
                os_.append(o1)
                ls_.append(l1)
                off += n
            import torch
            outs.append((torch.cat(os_, 1).cpu(), torch.cat(ls_, 1).cpu(), run.pool.refcounts(),
                         run.pool.free_list()))
    (oa, la, ra, fa), (ob, lb, rb, fb) = outs
    assert ra == rb and fa == fb
    assert np.array_equal(oa.numpy(), ob.numpy()) and np.array_equal(la.numpy(), lb.numpy())


def test_empty_and_rejected_batches(stlib):
    import paper_2608_13667_gb300 as stpkg
    w = _w(64, 8, 2, L=1, n_blocks=8)
    run = Run(w, max_seqs=4, max_decode_branches=4, max_splits=4)
    a, b = run.create(), run.create()
    run.append([a], 20, ("ctx",))
    snap = (run.pool.refcounts(), run.pool.free_list())
    q, o, lse, _ = run.prefill_batch([a, b], [0, 0], ("none",))
    assert o.shape[1] == 0 and snap == (run.pool.refcounts(), run.pool.free_list())
    # needs 0 + 7 pages, 6 are free: nothing changes
    import torch
    from workloads import kv_rows, queries
    k, v = kv_rows(w, ("big",), 120, device="cuda")
    q = queries(w, ("bq",), 120, device="cuda")
    with pytest.raises(stpkg.STError) as e:
        run.pool.prefill_batch([run.handle[a], run.handle[b]], [12, 108], q, k, v)
    assert e.value.status == stpkg.ST_ERR_OOM
    assert snap == (run.pool.refcounts(), run.pool.free_list())
    with pytest.raises(stpkg.STError):
        run.pool.prefill_batch([run.handle[a], run.handle[a]], [1, 1], q[:, :2].contiguous(),
                               k[:, :2].contiguous(), v[:, :2].contiguous())
