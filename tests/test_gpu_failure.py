"""The device-timeout path: every wait in the attention kernels is bounded.
With the ST_FLAG_HOLD_LOADS test hook nothing ever arrives on the decode's
or the merge's stage barriers; the waits run out (2 s), the kernel records
ST_ERR_TIMEOUT and returns without faulting, st_sync reports it, and the
context stays usable for a normal pool afterwards."""
import time

import pytest
import torch

import paper_2608_13667_gb300 as stpkg
from fg_harness import Run, compare
from workloads import Workload, kv_rows, queries

pytestmark = pytest.mark.gpu


def test_decode_wait_runs_out_and_is_reported(stlib):
    w = Workload(name="hold", n_layers=1, n_q_heads=8, n_kv_heads=1, head_dim=128, n_blocks=16, seed=41)
    pool = stpkg.Pool(n_layers=1, n_q_heads=8, n_kv_heads=1, head_dim=128, n_blocks=16, seed=41,
                      max_seqs=2, max_decode_branches=1, max_splits=2, flags=stpkg.ST_FLAG_HOLD_LOADS)
    a = pool.seq_create()
    k, v = kv_rows(w, ("ctx",), 20, device="cuda")
    pool.append_kv([a], k.view(1, 1, 20, 1, 128), v.view(1, 1, 20, 1, 128))
    q = queries(w, ("q",), 1, device="cuda")
    t0 = time.time()
    pool.decode_attn([a], q)                 # one CTA: its waits run out after ~2 s
    with pytest.raises(stpkg.STError) as e:
        pool.sync()
    assert e.value.status == stpkg.ST_ERR_TIMEOUT
    assert time.time() - t0 < 60
    pool.sync()                              # the status word was cleared
    pool.close()
    # the context is still usable
    run = Run(w, max_seqs=2, max_decode_branches=1, max_splits=2)
    b = run.create()
    run.append([b], 20, ("ctx2",))
    q2, o, lse = run.decode([b], ("q2",))
    run.pool.sync()
    o_ref, l_ref = run.oracle_decode([b], q2, 0)
    compare(o[0], lse[0], o_ref, l_ref, "after timeout")


@pytest.mark.parametrize("batched", [False, True])
def test_merge_wait_runs_out_and_is_reported(stlib, batched):
    w = Workload(name="holdm", n_layers=1, n_q_heads=8, n_kv_heads=2, head_dim=64, n_blocks=64, seed=43)
    pool = stpkg.Pool(n_layers=1, n_q_heads=8, n_kv_heads=2, head_dim=64, n_blocks=64, seed=43,
                      max_seqs=2, max_decode_branches=1, max_splits=2, flags=stpkg.ST_FLAG_HOLD_LOADS)
    a = pool.seq_create()
    k, v = kv_rows(w, ("ctx",), 40, device="cuda")
    pool.append_kv([a], k.view(1, 1, 40, 2, 64), v.view(1, 1, 40, 2, 64))
    km, vm = kv_rows(w, ("m",), 10, device="cuda")
    qm = queries(w, ("mq",), 10, device="cuda")
    t0 = time.time()
    if batched:
        pool.prefill_batch([a], [10], qm, km, vm)
    else:
        pool.merge(a, qm, km, vm)            # two CTAs (one per KV head): their waits run out
    with pytest.raises(stpkg.STError) as e:
        pool.sync()
    assert e.value.status == stpkg.ST_ERR_TIMEOUT
    assert time.time() - t0 < 60
    pool.sync()
    pool.close()
    run = Run(w, max_seqs=2, max_decode_branches=1, max_splits=2)
    b = run.create()
    run.append([b], 40, ("ctx2",))
    qm2, om, lm, L0 = run.merge(b, 10, ("m2",))
    run.pool.sync()
    from oracle import attention as A
    kk, vv = run.context(b, 0)
    o_ref, l_ref = A.merge_prefill(qm2[0].cpu(), kk, vv, L0)
    compare(om[0], lm[0], o_ref, l_ref, "merge after timeout")


def test_decode_step_stores_its_row_even_when_the_waits_run_out(stlib):
    """st_decode_step leaves each new row to the decode kernel that reads its
    page; that kernel stores the row before any wait, so a decode whose waits
    run out (ST_FLAG_HOLD_LOADS) still leaves the pool holding what the host
    tables say it holds."""
    w = Workload(name="hold_step", n_layers=2, n_q_heads=8, n_kv_heads=2, head_dim=128, n_blocks=32, seed=45)
    pool = stpkg.Pool(n_layers=2, n_q_heads=8, n_kv_heads=2, head_dim=128, n_blocks=32, seed=45,
                      max_seqs=4, max_decode_branches=2, max_splits=4, flags=stpkg.ST_FLAG_HOLD_LOADS)
    a, b = pool.seq_create(), pool.seq_create()
    k, v = kv_rows(w, ("ctx",), 20, device="cuda")
    pool.append_kv([a, b], k.view(2, 2, 10, 2, 128), v.view(2, 2, 10, 2, 128))
    kn, vn = kv_rows(w, ("new",), 2, device="cuda")            # [L][2 branches][Hkv][D]
    pool.decode_step([a, b], kn, vn, queries(w, ("q",), 2, device="cuda"))
    with pytest.raises(stpkg.STError) as e:
        pool.sync()
    assert e.value.status == stpkg.ST_ERR_TIMEOUT
    for i, h in enumerate((a, b)):
        table, n = pool.block_table(h)
        assert n == 11
        page, row = table[(n - 1) // 16], (n - 1) % 16
        assert torch.equal(pool.k_pool[:, page, :, row], kn[:, i])
        assert torch.equal(pool.v_pool[:, page, :, row], vn[:, i])
    pool.close()
