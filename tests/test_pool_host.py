"""The library's host allocator (a metadata-only pool: same code path as a
GPU pool, no device work) against the reference pool, bit-exactly: tables,
refcounts and free-list order after every operation of random traces."""
import random

import pytest

from oracle import pool as R


def _meta(stlib, n_blocks, seed, max_seqs=64, max_pages=None):
    return stlib.Pool(n_layers=1, n_q_heads=4, n_kv_heads=2, head_dim=64, n_blocks=n_blocks,
                      seed=seed, max_seqs=max_seqs, max_pages=max_pages or n_blocks, device=None)


def _same(lib_pool, ref, handles):
    assert lib_pool.refcounts() == ref.ref
    assert lib_pool.free_list() == list(ref.free)
    for rid, h in handles.items():
        if ref.seqs[rid].alive:
            table, n = lib_pool.block_table(h)
            assert table == ref.seqs[rid].table and n == ref.seqs[rid].length


@pytest.mark.parametrize("seed", range(12))
def test_random_traces_match_reference_bit_exactly(stlib, seed):
    r = random.Random(seed)
    n_blocks = r.choice([32, 64, 200])
    max_seqs = r.choice([4, 8, 16])
    lp = _meta(stlib, n_blocks, seed, max_seqs=max_seqs)
    ref = R.RefPool(n_blocks, seed, max_seqs=max_seqs)
    handles = {}
    rid = ref.create()
    handles[rid] = lp.seq_create()
    for _ in range(150):
        live = ref.live()
        op = r.random()
        if op < 0.5 and live:
            ids = r.sample(live, r.randint(1, min(5, len(live))))
            n = r.choice([1, 1, 1, 3, 15, 16, 17, 40])
            try:
                ref.append(ids, n)
                ok = True
            except R.OutOfBlocks:
                ok = False
            if ok:
                lp.append_kv([handles[i] for i in ids], n, None)
            else:
                with pytest.raises(stlib.STError) as e:
                    lp.append_kv([handles[i] for i in ids], n, None)
                assert e.value.status == stlib.ST_ERR_OOM
        elif op < 0.65 and live:
            parent = r.choice(live)
            n_aux = r.randint(1, 4)
            at = r.random() < 0.4
            cut = r.randint(0, ref.seqs[parent].length)
            try:
                kids = ref.fork_at(parent, cut, n_aux) if at else ref.fork(parent, n_aux)
            except R.OutOfSlots:
                with pytest.raises(stlib.STError) as e:
                    lp.fork_at(handles[parent], cut, n_aux) if at else lp.fork(handles[parent], n_aux)
                assert e.value.status == stlib.ST_ERR_OOM
            else:
                new = lp.fork_at(handles[parent], cut, n_aux) if at else lp.fork(handles[parent], n_aux)
                for k, h in zip(kids, new):
                    handles[k] = h
        elif op < 0.75 and live:
            m = r.choice(live)
            T = r.choice([0, 1, 7, 33])
            try:
                ref.merge(m, T)
                ok = True
            except R.OutOfBlocks:
                ok = False
            if ok:
                lp.merge(handles[m], T, None, None)
            else:
                with pytest.raises(stlib.STError):
                    lp.merge(handles[m], T, None, None)
        elif op < 0.82 and live:
            # batched prefill: ragged counts (zeros included), sequences in order
            ids = r.sample(live, r.randint(1, min(5, len(live))))
            counts = [r.choice([0, 1, 5, 16, 17, 40]) for _ in ids]
            try:
                ref.prefill_batch(ids, counts)
                ok = True
            except R.OutOfBlocks:
                ok = False
            if ok:
                lp.prefill_batch([handles[i] for i in ids], counts, None, None, None)
            else:
                with pytest.raises(stlib.STError) as e:
                    lp.prefill_batch([handles[i] for i in ids], counts, None, None, None)
                assert e.value.status == stlib.ST_ERR_OOM
        elif op < 0.9 and len(live) > 1:
            x = r.choice(live)
            ref.release(x)
            lp.release(handles[x])
        elif len(live) < max_seqs:
            rid = ref.create()
            handles[rid] = lp.seq_create()
        _same(lp, ref, handles)


def test_cycle_shaped_trace(stlib):
    # fork 4 -> 64 steps of 1 row on all 5 -> merge 256 -> release 4, three turns,
    # with a prefix that ends mid-page so every branch copies the shared page.
    lp = _meta(stlib, 2048, 7)
    ref = R.RefPool(2048, 7)
    m_r, m_h = ref.create(), lp.seq_create()
    ref.append([m_r], 1000)
    lp.append_kv([m_h], 1000, None)
    for turn in range(3):
        aux_r = ref.fork(m_r, 4)
        aux_h = lp.fork(m_h, 4)
        for step in range(64):
            ref.append([m_r] + aux_r, 1)
            lp.append_kv([m_h] + aux_h, 1, None)
        ref.merge(m_r, 256)
        lp.merge(m_h, 256, None, None)
        for a, h in zip(aux_r, aux_h):
            ref.release(a)
            lp.release(h)
        _same(lp, ref, {m_r: m_h})


def test_handles_go_stale_after_release(stlib):
    lp = _meta(stlib, 16, 0)
    a = lp.seq_create()
    lp.append_kv([a], 5, None)
    lp.release(a)
    for call in (lambda: lp.release(a), lambda: lp.append_kv([a], 1, None),
                 lambda: lp.fork(a, 1), lambda: lp.block_table(a)):
        with pytest.raises(stlib.STError) as e:
            call()
        assert e.value.status == stlib.ST_ERR_INVALID
    b = lp.seq_create()          # reuses the slot with a new generation
    assert b != a and (b & 0xffffffff) == (a & 0xffffffff)


def test_duplicate_branch_in_one_call_is_rejected(stlib):
    lp = _meta(stlib, 16, 0)
    a = lp.seq_create()
    with pytest.raises(stlib.STError) as e:
        lp.append_kv([a, a], 1, None)
    assert e.value.status == stlib.ST_ERR_INVALID
    assert lp.block_table(a) == ([], 0)


def test_oom_changes_nothing(stlib):
    lp = _meta(stlib, 4, 1, max_seqs=3)
    a, b = lp.seq_create(), lp.seq_create()
    lp.append_kv([a], 40, None)
    snap = (lp.refcounts(), lp.free_list(), lp.block_table(a), lp.block_table(b))
    with pytest.raises(stlib.STError) as e:
        lp.append_kv([b, a], 16, None)
    assert e.value.status == stlib.ST_ERR_OOM
    with pytest.raises(stlib.STError) as e:
        lp.fork(a, 2)             # one slot left
    assert e.value.status == stlib.ST_ERR_OOM
    with pytest.raises(stlib.STError) as e:
        lp.merge(a, 100, None, None)
    assert e.value.status == stlib.ST_ERR_OOM
    assert snap == (lp.refcounts(), lp.free_list(), lp.block_table(a), lp.block_table(b))


def test_max_pages_is_enforced(stlib):
    lp = _meta(stlib, 64, 0, max_pages=4)
    a = lp.seq_create()
    lp.append_kv([a], 64, None)
    with pytest.raises(stlib.STError) as e:
        lp.append_kv([a], 1, None)
    assert e.value.status == stlib.ST_ERR_OOM


def test_merge_of_nothing_is_a_noop(stlib):
    lp = _meta(stlib, 16, 0)
    a = lp.seq_create()
    lp.append_kv([a], 20, None)
    snap = (lp.refcounts(), lp.free_list(), lp.block_table(a))
    lp.merge(a, 0, None, None)
    assert snap == (lp.refcounts(), lp.free_list(), lp.block_table(a))


def test_fork_then_release_is_identity(stlib):
    lp = _meta(stlib, 64, 3)
    a = lp.seq_create()
    lp.append_kv([a], 37, None)
    snap = (lp.refcounts(), lp.free_list())
    kids = lp.fork(a, 4)
    assert all(lp.refcounts()[b] == 5 for b in lp.block_table(a)[0])
    for k in kids:
        lp.release(k)
    assert snap == (lp.refcounts(), lp.free_list())


def test_metadata_pool_refuses_attention(stlib):
    import torch
    lp = _meta(stlib, 16, 0)
    a = lp.seq_create()
    lp.append_kv([a], 3, None)
    L = stlib.lib()
    import ctypes
    arr = (ctypes.c_int64 * 1)(a)
    st = L.st_decode_attn(lp._h, arr, 1, ctypes.c_void_p(16), ctypes.c_void_p(16), ctypes.c_void_p(16), None)
    assert st == stlib.ST_ERR_STATE


def test_fork_at_rejects_points_past_the_end(stlib):
    lp = _meta(stlib, 16, 0)
    a = lp.seq_create()
    lp.append_kv([a], 20, None)
    for bad in (-1, 21):
        with pytest.raises(stlib.STError) as e:
            lp.fork_at(a, bad, 1)
        assert e.value.status == stlib.ST_ERR_INVALID
    (c,) = lp.fork_at(a, 0, 1)
    assert lp.block_table(c) == ([], 0)
