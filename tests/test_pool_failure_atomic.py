"""A call that the library rejects after its capacity checks leaves the pool
as it was.  Plans too large for one staging slot are refused before any
table changes (metadata-only pools run the same host code as GPU pools)."""
import pytest

from oracle import pool as R


def _meta(stlib, n_blocks, max_seqs, **kw):
    return stlib.Pool(n_layers=1, n_q_heads=4, n_kv_heads=2, head_dim=64, n_blocks=n_blocks, seed=7,
                      max_seqs=max_seqs, max_pages=kw.pop("max_pages", n_blocks), device=None, **kw)


def _state(pool, handles):
    return pool.refcounts(), pool.free_list(), [pool.block_table(h) for h in handles]


def test_oversized_append_plan_changes_nothing(stlib):
    # 65538 sequences, each holding the same partial page: an append of one
    # row to all of them may copy that page for every one, so its plan (one
    # 16-byte record per sequence plus one per copy) would need 2 MiB + 64 B,
    # more than one staging slot.  The call is refused before any change.
    n = 65538
    lp = _meta(stlib, n_blocks=70000, max_seqs=n)
    main = lp.seq_create()
    lp.append_kv([main], 5, None)
    kids = lp.fork(main, n - 1)
    handles = [main] + kids
    before = _state(lp, handles)
    with pytest.raises(stlib.STError) as e:
        lp.append_kv(handles, 1, None)
    assert e.value.status == stlib.ST_ERR_INVALID
    assert "plan" in str(e.value)
    assert _state(lp, handles) == before
    # a call that fits still goes through, bit-exact with the oracle
    ref = R.RefPool(70000, 7)
    m = ref.create()
    ref.append([m], 5)
    rk = ref.fork(m, n - 1)
    ids = [m] + rk[:999]
    ref.append(ids, 1)
    lp.append_kv(handles[:1000], 1, None)
    assert lp.refcounts() == ref.ref
    assert lp.free_list() == list(ref.free)
    for i in (0, 1, 500, 999):
        assert lp.block_table(handles[i])[0] == ref.seqs[ids[i]].table


def test_oversized_prefill_plan_changes_nothing(stlib):
    # G = 2: one work item per 128 rows; 65537 items of 32 bytes exceed a slot
    rows = 65537 * 128
    lp = _meta(stlib, n_blocks=rows // 16 + 64, max_seqs=4)
    a, b = lp.seq_create(), lp.seq_create()
    lp.append_kv([a], 3, None)
    before = _state(lp, [a, b])
    with pytest.raises(stlib.STError) as e:
        lp.prefill_batch([a, b], [1, rows], None, None, None)
    assert e.value.status == stlib.ST_ERR_INVALID
    assert _state(lp, [a, b]) == before
    lp.prefill_batch([a, b], [0, rows - 128], None, None, None)  # 65536 items fill a slot exactly
    assert lp.block_table(b)[1] == rows - 128 and lp.block_table(a)[1] == 3


def test_ragged_prefill_out_of_pages_changes_nothing(stlib):
    lp = _meta(stlib, n_blocks=10, max_seqs=4)
    ref = R.RefPool(10, 7)
    hs = [lp.seq_create() for _ in range(3)]
    rs = [ref.create() for _ in range(3)]
    lp.prefill_batch(hs, [5, 17, 0], None, None, None)
    ref.prefill_batch(rs, [5, 17, 0])
    before = _state(lp, hs)
    # needs 1 + 1 + 6 = 8 pages, 7 are free
    with pytest.raises(stlib.STError) as e:
        lp.prefill_batch(hs, [12, 20, 96], None, None, None)
    assert e.value.status == stlib.ST_ERR_OOM
    with pytest.raises(R.OutOfBlocks):
        ref.prefill_batch(rs, [12, 20, 96])
    assert _state(lp, hs) == before
    assert lp.refcounts() == ref.ref and lp.free_list() == list(ref.free)
    # 1 + 1 + 5 = 7 pages: exactly what is left
    lp.prefill_batch(hs, [12, 20, 80], None, None, None)
    ref.prefill_batch(rs, [12, 20, 80])
    assert lp.free_list() == list(ref.free) == []
    assert [lp.block_table(h)[0] for h in hs] == [ref.seqs[r].table for r in rs]


def test_decode_calls_on_a_metadata_pool_change_nothing(stlib):
    """A metadata-only pool has no KV storage: the attention calls, and the
    decode step that would append before its decode, are refused with
    ST_ERR_STATE and leave the tables as they were."""
    import ctypes
    lp = _meta(stlib, n_blocks=16, max_seqs=4)
    a = lp.seq_create()
    lp.append_kv([a], 5, None)
    before = _state(lp, [a])
    L = stlib.lib()
    arr = (ctypes.c_int64 * 1)(a)
    assert L.st_decode_step(lp._h, arr, 1, None, None, None, None, None, None) == stlib.ST_ERR_STATE
    assert L.st_decode_attn(lp._h, arr, 1, None, None, None, None) == stlib.ST_ERR_STATE
    assert _state(lp, [a]) == before
