"""Pins for the reference block pool: the published generator values, the
shuffle computed by hand from them, and invariants that a wrong refcount,
a missing copy-on-write or a wrong free order would break."""
import random

import pytest

from oracle import pool as P
from conftest import read_golden

MASK = (1 << 64) - 1


def test_splitmix64_published_values():
    want = [int(x[0], 16) for x in read_golden("splitmix64_seed0.txt")]
    gen = P.splitmix64(0)
    assert [next(gen) for _ in want] == want


def test_free_list_shuffle_by_hand():
    # Fisher-Yates on [0,1,2] with the published seed-0 outputs x1, x2:
    # i=2 swaps with x1 % 3, then i=1 swaps with x2 % 2.
    x1, x2, _ = [int(x[0], 16) for x in read_golden("splitmix64_seed0.txt")]
    a = [0, 1, 2]
    j = x1 % 3
    a[2], a[j] = a[j], a[2]
    j = x2 % 2
    a[1], a[j] = a[j], a[1]
    assert P.initial_free_list(3, 0) == a


@pytest.mark.parametrize("n,seed", [(1, 0), (2, 5), (64, 0), (1000, 123)])
def test_free_list_is_a_permutation(n, seed):
    fl = P.initial_free_list(n, seed)
    assert sorted(fl) == list(range(n))


def _check_invariants(pool):
    live = pool.live()
    # every reference is held by exactly one table entry of a live sequence
    counts = [0] * pool.n_blocks
    for i in live:
        s = pool.seqs[i]
        assert len(s.table) == -(-s.length // pool.page)
        for b in s.table:
            counts[b] += 1
    assert counts == pool.ref
    # conservation: free pages are exactly the unreferenced ones, each once
    assert len(set(pool.free)) == len(pool.free)
    assert sorted(pool.free) == [b for b in range(pool.n_blocks) if pool.ref[b] == 0]
    assert len(pool.free) + sum(1 for r in pool.ref if r > 0) == pool.n_blocks


def test_random_operation_sequences_keep_invariants_and_content():
    r = random.Random(42)
    for trial in range(30):
        pool = P.RefPool(n_blocks=r.choice([24, 48, 96]), seed=trial, track_content=True)
        history = {}   # seq -> list of labels it must read back
        m = pool.create()
        history[m] = []
        for step in range(60):
            live = pool.live()
            op = r.random()
            try:
                if op < 0.45 and live:
                    ids = r.sample(live, r.randint(1, min(3, len(live))))
                    n = r.choice([0, 1, 1, 2, 5, 16, 17, 33])
                    labels = [[(i, len(history[i]) + t, trial) for t in range(n)] for i in ids]
                    pool.append(ids, n, labels)
                    for i, lab in zip(ids, labels):
                        history[i] += lab
                elif op < 0.58 and live:
                    parent = r.choice(live)
                    for c in pool.fork(parent, r.randint(1, 4)):
                        history[c] = list(history[parent])
                elif op < 0.65 and live:
                    parent = r.choice(live)
                    cut = r.randint(0, pool.seqs[parent].length)
                    for c in pool.fork_at(parent, cut, r.randint(1, 3)):
                        history[c] = list(history[parent][:cut])
                elif op < 0.85 and len(live) > 1:
                    pool.release(r.choice(live))
                else:
                    c = pool.create()
                    history[c] = []
            except P.OutOfBlocks:
                pass
            _check_invariants(pool)
            for i in pool.live():
                assert pool.read(i) == history[i]


def test_fork_then_release_restores_refcounts_and_free_list():
    pool = P.RefPool(n_blocks=64, seed=3)
    m = pool.create()
    pool.append([m], 40)
    before = (list(pool.ref), list(pool.free))
    aux = pool.fork(m, 4)
    assert all(pool.ref[b] == 5 for b in pool.seqs[m].table)
    for a in aux:
        pool.release(a)
    assert (list(pool.ref), list(pool.free)) == before


def test_copy_on_write_first_appender_copies_last_holder_writes_in_place():
    pool = P.RefPool(n_blocks=32, seed=1)
    m = pool.create()
    pool.append([m], 20)              # pages: one full, one with 4 rows
    partial = pool.seqs[m].table[1]
    aux = pool.fork(m, 2)
    ev = pool.append([aux[0]], 1)     # shared partial page -> copy 4 rows
    assert len(ev) == 1 and ev[0][0] == partial and ev[0][2] == 4
    ev = pool.append([m], 1)          # still shared by m and aux[1] -> copy
    assert len(ev) == 1 and ev[0][0] == partial
    assert pool.ref[partial] == 1     # only aux[1] holds it now
    ev = pool.append([aux[1]], 1)     # last holder writes in place
    assert ev == [] and pool.seqs[aux[1]].table[1] == partial
    # the full first page is never copied
    assert pool.seqs[aux[0]].table[0] == pool.seqs[m].table[0] == pool.seqs[aux[1]].table[0]


def test_append_at_page_boundary_allocates_without_copy():
    pool = P.RefPool(n_blocks=16, seed=2)
    m = pool.create()
    pool.append([m], 32)
    aux = pool.fork(m, 1)
    free_before = len(pool.free)
    assert pool.append(aux, 1) == []
    assert len(pool.free) == free_before - 1
    assert pool.seqs[aux[0]].table[:2] == pool.seqs[m].table


def test_allocation_follows_the_fifo_and_release_refills_its_tail():
    pool = P.RefPool(n_blocks=8, seed=9)
    order = P.initial_free_list(8, 9)
    a = pool.create()
    pool.append([a], 48)                       # three pages: the FIFO head
    assert pool.seqs[a].table == order[:3]
    pool.release(a)
    assert list(pool.free) == order[3:] + order[:3]


def test_out_of_blocks_changes_nothing():
    pool = P.RefPool(n_blocks=4, seed=0)
    a = pool.create()
    b = pool.create()
    pool.append([a], 40)                       # 3 pages
    snap = (list(pool.ref), list(pool.free), list(pool.seqs[a].table), pool.seqs[a].length)
    with pytest.raises(P.OutOfBlocks):
        pool.append([b, a], 16)                # needs 1 + 1 > 1 free
    assert snap == (list(pool.ref), list(pool.free), list(pool.seqs[a].table), pool.seqs[a].length)
    assert pool.seqs[b].length == 0


def test_out_of_slots_changes_nothing():
    pool = P.RefPool(n_blocks=8, seed=0, max_seqs=3)
    a = pool.create()
    pool.append([a], 5)
    snap = list(pool.ref)
    with pytest.raises(P.OutOfSlots):
        pool.fork(a, 3)
    assert pool.ref == snap and len(pool.live()) == 1


def test_merge_is_an_append_to_main():
    p1 = P.RefPool(n_blocks=32, seed=4)
    p2 = P.RefPool(n_blocks=32, seed=4)
    for p in (p1, p2):
        m = p.create()
        p.append([m], 37)
    p1.merge(0, 50)
    p2.append([0], 50)
    assert p1.seqs[0].table == p2.seqs[0].table and list(p1.free) == list(p2.free)


def test_fork_at_full_length_is_fork():
    p1, p2 = P.RefPool(64, 5), P.RefPool(64, 5)
    for p in (p1, p2):
        p.create()
        p.append([0], 37)
    a = p1.fork(0, 2)
    b = p2.fork_at(0, 37, 2)
    assert [p1.seqs[i].table for i in a] == [p2.seqs[i].table for i in b] and p1.ref == p2.ref


def test_fork_at_mid_page_copies_on_first_append():
    pool = P.RefPool(32, 6, track_content=True)
    m = pool.create()
    pool.append([m], 40, [[("m", i) for i in range(40)]])
    (c,) = pool.fork_at(m, 21, 1)                 # page 1 holds rows 16..31 of main; the child sees 16..20
    assert pool.seqs[c].table == pool.seqs[m].table[:2]
    ev = pool.append([c], 1, [[("c", 0)]])
    assert len(ev) == 1 and ev[0][0] == pool.seqs[m].table[1] and ev[0][2] == 5
    assert pool.read(c) == [("m", i) for i in range(21)] + [("c", 0)]
    assert pool.read(m) == [("m", i) for i in range(40)]


def _fork_family(seed):
    """main with 37 rows (a partial third page) and three forks of it, plus a
    fresh sequence: content tracked, labels (sequence, row)."""
    pool = P.RefPool(n_blocks=64, seed=seed, track_content=True)
    m = pool.create()
    pool.append([m], 37, [[("m", i) for i in range(37)]])
    kids = pool.fork(m, 3)
    fresh = pool.create()
    return pool, [m] + kids + [fresh]


def test_ragged_prefill_equals_appends_one_by_one():
    counts = [5, 0, 27, 1, 40]     # unequal; one empty; copies of the shared partial page
    a, ids = _fork_family(8)
    b, _ = _fork_family(8)
    labels = [[(i, t) for t in range(n)] for i, n in zip(ids, counts)]
    ev_batch = a.prefill_batch(ids, counts, labels)
    ev_single = []
    for i, n, lab in zip(ids, counts, labels):
        ev_single += b.prefill_batch([i], [n], [lab])
    assert ev_batch == ev_single
    assert [a.seqs[i].table for i in ids] == [b.seqs[i].table for i in ids]
    assert [a.seqs[i].length for i in ids] == [37 + 5, 37, 37 + 27, 37 + 1, 40]
    assert a.ref == b.ref and list(a.free) == list(b.free)
    # every sequence reads back its own rows after its history, nobody else's
    hist = {ids[0]: [("m", r) for r in range(37)]}
    for k in ids[1:4]:
        hist[k] = [("m", r) for r in range(37)]
    hist[ids[4]] = []
    for i, lab in zip(ids, labels):
        assert a.read(i) == hist[i] + lab
    _check_invariants(a)


def test_ragged_prefill_copies_the_shared_page_only_for_sequences_that_grow():
    pool, ids = _fork_family(2)
    shared = pool.seqs[ids[0]].table[2]
    ev = pool.prefill_batch(ids[:4], [0, 3, 0, 1])
    # the two growing forks copy rows [0, 5) of the shared third page; the
    # main thread and the idle fork keep referencing it
    assert [e[0] for e in ev] == [shared, shared] and all(e[2] == 5 for e in ev)
    assert pool.ref[shared] == 2
    assert pool.seqs[ids[0]].table[2] == pool.seqs[ids[2]].table[2] == shared


def test_ragged_prefill_capacity_is_checked_for_the_whole_call():
    # 10 pages; after a = 5 rows (1 page) and b = 17 rows (2 pages) 7 are free.
    # [12, 20, 96] needs 1 + 1 + 6 = 8 pages: refused, nothing changes.
    # [12, 20, 80] needs 1 + 1 + 5 = 7 pages: taken, the free list empties.
    pool = P.RefPool(n_blocks=10, seed=4, track_content=True)
    a, b, c = pool.create(), pool.create(), pool.create()
    pool.prefill_batch([a, b, c], [5, 17, 0])
    assert len(pool.free) == 7
    snap = (list(pool.ref), list(pool.free), [list(pool.seqs[i].table) for i in (a, b, c)],
            [pool.seqs[i].length for i in (a, b, c)])
    with pytest.raises(P.OutOfBlocks):
        pool.prefill_batch([a, b, c], [12, 20, 96])
    assert snap == (list(pool.ref), list(pool.free), [list(pool.seqs[i].table) for i in (a, b, c)],
                    [pool.seqs[i].length for i in (a, b, c)])
    pool.prefill_batch([a, b, c], [12, 20, 80])
    assert len(pool.free) == 0
    assert [len(pool.seqs[i].table) for i in (a, b, c)] == [2, 3, 5]
    _check_invariants(pool)
