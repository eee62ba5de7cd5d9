"""The decode planner (host logic, no GPU): the items st_decode_attn would
launch, reported by st_decode_plan on metadata-only pools, cover every
branch's context exactly once (Section 3.3: the snapshot is shared, so a
page held by a whole fork group is read once for all of it), every partial
slot is written by one item, and the tile choice matches the stacked rows."""
import numpy as np
import pytest

import paper_2608_13667_gb300 as stpkg

PAGE = 16
NARROW_ROWS, WIDE_ROWS, PAIR_ROWS = 64, 128, 256
WIDE, REREAD, PAIR = 2, 1, 4


def _pool(G, Hkv, max_splits, n_blocks=1 << 15):
    return stpkg.Pool(n_layers=2, n_q_heads=G * Hkv, n_kv_heads=Hkv, head_dim=128, n_blocks=n_blocks, device=None,
                      max_seqs=96, max_decode_branches=48, max_splits=max_splits)


def check_plan(P, br, G, max_splits):
    items, members, ns = P.decode_plan(br)
    tables, lens = zip(*(P.block_table(h) for h in br))
    n = len(br)
    covered = [dict() for _ in range(n)]   # logical page -> physical id, per branch
    tokens = [0] * n
    splits = [[] for _ in range(n)]
    last_tile = 0
    for it in items:
        mem = members[it["member_base"]:it["member_base"] + it["n_members"]]
        own = tables[it["owner"]]
        p0, np_ = it["page_begin"], it["n_pages"]
        assert np_ >= 1 and it["n_tokens"] >= 1
        tile = 2 if it["flags"] & PAIR else 1 if it["flags"] & WIDE else 0
        assert not (it["flags"] & PAIR and it["flags"] & WIDE)
        assert len(mem) * G <= (NARROW_ROWS, WIDE_ROWS, PAIR_ROWS)[tile]
        assert not (it["flags"] & REREAD) or tile == 2, "only families beyond one paired tile are split"
        assert tile >= last_tile, "narrow items first, then wide, then paired"
        last_tile = tile
        if len(mem) > 1:
            assert it["n_tokens"] == np_ * PAGE   # a shared run holds full pages only
        else:
            assert mem == [it["owner"]]
        for i in mem:
            for p in range(p0, p0 + np_):
                assert p not in covered[i], f"branch {i} page {p} read twice"
                assert tables[i][p] == own[p], f"branch {i} page {p} read from another table"
                covered[i][p] = own[p]
            if len(mem) > 1:
                assert (p0 + np_) * PAGE <= lens[i]
            tokens[i] += it["n_tokens"]
            splits[i].append(it["split"])
    for i in range(n):
        assert sorted(covered[i]) == list(range(len(tables[i]))), f"branch {i} pages not covered once"
        assert tokens[i] == lens[i]
        assert sorted(splits[i]) == list(range(ns[i])) and ns[i] <= max_splits
    return items, members


def _random_case(rng):
    G = int(rng.choice([1, 2, 4, 8, 12, 16, 48]))
    Hkv = int(rng.choice([1, 2]))
    max_splits = int(rng.choice([2, 3, 8, 16, 32]))
    P = _pool(G, Hkv, max_splits)
    br = []
    for f in range(int(rng.integers(1, 4))):
        m = P.seq_create()
        P.append_kv([m], int(rng.integers(1, 5000)), None)
        fam = [m]
        n_aux = int(rng.integers(0, 21))
        if n_aux:
            L = P.block_table(m)[1]
            kids = P.fork_at(m, int(rng.integers(0, L + 1)), n_aux) if rng.random() < 0.3 else P.fork(m, n_aux)
            fam += kids
            if rng.random() < 0.3:   # a fork of a fork
                fam += P.fork(kids[0], int(rng.integers(1, 4)))
        for h in fam:
            s = int(rng.integers(0, 100))
            if s:
                P.append_kv([h], s, None)
        br += [h for h in fam if P.block_table(h)[1] > 0]
    for _ in range(int(rng.integers(0, 4))):
        h = P.seq_create()
        P.append_kv([h], int(rng.integers(1, 600)), None)
        br.append(h)
    br = br[:48]
    rng.shuffle(br)
    return P, br, G, max_splits


@pytest.mark.parametrize("seed", range(60))
def test_random_plans_cover_each_context_once(stlib, seed):
    P, br, G, max_splits = _random_case(np.random.default_rng(7000 + seed))
    check_plan(P, br, G, max_splits)
    P.close()


def test_shared_prefix_is_read_once_per_group(stlib):
    """The paper's 1 + 4 branches at G = 8 (40 stacked rows: one narrow tile):
    the shared full pages are read by group items only, once."""
    P = _pool(8, 2, 32)
    m = P.seq_create()
    P.append_kv([m], 8192 + 5, None)
    br = [m] + P.fork(m, 4)
    for h in br:
        P.append_kv([h], 40, None)
    items, members = check_plan(P, br, 8, 32)
    shared = [it for it in items if it["n_members"] > 1]
    assert sum(it["n_pages"] for it in shared) == 8192 // PAGE
    assert all(it["n_members"] == 5 and not it["flags"] & WIDE for it in shared)


@pytest.mark.parametrize("n_br,G,tiles", [(6, 8, 1), (7, 8, 1), (8, 8, 1), (9, 8, 1), (13, 5, 1), (16, 8, 1),
                                         (17, 8, 1), (40, 4, 1), (9, 16, 1), (32, 8, 1), (33, 8, 2), (48, 8, 2),
                                         (6, 48, 2), (48, 16, 3)])
def test_tile_choice_follows_the_stacked_rows(stlib, n_br, G, tiles):
    """Up to 64 stacked rows: narrow; up to 128: one wide tile; up to 256: one
    paired tile; beyond: balanced paired subgroups, each over the family's
    common pages, flagged so the sibling's read of a page comes from L2."""
    P = _pool(G, 1, 32)
    m = P.seq_create()
    P.append_kv([m], 4096, None)
    br = [m] + P.fork(m, n_br - 1)
    for h in br:
        P.append_kv([h], 3, None)
    items, members = check_plan(P, br, G, 32)
    shared = [it for it in items if it["n_members"] > 1]
    groups = {it["member_base"] for it in shared}
    assert len(groups) == tiles
    rows = n_br * G
    assert all(bool(it["flags"] & WIDE) == (NARROW_ROWS < rows <= WIDE_ROWS) for it in shared)
    assert all(bool(it["flags"] & PAIR) == (rows > WIDE_ROWS) for it in shared)
    assert all(bool(it["flags"] & REREAD) == (tiles > 1) for it in shared)
    if tiles > 1:
        sizes = sorted(it["n_members"] for it in shared if it["split"] == 0)
        assert sizes[-1] - sizes[0] <= 1   # balanced subgroups


def test_plan_rejects_what_decode_rejects(stlib):
    P = _pool(4, 2, 8)
    m = P.seq_create()
    with pytest.raises(stpkg.STError):
        P.decode_plan([m])            # an empty sequence
    P.append_kv([m], 10, None)
    with pytest.raises(stpkg.STError):
        P.decode_plan([m, m])         # listed twice
