"""GPU parity: the CUDA path (through the C ABI) against the float64 oracle on
the same seeded inputs.  Block tables, refcounts and the free list must match
bit-exactly; O within 2e-3 + 1e-2|ref| element-wise, LSE within 1e-4."""
import numpy as np
import pytest
import torch

from fg_harness import Run, compare
from oracle import attention as A
from workloads import Workload, get

pytestmark = pytest.mark.gpu

CHUNK = 8192  # prefix rows per append call


def _prefix(run, rid, P, tag):
    for c0 in range(0, P, CHUNK):
        run.append([rid], min(CHUNK, P - c0), (tag, c0))


def _run(w, **kw):
    lim = dict(w.limits)
    lim.update(kw)
    return Run(w, **lim)


def test_cfg1_tiny_fork_group(stlib):
    w = get(1)
    run = _run(w)
    m = run.create()
    run.append([m], w.prefix[0], ("prefix",))
    aux = run.fork(m, w.n_aux)
    for i, (a, s) in enumerate(zip(aux, w.suffix[0][1:])):
        run.append([a], s, ("suffix", i))
    rids = [m] + aux
    q, o, lse = run.decode(rids, ("q",))
    run.pool.sync()
    run.check_tables()
    o_ref, l_ref = run.oracle_decode(rids, q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "cfg1")
    # the prefix pages are permuted in physical memory
    table = run.pool.block_table(run.handle[m])[0]
    assert table != sorted(table)


def test_cfg2_single_agent_turn(stlib):
    w = get(2)
    run = _run(w)
    m = run.create()
    run.append([m], w.prefix[0], ("prefix",))
    aux = run.fork(m, w.n_aux)
    rids = [m] + aux
    run.append(rids, w.suffix[0][0], ("suffix",))
    checks = {0, 1, 15, 16, 100, w.steps - 1}
    for step in range(w.steps):
        run.append(rids, 1, ("step", step))
        q, o, lse = run.decode(rids, ("q", step))
        if step in checks:
            o_ref, l_ref = run.oracle_decode(rids, q, 0)
            compare(o[0], lse[0], o_ref, l_ref, f"cfg2 step {step}")
    run.pool.sync()
    run.check_tables()


def test_cfg3_batched_agent_serving(stlib):
    w = get(3)
    run = _run(w)
    groups = []
    for t in range(w.n_tasks):
        m = run.create()
        _prefix(run, m, w.prefix[t], ("prefix", t))
        aux = run.fork(m, w.n_aux)
        br = [m] + aux
        for b, (rid, s) in enumerate(zip(br, w.suffix[t])):
            if s:
                run.append([rid], s, ("suffix", t, b))
        groups.append(br)
    rids = [r for g in groups for r in g]
    run.append(rids, 1, ("step",))
    q, o, lse = run.decode(rids, ("q",))
    run.pool.sync()
    run.check_tables()
    o_ref, l_ref = run.oracle_decode(rids, q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "cfg3")


def _long_groups(run, w):
    groups = []
    for t in range(w.n_tasks):
        m = run.create()
        _prefix(run, m, w.prefix[t], ("prefix", t))
        aux = run.fork(m, w.n_aux)
        br = [m] + aux
        for b, (rid, s) in enumerate(zip(br, w.suffix[t])):
            if s:
                run.append([rid], s, ("suffix", t, b))
        groups.append(br)
    return groups


def _check_every_layer(run, w, groups, q, o, lse, jobs, what, pick=None):
    """Every branch of every group (or the branches `pick` chooses by their
    index in the group) on every layer, one (layer, group) oracle job each,
    spread over the worker processes."""
    o_cpu, l_cpu, q_cpu = o.cpu(), lse.cpu(), q.cpu()
    futs, col = [], 0
    for g in groups:
        sel = sorted(set(pick(len(g)))) if pick else list(range(len(g)))
        idx = [col + i for i in sel]
        col += len(g)
        for layer in range(w.n_layers):
            futs.append((layer, idx, jobs.decode(w, layer, q_cpu[layer, idx], [run.hist[g[i]] for i in sel],
                                                  run.sizes)))
    for layer, idx, f in futs:
        o_ref, l_ref = f.get()
        compare(o_cpu[layer, idx], l_cpu[layer, idx], o_ref, l_ref, f"{what} layer {layer} rows {idx[0]}..")


def test_cfg4_long_trajectory_every_layer(stlib, oracle_jobs):
    """The long-trajectory workload at full size (4 groups x 131072-token
    prefixes, 32 layers): every branch checked on every layer."""
    w = get(4)
    run = _run(w, cache_layers=48)
    groups = _long_groups(run, w)
    rids = [r for g in groups for r in g]
    run.append(rids, 1, ("step",))
    q, o, lse = run.decode(rids, ("q",))
    run.pool.sync()
    run.check_tables()
    _check_every_layer(run, w, groups, q, o, lse, oracle_jobs, "cfg4")


@pytest.mark.parametrize("n_aux", [7, 8, 16])
def test_cfg4_long_trajectory_wide_every_layer(stlib, oracle_jobs, n_aux):
    """The long-trajectory workload at full size with 8 branches per group (64
    stacked rows: a full narrow tile, all four softmax warps), 9 (72 rows: one
    wide tile per group) and 17 (136 rows: the paired tile, 128 rows in its
    first tile and 8 in its second), as `bench.py --n-aux` times it; on every
    layer, six branches per group: the first two, two in the middle and the
    last two (the last one in the paired tile's second tile)."""
    from workloads.configs import long_with_branches
    w = long_with_branches(n_aux)
    run = _run(w, cache_layers=48)
    groups = _long_groups(run, w)
    rids = [r for g in groups for r in g]
    run.append(rids, 1, ("step",))
    q, o, lse = run.decode(rids, ("q",))
    run.pool.sync()
    run.check_tables()
    _check_every_layer(run, w, groups, q, o, lse, oracle_jobs, w.name,
                       pick=lambda n: [0, 1, n // 2, n // 2 + 1, n - 2, n - 1])


def test_cfg5_full_cycle(stlib, oracle_jobs):
    """The full cycle (8 tasks x 5 turns of fork, 512 append + decode steps,
    merge of 2048 thought rows, release; 64 unforked sequences per turn).
    Tables, refcounts and the free list are compared after every turn; O and
    LSE of all 104 branches at steps 1, 64, 128, ..., 512 of every turn (each
    check on its own layer); every row of turn 1 / task 0's merge, and for the
    other merges 1 row in 16: the first and last row of each 64-row work item
    plus a seeded sample."""
    w = get(5)
    run = _run(w, cache_layers=32)
    mains = []
    for t in range(w.n_tasks):
        m = run.create()
        _prefix(run, m, w.prefix[t], ("prefix", t))
        mains.append(m)
    rng = np.random.default_rng(5)
    check_steps = [0] + list(range(63, w.steps, 64))   # steps 1, 64, 128, ..., 512 counted from 1
    T = w.merge_tokens
    chunk = 256 // w.group                               # thought rows per merge work item
    futs = []
    n_check = 0
    for turn in range(w.turns):
        singles = [run.create() for _ in range(w.singletons)]
        for i in range(0, w.singletons, 8):
            run.append(singles[i:i + 8], w.singleton_len, ("single", turn, i))
        groups = [[m] + run.fork(m, w.n_aux) for m in mains]
        rids = [r for g in groups for r in g] + singles
        for step in range(w.steps):
            run.append(rids, 1, ("step", turn, step))
            q, o, lse = run.decode(rids, ("q", turn, step))
            if step in check_steps:
                layer = (5 * n_check + 3) % w.n_layers
                n_check += 1
                o_c, l_c, q_c = o[layer].cpu(), lse[layer].cpu(), q[layer].cpu()
                for b0 in range(0, len(rids), 26):
                    sl = slice(b0, b0 + 26)
                    f = oracle_jobs.decode(w, layer, q_c[sl], [list(run.hist[r]) for r in rids[sl]],
                                           dict(run.sizes))
                    futs.append((f"cfg5 turn {turn} step {step + 1} layer {layer} branches {b0}..",
                                 o_c[sl], l_c[sl], f))
        for t, m in enumerate(mains):
            pieces = list(run.hist[m])
            qm, om, lm, L0 = run.merge(m, T, ("merge", turn, t))
            layer = (11 * turn + 3 * t + 1) % w.n_layers
            if turn == 0 and t == 0:
                rows = list(range(T))
            else:
                edge = {r for c0 in range(0, T, chunk) for r in (c0, min(c0 + chunk, T) - 1)}
                rest = sorted(set(range(T)) - edge)
                rows = sorted(edge | set(rng.choice(rest, T // 16 - len(edge), replace=False).tolist()))
            pieces = pieces + [(("merge", turn, t), 0, T)]
            q_c, o_c, l_c = qm[layer].cpu(), om[layer].cpu(), lm[layer].cpu()
            for r0 in range(0, len(rows), 128):
                part = rows[r0:r0 + 128]
                f = oracle_jobs.merge(w, layer, q_c, pieces, dict(run.sizes), L0, part)
                futs.append((f"cfg5 merge turn {turn} task {t} layer {layer} rows {part[0]}..{part[-1]}",
                             o_c[part], l_c[part], f))
        for g in groups:
            for a in g[1:]:
                run.release(a)
        for s in singles:
            run.release(s)
        run.pool.sync()
        run.check_tables()
    for what, o_g, l_g, f in futs:
        o_ref, l_ref = f.get()
        compare(o_g, l_g, o_ref, l_ref, what)


# ---- edge cases on small shapes -------------------------------------------

def _small(D, Hq, Hkv, n_blocks=512, L=2, seed=11, scale=1.0):
    return Workload(name=f"edge_{D}_{Hq}_{Hkv}", n_layers=L, n_q_heads=Hq, n_kv_heads=Hkv,
                    head_dim=D, n_blocks=n_blocks, seed=seed, value_scale=scale)


@pytest.mark.parametrize("D,Hq,Hkv,n_aux,P,suffix", [
    (64, 8, 2, 4, 512, (0, 16, 33, 47, 64)),
    (128, 32, 8, 1, 1000, (5, 0)),
    (128, 8, 8, 7, 777, (1, 2, 3, 0, 16, 17, 31, 100)),      # G = 1, eight branches
    (128, 64, 8, 4, 300, (0, 1, 15, 16, 17)),                # G = 8, 40 stacked rows
    (128, 64, 8, 8, 4100, (3,) * 9),                         # 9 x 8 = 72 rows: one wide tile
    (128, 16, 1, 3, 2000, (0, 9, 0, 40)),                    # G = 16, 64 rows: a full narrow tile
    (128, 64, 8, 6, 2222, (0, 3, 17, 0, 1, 2, 40)),          # G = 8, 56 rows: narrow, four softmax warps
    (128, 40, 8, 12, 1800, (1,) * 13),                       # G = 5, 65 rows: one past narrow, wide
    (64, 64, 4, 3, 1000, (5, 0, 16, 33)),                    # G = 16, 64 rows, D 64: narrow
    (64, 48, 4, 7, 900, (2,) * 8),                           # G = 12, 96 rows: wide, D 64
    (128, 32, 1, 3, 1500, (0, 5, 9, 33)),                    # G = 32, 128 rows: a full wide tile
    (128, 48, 1, 4, 700, (1, 2, 3, 4, 5)),                   # G = 48, 240 rows: wide subgroups 1 + 2 + 2
    (64, 20, 2, 5, 3333, (0, 7, 16, 31, 64, 65)),            # G = 10, 60 rows: narrow, D 64
    (128, 32, 1, 1, 100, (0, 0)),                            # G = 32, no suffixes
    (64, 4, 1, 0, 50, (0,)),                                 # a lone main thread
    (64, 12, 3, 2, 16, (0, 1, 2)),                           # one-page prefix
    (128, 32, 8, 4, 15, (0, 1, 2, 3, 4)),                    # prefix shorter than a page
])
def test_shapes(stlib, D, Hq, Hkv, n_aux, P, suffix):
    w = _small(D, Hq, Hkv)
    run = Run(w, max_seqs=16, max_decode_branches=16, max_splits=8)
    m = run.create()
    run.append([m], P, ("prefix",))
    br = [m] + (run.fork(m, n_aux) if n_aux else [])
    for b, (rid, s) in enumerate(zip(br, suffix)):
        if s:
            run.append([rid], s, ("suffix", b))
    q, o, lse = run.decode(br, ("q",))
    run.pool.sync()
    run.check_tables()
    for layer in range(w.n_layers):
        o_ref, l_ref = run.oracle_decode(br, q, layer)
        compare(o[layer], lse[layer], o_ref, l_ref, f"layer {layer}")


@pytest.mark.parametrize("D,Hq,Hkv,n_br,P", [
    (128, 64, 8, 17, 3000),    # G = 8, 136 rows: one paired tile, its second tile 8 rows
    (128, 128, 8, 16, 2000),   # G = 16, 256 rows: a full paired tile
    (64, 48, 16, 43, 1500),    # G = 3, 129 rows
    (128, 64, 8, 40, 5000),    # 320 rows: two paired subgroups of 160
    (64, 32, 2, 20, 777),      # G = 16, D 64, 320 rows
])
def test_large_fork_groups(stlib, D, Hq, Hkv, n_br, P):
    """Fork groups beyond 128 stacked rows: one paired tile (two M = 128 tiles
    of one CTA over every stage) up to 256, balanced paired subgroups beyond,
    each branch with a suffix of its own; every layer against the oracle."""
    w = _small(D, Hq, Hkv, n_blocks=4096, L=2, seed=13)
    run = Run(w, max_seqs=64, max_decode_branches=48, max_splits=8)
    m = run.create()
    run.append([m], P, ("prefix",))
    br = [m] + run.fork(m, n_br - 1)
    for b, rid in enumerate(br):
        if b % 3 and (7 * b) % 41:
            run.append([rid], (7 * b) % 41, ("suffix", b))
    q, o, lse = run.decode(br, ("q",))
    run.pool.sync()
    run.check_tables()
    for layer in range(w.n_layers):
        o_ref, l_ref = run.oracle_decode(br, q, layer)
        compare(o[layer], lse[layer], o_ref, l_ref, f"{n_br} branches, layer {layer}")


def test_many_splits_on_a_long_singleton(stlib):
    w = _small(128, 32, 8, n_blocks=4096, L=1)
    run = Run(w, max_seqs=4, max_decode_branches=4, max_splits=32)
    a = run.create()
    for c0 in range(0, 40000, 8000):
        run.append([a], 8000, ("ctx", c0))
    b = run.create()
    run.append([b], 3, ("short",))
    q, o, lse = run.decode([a, b], ("q",))
    o_ref, l_ref = run.oracle_decode([a, b], q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "long singleton")


def test_stale_nan_pool_memory_does_not_leak(stlib):
    w = _small(128, 32, 8, n_blocks=256, L=1)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=8)
    run.pool.k_pool.fill_(float("nan"))
    run.pool.v_pool.fill_(float("nan"))
    m = run.create()
    run.append([m], 999, ("prefix",))
    br = [m] + run.fork(m, 4)
    for b, rid in enumerate(br):
        run.append([rid], b * 5 + 1, ("suffix", b))
    q, o, lse = run.decode(br, ("q",))
    o_ref, l_ref = run.oracle_decode(br, q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "nan pool")
    T = 37
    qm, om, lm, L0 = run.merge(m, T, ("merge",))
    k, v = run.context(m, 0)
    o_ref, l_ref = A.merge_prefill(qm[0].cpu(), k, v, L0)
    compare(om[0], lm[0], o_ref, l_ref, "nan pool merge")


def test_outputs_do_not_depend_on_page_placement(stlib):
    outs = []
    for seed in (1, 2):
        w = _small(128, 32, 8, n_blocks=512, L=1)
        run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=8, pool_seed=seed)
        m = run.create()
        run.append([m], 3000, ("prefix",))
        br = [m] + run.fork(m, 4)
        for b, rid in enumerate(br[1:], start=1):
            run.append([rid], 7 * b, ("suffix", b))
        q, o, lse = run.decode(br, ("q",))
        outs.append((o.clone(), lse.clone(), run.pool.block_table(run.handle[m])[0]))
    assert outs[0][2] != outs[1][2]
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])


def test_copy_on_write_keeps_siblings_intact(stlib):
    w = _small(64, 8, 2, n_blocks=128, L=2)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=8)
    m = run.create()
    run.append([m], 40, ("prefix",))      # two full pages + 8 rows in a shared page
    aux = run.fork(m, 2)
    run.append([aux[0]], 20, ("a0",))     # copies the shared page, then writes
    run.append([m], 3, ("m",))            # copies too (still shared with aux[1])
    run.append([aux[1]], 1, ("a1",))      # last holder: writes in place
    br = [m] + aux
    q, o, lse = run.decode(br, ("q",))
    run.pool.sync()
    run.check_tables()
    for layer in range(2):
        o_ref, l_ref = run.oracle_decode(br, q, layer)
        compare(o[layer], lse[layer], o_ref, l_ref, f"cow layer {layer}")


@pytest.mark.parametrize("D,Hq,Hkv,L0,T", [
    (128, 32, 8, 1000, 1), (128, 32, 8, 1000, 5), (128, 32, 8, 1003, 17), (128, 64, 8, 512, 100),
    (64, 8, 2, 77, 64), (128, 8, 8, 33, 130), (128, 32, 1, 16, 9),
])
def test_merge_prefill(stlib, D, Hq, Hkv, L0, T):
    w = _small(D, Hq, Hkv, n_blocks=512, L=2)
    run = Run(w, max_seqs=4, max_decode_branches=4, max_splits=8)
    m = run.create()
    run.append([m], L0, ("ctx",))
    aux = run.fork(m, 1)                  # a live sibling shares main's pages
    qm, om, lm, L0r = run.merge(m, T, ("merge",))
    assert L0r == L0
    run.pool.sync()
    run.check_tables()
    for layer in range(2):
        k, v = run.context(m, layer)
        o_ref, l_ref = A.merge_prefill(qm[layer].cpu(), k, v, L0)
        compare(om[layer], lm[layer], o_ref, l_ref, f"merge layer {layer}")
    # the sibling still sees only the pre-merge context
    q, o, lse = run.decode(aux, ("q",))
    o_ref, l_ref = run.oracle_decode(aux, q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "sibling after merge")


@pytest.mark.parametrize("D,Hq,Hkv,L0,T", [
    (128, 32, 8, 2047, 1),      # 2048 keys: the last merge on the two-term path
    (128, 32, 8, 2048, 1),      # 2049 keys: the first on the paired-tile path
    (64, 8, 2, 2100, 64),       # D 64, one CTA, tile B partly filled
    (128, 32, 8, 2500, 37),     # 148 stacked rows: tile B ragged
    (128, 64, 8, 3001, 40),     # 320 rows: a second CTA, context ends mid-page
    (128, 8, 8, 4096, 300),     # G 1, page-aligned context
    (64, 32, 4, 5000, 129),     # short last stage (few pages loaded)
])
def test_merge_prefill_long_context(stlib, D, Hq, Hkv, L0, T):
    w = _small(D, Hq, Hkv, n_blocks=1024, L=2)
    run = Run(w, max_seqs=4, max_decode_branches=4, max_splits=8)
    m = run.create()
    run.append([m], L0, ("ctx",))
    qm, om, lm, L0r = run.merge(m, T, ("merge",))
    assert L0r == L0
    run.pool.sync()
    run.check_tables()
    for layer in range(2):
        k, v = run.context(m, layer)
        o_ref, l_ref = A.merge_prefill(qm[layer].cpu(), k, v, L0)
        compare(om[layer], lm[layer], o_ref, l_ref, f"long merge layer {layer}")


@pytest.mark.parametrize("D,kind", [(128, "merge"), (64, "merge"), (128, "decode"), (64, "decode")])
def test_running_max_raised_after_the_first_stage(stlib, D, kind):
    # values x3: scores have a standard deviation near 9, so later stages keep
    # exceeding the running max by more than 2^8 and O is rescaled in TMEM
    w = _small(D, 16, 4, n_blocks=1024, L=1, scale=3.0)
    run = Run(w, max_seqs=4, max_decode_branches=4, max_splits=8)
    m = run.create()
    run.append([m], 6000, ("ctx",))
    if kind == "merge":
        qm, om, lm, L0 = run.merge(m, 50, ("merge",))
        k, v = run.context(m, 0)
        o_ref, l_ref = A.merge_prefill(qm[0].cpu(), k, v, L0)
        compare(om[0], lm[0], o_ref, l_ref, "merge with rescales")
    else:
        aux = run.fork(m, 2)
        br = [m] + aux
        run.append(br, 1, ("s",))
        q, o, lse = run.decode(br, ("q",))
        o_ref, l_ref = run.oracle_decode(br, q, 0)
        compare(o[0], lse[0], o_ref, l_ref, "decode with rescales")


def test_merge_of_one_row_equals_decode_after_append(stlib):
    w = _small(128, 32, 8, n_blocks=256, L=1)
    run = Run(w, max_seqs=4, max_decode_branches=4, max_splits=8)
    m = run.create()
    run.append([m], 500, ("ctx",))
    qm, om, lm, _ = run.merge(m, 1, ("merge",))
    o, lse = run.pool.decode_attn([run.handle[m]], qm.view(1, 1, w.n_q_heads, w.head_dim).contiguous())
    torch.testing.assert_close(o[0, 0], om[0, 0], atol=2e-3, rtol=1e-2)
    torch.testing.assert_close(lse[0, 0], lm[0, 0], atol=1e-4, rtol=0)


def test_merge_of_nothing_changes_nothing(stlib):
    w = _small(128, 32, 8, n_blocks=64, L=1)
    run = Run(w, max_seqs=4, max_decode_branches=4, max_splits=8)
    m = run.create()
    run.append([m], 20, ("ctx",))
    snap = (run.pool.refcounts(), run.pool.free_list(), run.pool.block_table(run.handle[m]))
    e = torch.empty((1, 0, w.n_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    kv = torch.empty((1, 0, w.n_kv_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    run.pool.merge(run.handle[m], e, kv, kv)
    assert snap == (run.pool.refcounts(), run.pool.free_list(), run.pool.block_table(run.handle[m]))
    run.pool.sync()


@pytest.mark.parametrize("variant", ["without_r_t", "fork_onset"])
def test_fork_point_variants(stlib, variant):
    """Table 2 of the paper: branches that do not see the just-finished
    thought R_t ("w/o R_t": fork at the end of H_t) or fork when the turn
    starts ("fork onset": the window also covers the Thought phase, so the
    branches decode while main is still writing R_t)."""
    w = _small(128, 32, 8, n_blocks=512, L=2)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=8)
    m = run.create()
    run.append([m], 1003, ("H_t",))                     # history, ends mid-page
    if variant == "without_r_t":
        run.append([m], 77, ("R_t",))                   # main's thought
        aux = run.fork_at(m, 1003, 4)                   # branches see H_t only
    else:
        aux = run.fork(m, 4)                            # fork at turn onset
        run.append([m], 77, ("R_t",))                   # main thinks while branches run
    for step in range(20):
        run.append([m] + aux, 1, ("step", step))
        q, o, lse = run.decode([m] + aux, ("q", step))
        if step in (0, 19):
            for layer in range(2):
                o_ref, l_ref = run.oracle_decode([m] + aux, q, layer)
                compare(o[layer], lse[layer], o_ref, l_ref, f"{variant} step {step} layer {layer}")
    run.pool.sync()
    run.check_tables()


def test_profile_counts_device_kernels(stlib):
    """A decode call whose fork group needs the wide tile (9 branches x G = 8 =
    72 stacked rows) while each branch's own pages take narrow tiles launches
    two decode kernels; the profile counts calls and kernels apart."""
    w = Workload(name="kernel_count", n_layers=1, n_q_heads=8, n_kv_heads=1, head_dim=64, n_blocks=256, seed=0)
    run = Run(w, max_seqs=16, max_decode_branches=16, max_splits=8)
    m = run.create()
    run.append([m], 256, ("p",))
    rids = [m] + run.fork(m, 8)
    for b, r in enumerate(rids):
        run.append([r], 20, ("s", b))
    run.pool.profile_read()
    q, o, lse = run.decode(rids, ("q",))
    st = run.pool.profile_read()["decode_partial"]
    assert (st["launches"], st["kernels"]) == (1, 2)
    o_ref, l_ref = run.oracle_decode(rids, q, 0)
    compare(o[0], lse[0], o_ref, l_ref, "wide + narrow")
    q, o, lse = run.decode(rids[:2], ("q2",))  # 16 rows: narrow tiles only
    st = run.pool.profile_read()["decode_partial"]
    assert (st["launches"], st["kernels"]) == (1, 1)
