"""st_decode_step -- one KV row appended to every branch, then the decode, the
row written into its page by the decode kernel that reads it -- against
st_append_kv followed by st_decode_attn on a twin pool (same seeds, same
pages): tables equal, outputs bitwise equal, and both against the float64
oracle."""
import pytest
import torch

from fg_harness import Run, compare
from workloads import Workload, kv_rows, queries

pytestmark = pytest.mark.gpu


def _step_fused(run, rids, tag, qtag):
    w = run.w
    k, v = kv_rows(w, tag, len(rids), device="cuda")        # [L][n_br][Hkv][D]
    q = queries(w, qtag, len(rids), device="cuda")
    o, lse = run.pool.decode_step([run.handle[r] for r in rids], k, v, q)
    run.ref.append(rids, 1)
    run.sizes[tag] = len(rids)
    for i, r in enumerate(rids):
        run.hist[r].append((tag, i, 1))
    return q, o, lse


def _twins(w, setup, **kw):
    runs = [Run(w, **kw), Run(w, **kw)]
    rids = [setup(r) for r in runs]
    assert rids[0] == rids[1]
    return runs, rids[0]


def _drive(runs, rids, steps, checks):
    a, b = runs
    for step in range(steps):
        a.append(rids, 1, ("step", step))
        qa, oa, la = a.decode(rids, ("q", step))
        qb, ob, lb = _step_fused(b, rids, ("step", step), ("q", step))
        assert torch.equal(oa, ob) and torch.equal(la, lb), f"step {step}: fused and separate differ"
        if step in checks:
            b.pool.sync()
            for layer in range(b.w.n_layers):
                o_ref, l_ref = b.oracle_decode(rids, qb, layer)
                compare(ob[layer], lb[layer], o_ref, l_ref, f"step {step} layer {layer}")
    for r in runs:
        r.pool.sync()
        r.check_tables()
    assert a.pool.block_table(a.handle[rids[0]]) == b.pool.block_table(b.handle[rids[0]])


def test_decode_step_single_agent(stlib):
    """1 + 4 branches forked off a 1000-token prefix (its last page shared and
    partly filled: the first step copies it with a separate append), then
    steps across page boundaries."""
    w = Workload(name="step_single", n_layers=2, n_q_heads=32, n_kv_heads=8, head_dim=128, n_blocks=1024, seed=31)

    def setup(run):
        m = run.create()
        run.append([m], 1000, ("prefix",))
        return [m] + run.fork(m, 4)

    runs, rids = _twins(w, setup, max_seqs=8, max_decode_branches=8, max_splits=16)
    _drive(runs, rids, 40, {0, 1, 8, 24, 39})


def test_decode_step_mixed_groups(stlib):
    """A 9-branch fork group (the wide tile) with suffixes, a lone sequence,
    and a sequence that is empty before the first step."""
    w = Workload(name="step_mixed", n_layers=1, n_q_heads=64, n_kv_heads=8, head_dim=128, n_blocks=2048, seed=32)

    def setup(run):
        m = run.create()
        run.append([m], 2048, ("prefix",))
        br = [m] + run.fork(m, 8)
        for i, r in enumerate(br):
            run.append([r], 3 + 5 * i, ("s", i))
        lone = run.create()
        run.append([lone], 333, ("lone",))
        empty = run.create()
        return br + [lone, empty]

    runs, rids = _twins(w, setup, max_seqs=16, max_decode_branches=16, max_splits=16)
    _drive(runs, rids, 20, {0, 13, 19})


def test_decode_step_paired_group_and_head_dim_64(stlib):
    """17 branches at G = 8 (the paired tile and the separate combine), and a
    D = 64 pool."""
    w = Workload(name="step_pair", n_layers=1, n_q_heads=64, n_kv_heads=8, head_dim=128, n_blocks=2048, seed=33)

    def setup(run):
        m = run.create()
        run.append([m], 1600, ("prefix",))
        return [m] + run.fork(m, 16)

    runs, rids = _twins(w, setup, max_seqs=24, max_decode_branches=20, max_splits=16)
    _drive(runs, rids, 6, {0, 5})

    w64 = Workload(name="step_d64", n_layers=3, n_q_heads=8, n_kv_heads=2, head_dim=64, n_blocks=512, seed=34)

    def setup64(run):
        m = run.create()
        run.append([m], 512, ("prefix",))        # page-aligned: no copy at the first step
        return [m] + run.fork(m, 4)

    runs, rids = _twins(w64, setup64, max_seqs=8, max_decode_branches=8, max_splits=8)
    _drive(runs, rids, 20, {0, 15, 19})
