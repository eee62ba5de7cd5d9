"""Randomised parity sweep: random geometries, split budgets, fork points,
group mixes and step counts, every decode, merge and batched prefill checked
against the float64 oracle, tables and refcounts checked bit-exactly."""
import numpy as np
import pytest

from fg_harness import Run, compare
from oracle import attention as A
from workloads import Workload

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("seed", range(40))
def test_random_fork_groups(stlib, seed):
    rng = np.random.default_rng(1000 + seed)
    D = int(rng.choice([64, 128]))
    Hkv = int(rng.choice([1, 2, 4, 8]))
    G = int(rng.choice([1, 2, 4, 8, 12]))
    L = int(rng.integers(1, 3))
    w = Workload(name=f"fuzz{seed}", n_layers=L, n_q_heads=Hkv * G, n_kv_heads=Hkv, head_dim=D,
                 n_blocks=1024, seed=seed)
    run = Run(w, max_seqs=32, max_decode_branches=32, max_splits=int(rng.choice([2, 3, 8, 32])))
    rids = []
    for g in range(int(rng.integers(1, 4))):                  # fork groups
        m = run.create()
        run.append([m], int(rng.integers(1, 3000)), ("p", g))
        n_aux = int(rng.integers(0, 6))
        if n_aux:
            if rng.random() < 0.3:
                kids = run.fork_at(m, int(rng.integers(0, run.ref.seqs[m].length + 1)), n_aux)
            else:
                kids = run.fork(m, n_aux)
        else:
            kids = []
        for b, r in enumerate([m] + kids):
            s = int(rng.integers(0, 70))
            if s:
                run.append([r], s, ("s", g, b))
        rids += [r for r in [m] + kids if run.ref.seqs[r].length > 0]
    for _ in range(int(rng.integers(0, 3))):                  # unforked sequences
        r = run.create()
        run.append([r], int(rng.integers(1, 500)), ("single", len(rids)))
        rids.append(r)
    rng.shuffle(rids)
    for step in range(3):
        run.append(rids, 1, ("step", step))
        q, o, lse = run.decode(rids, ("q", step))
        layer = int(rng.integers(0, L))
        o_ref, l_ref = run.oracle_decode(rids, q, layer)
        compare(o[layer], lse[layer], o_ref, l_ref, f"seed {seed} step {step}")
    m = rids[0]
    T = int(rng.integers(1, 90))
    qm, om, lm, L0 = run.merge(m, T, ("merge",))
    layer = int(rng.integers(0, L))
    k, v = run.context(m, layer)
    o_ref, l_ref = A.merge_prefill(qm[layer].cpu(), k, v, L0)
    compare(om[layer], lm[layer], o_ref, l_ref, f"seed {seed} merge")
    # a batched prefill over a random subset (ragged counts, zeros included)
    sub = [rids[i] for i in sorted(rng.choice(len(rids), size=int(rng.integers(1, len(rids) + 1)),
                                              replace=False))]
    counts = [int(rng.choice([0, 1, 9, 16, 17, 40, 77])) for _ in sub]
    qp, op, lp, L0s = run.prefill_batch(sub, counts, ("batch",))
    layer = int(rng.integers(0, L))
    off = 0
    for r, n, l0 in zip(sub, counts, L0s):
        if n:
            k, v = run.context(r, layer)
            o_ref, l_ref = A.merge_prefill(qp[layer, off:off + n].cpu(), k, v, l0)
            compare(op[layer, off:off + n], lp[layer, off:off + n], o_ref, l_ref, f"seed {seed} batch seq {r}")
        off += n
    run.pool.sync()
    run.check_tables()


@pytest.mark.parametrize("seed", range(12))
def test_random_large_fork_groups(stlib, seed):
    """Large fork groups: 7 to 21 branches at G = 4 or 8 (28 to 168 stacked
    rows: wide tiles, and balanced wide subgroups beyond 128 rows), prefixes
    of up to 6000 tokens with random fork points, ragged suffixes."""
    rng = np.random.default_rng(5000 + seed)
    D = int(rng.choice([64, 128]))
    Hkv = int(rng.choice([1, 2, 4]))
    G = int(rng.choice([4, 8]))
    w = Workload(name=f"fuzz_large{seed}", n_layers=1, n_q_heads=Hkv * G, n_kv_heads=Hkv, head_dim=D,
                 n_blocks=2048, seed=seed)
    run = Run(w, max_seqs=48, max_decode_branches=48, max_splits=int(rng.choice([4, 16, 32])))
    rids = []
    for g in range(int(rng.integers(1, 3))):
        m = run.create()
        run.append([m], int(rng.integers(200, 6000)), ("p", g))
        n_aux = int(rng.integers(6, 21))
        point = run.ref.seqs[m].length if rng.random() < 0.5 else int(rng.integers(0, run.ref.seqs[m].length + 1))
        kids = run.fork_at(m, point, n_aux)
        for b, r in enumerate([m] + kids):
            s = int(rng.integers(0, 90))
            if s:
                run.append([r], s, ("s", g, b))
        rids += [r for r in [m] + kids if run.ref.seqs[r].length > 0]
    rng.shuffle(rids)
    for step in range(2):
        run.append(rids, 1, ("step", step))
        q, o, lse = run.decode(rids, ("q", step))
        o_ref, l_ref = run.oracle_decode(rids, q, 0)
        compare(o[0], lse[0], o_ref, l_ref, f"seed {seed} step {step}")
    run.pool.sync()
    run.check_tables()
