"""Device harvest against the reference harvest (bit-exact), and a full turn
in which the harvested count drives st_merge (Section 3.5)."""
import numpy as np
import pytest
import torch

import paper_2608_13667_gb300 as stpkg
from fg_harness import Run, compare
from oracle import attention as A
from oracle.harvest import harvest
from workloads import Workload

pytestmark = pytest.mark.gpu

OPEN, CLOSE = 7, 8


def _streams(rng, n_br, stride, p_open=0.06, p_close=0.08):
    s = rng.integers(100, 5000, size=(n_br, stride)).astype(np.int32)
    r = rng.random((n_br, stride))
    s[r < p_open] = OPEN
    s[(r >= p_open) & (r < p_open + p_close)] = CLOSE
    lens = rng.integers(0, stride + 1, size=n_br).astype(np.int32)
    return s, lens


def _device(s, lens):
    return torch.from_numpy(s).cuda(), torch.from_numpy(lens).cuda()


@pytest.mark.parametrize("seed,n_br,stride,cap", [(0, 4, 512, 5), (1, 4, 64, 5), (2, 1, 300, 5), (3, 8, 200, 3),
                                                  (4, 32, 33, 64), (5, 4, 512, 0)])
def test_harvest_matches_reference(stlib, seed, n_br, stride, cap):
    rng = np.random.default_rng(seed)
    s, lens = _streams(rng, n_br, stride)
    ids, src, atoms = stpkg.st_harvest(*_device(s, lens), OPEN, CLOSE, cap)
    ref_ids, ref_src, ref_atoms = harvest([list(s[b, :lens[b]]) for b in range(n_br)], OPEN, CLOSE, cap)
    assert ids.cpu().tolist() == ref_ids
    assert src.cpu().tolist() == [b * stride + p for b, p in ref_src]
    assert atoms.cpu().tolist() == ref_atoms


def test_harvest_of_nothing_is_empty(stlib):
    s = np.full((4, 16), 123, dtype=np.int32)
    s[1, 3] = OPEN                                     # an unfinished unit only
    ids, src, atoms = stpkg.st_harvest(*_device(s, np.full(4, 16, np.int32)), OPEN, CLOSE)
    assert ids.numel() == 0 and atoms.cpu().tolist() == [0, 0, 0, 0]


def test_turn_fork_decode_harvest_merge(stlib):
    """fork 4 -> branches decode 40 steps generating token ids -> harvest ->
    merge the harvested rows into main -> main's next decode sees them."""
    w = Workload(name="turn", n_layers=2, n_q_heads=32, n_kv_heads=8, head_dim=128, n_blocks=512, seed=31)
    run = Run(w, max_seqs=8, max_decode_branches=8, max_splits=8)
    m = run.create()
    run.append([m], 700, ("prefix",))
    aux = run.fork(m, 4)
    rng = np.random.default_rng(9)
    steps = 40
    toks = np.zeros((4, steps), dtype=np.int32)
    for step in range(steps):
        run.append([m] + aux, 1, ("step", step))
        run.decode([m] + aux, ("q", step))
        # stand-in for sampling: branch tokens follow a fixed atom pattern with noise
        for b in range(4):
            toks[b, step] = OPEN if step % 9 == b else (CLOSE if step % 9 == b + 4 else rng.integers(100, 900))
    ids, src, atoms = stpkg.st_harvest(*_device(toks, np.full(4, steps, np.int32)), OPEN, CLOSE, 5)
    ref_ids, _, ref_atoms = harvest([list(toks[b]) for b in range(4)], OPEN, CLOSE, 5)
    assert ids.cpu().tolist() == ref_ids and atoms.cpu().tolist() == ref_atoms
    T = ids.numel()
    assert T > 0
    for a in aux:                                      # cancel the branches
        run.release(a)
    qm, om, lm, L0 = run.merge(m, T, ("merge",))       # thought rows appended after main's context
    for layer in range(w.n_layers):
        k, v = run.context(m, layer)
        o_ref, l_ref = A.merge_prefill(qm[layer].cpu(), k, v, L0)
        compare(om[layer], lm[layer], o_ref, l_ref, f"merge layer {layer}")
    run.pool.sync()
    run.check_tables()
