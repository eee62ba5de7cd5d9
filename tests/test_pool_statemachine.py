"""Property test: the library's block pool (metadata-only, same host code as
a GPU pool) and the reference pool stay bit-identical -- refcounts, free-list
order, every live table and length -- under arbitrary sequences of create,
fork, fork_at, append (single and multi-branch), merge and release, including
the calls that fail for lack of pages or slots."""
import pytest

hyp = pytest.importorskip("hypothesis")
from hypothesis import settings, strategies as st_
from hypothesis.stateful import RuleBasedStateMachine, invariant, precondition, rule

import paper_2608_13667_gb300 as stpkg
from oracle import pool as R

N_BLOCKS, MAX_SEQS = 40, 6


class PoolMachine(RuleBasedStateMachine):
    def __init__(self):
        super().__init__()
        stpkg.build()
        self.lib = stpkg.Pool(n_layers=1, n_q_heads=4, n_kv_heads=1, head_dim=64, n_blocks=N_BLOCKS,
                              seed=11, max_seqs=MAX_SEQS, max_pages=N_BLOCKS, device=None)
        self.ref = R.RefPool(N_BLOCKS, 11, max_seqs=MAX_SEQS)
        self.h = {}

    def _live(self):
        return self.ref.live()

    @rule()
    def create(self):
        try:
            rid = self.ref.create()
        except R.OutOfSlots:
            with pytest.raises(stpkg.STError):
                self.lib.seq_create()
            return
        self.h[rid] = self.lib.seq_create()

    @precondition(lambda self: self._live())
    @rule(data=st_.data(), n=st_.integers(0, 3), at=st_.booleans())
    def fork(self, data, n, at):
        p = data.draw(st_.sampled_from(self._live()))
        cut = data.draw(st_.integers(0, self.ref.seqs[p].length)) if at else self.ref.seqs[p].length
        try:
            kids = self.ref.fork_at(p, cut, n)
        except R.OutOfSlots:
            with pytest.raises(stpkg.STError) as e:
                self.lib.fork_at(self.h[p], cut, n)
            assert e.value.status == stpkg.ST_ERR_OOM
            return
        for k, hh in zip(kids, self.lib.fork_at(self.h[p], cut, n) if n else []):
            self.h[k] = hh

    @precondition(lambda self: self._live())
    @rule(data=st_.data(), n_tok=st_.sampled_from([0, 1, 2, 15, 16, 17, 40]))
    def append(self, data, n_tok):
        ids = data.draw(st_.lists(st_.sampled_from(self._live()), min_size=1, max_size=4, unique=True))
        try:
            self.ref.append(ids, n_tok)
        except R.OutOfBlocks:
            with pytest.raises(stpkg.STError) as e:
                self.lib.append_kv([self.h[i] for i in ids], n_tok, None)
            assert e.value.status == stpkg.ST_ERR_OOM
            return
        self.lib.append_kv([self.h[i] for i in ids], n_tok, None)

    @precondition(lambda self: self._live())
    @rule(data=st_.data(), T=st_.integers(0, 50))
    def merge(self, data, T):
        m = data.draw(st_.sampled_from(self._live()))
        try:
            self.ref.merge(m, T)
        except R.OutOfBlocks:
            with pytest.raises(stpkg.STError):
                self.lib.merge(self.h[m], T, None, None)
            return
        self.lib.merge(self.h[m], T, None, None)

    @precondition(lambda self: self._live())
    @rule(data=st_.data())
    def release(self, data):
        x = data.draw(st_.sampled_from(self._live()))
        self.ref.release(x)
        self.lib.release(self.h[x])

    @invariant()
    def identical(self):
        assert self.lib.refcounts() == self.ref.ref
        assert self.lib.free_list() == list(self.ref.free)
        for rid in self._live():
            t, n = self.lib.block_table(self.h[rid])
            assert t == self.ref.seqs[rid].table and n == self.ref.seqs[rid].length


TestPoolMachine = PoolMachine.TestCase
TestPoolMachine.settings = settings(max_examples=60, stateful_step_count=40, deadline=None)
