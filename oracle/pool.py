"""Reference block pool: the allocation rules, one Python operation at a time.

Test infrastructure only (see the package docstring).

The paper (Section 3.3) only says that all branches reuse the prefix KV of
the snapshot H_t + R_t; it fixes no allocator.  The rules below are this
project's reading, and the CUDA library must reproduce them bit-exactly:

* The free list is a FIFO.  It starts as a Fisher-Yates shuffle of
  [0, n_blocks) driven by splitmix64(seed) (Steele, Lea & Flood 2014;
  S. Vigna's public-domain reference code): for i = n-1 down to 1, take
  j = next() mod (i+1) and swap entries i and j.  Allocation pops the head.
* Append places each new row at logical slot len: a fresh page when
  len % page == 0; otherwise, if the last page is shared (refcount > 1), it
  is first copied (copy-on-write): allocate a page, copy rows [0, len % page)
  for every layer, drop one reference on the old page, point the table entry
  at the copy.  A page with refcount 1 is written in place.
* Fork copies the parent's table and takes one reference on every entry; it
  allocates no page.  It fails without any change if fewer than n_aux
  sequence slots are free.  A fork at an earlier point (Table 2's "w/o R_t"
  and "fork onset": the branches see only the first `length` rows of the
  parent) copies the first ceil(length / page) entries; the child's last page
  may then hold parent rows past the child's length, which the child's first
  append copies away like any shared partial page.
* Release drops one reference per table entry in logical order; pages that
  reach zero are pushed to the FIFO tail in that order.
* A multi-branch append processes branches in the order given; it fails
  without any change if the pool lacks the pages the whole call needs.
* Merge (Section 3.5: thoughts appended after the existing context) is an
  append of the thought rows to the main sequence.
"""
from collections import deque

MASK64 = (1 << 64) - 1


class OutOfBlocks(Exception):
    pass


class OutOfSlots(Exception):
    pass


def splitmix64(seed):
    """Generator of splitmix64 outputs (Vigna's reference algorithm)."""
    state = seed & MASK64
    while True:
        state = (state + 0x9E3779B97F4A7C15) & MASK64
        z = state
        z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
        z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
        yield z ^ (z >> 31)


def initial_free_list(n_blocks, seed):
    order = list(range(n_blocks))
    gen = splitmix64(seed)
    for i in range(n_blocks - 1, 0, -1):
        j = next(gen) % (i + 1)
        order[i], order[j] = order[j], order[i]
    return order


class Seq:
    __slots__ = ("table", "length", "alive")

    def __init__(self):
        self.table = []
        self.length = 0
        self.alive = True


class RefPool:
    """The allocator state: free FIFO, per-page refcounts, per-sequence tables.

    ``content`` optionally tracks, per physical (page, row), a label of the
    row stored there, so tests can read a sequence back through its table.
    Operations return the copy-on-write events they caused as
    (old_page, new_page, rows_copied) tuples.
    """

    def __init__(self, n_blocks, seed, page_size=16, max_seqs=1 << 30, track_content=False):
        self.n_blocks = n_blocks
        self.page = page_size
        self.free = deque(initial_free_list(n_blocks, seed))
        self.ref = [0] * n_blocks
        self.seqs = []
        self.max_seqs = max_seqs
        self.content = [[None] * page_size for _ in range(n_blocks)] if track_content else None

    # -- helpers --------------------------------------------------------
    def live(self):
        return [i for i, s in enumerate(self.seqs) if s.alive]

    def _pop(self):
        b = self.free.popleft()
        assert self.ref[b] == 0
        self.ref[b] = 1
        return b

    def _pages_needed(self, s, n_tok):
        """Pages an append of n_tok rows to s takes from the free list."""
        if n_tok == 0:
            return 0
        p = self.page
        need = -(-(s.length + n_tok) // p) - (-(-s.length // p))
        if s.length % p != 0 and self.ref[s.table[-1]] > 1:
            need += 1  # copy-on-write of the shared partial page
        return need

    # -- operations -----------------------------------------------------
    def create(self):
        if len(self.live()) >= self.max_seqs:
            raise OutOfSlots()
        self.seqs.append(Seq())
        return len(self.seqs) - 1

    def fork(self, parent, n_aux):
        src = self.seqs[parent]
        assert src.alive
        if len(self.live()) + n_aux > self.max_seqs:
            raise OutOfSlots()
        out = []
        for _ in range(n_aux):
            s = Seq()
            s.table = list(src.table)
            s.length = src.length
            for b in s.table:
                self.ref[b] += 1
            self.seqs.append(s)
            out.append(len(self.seqs) - 1)
        return out

    def fork_at(self, parent, length, n_aux):
        src = self.seqs[parent]
        assert src.alive and 0 <= length <= src.length
        if len(self.live()) + n_aux > self.max_seqs:
            raise OutOfSlots()
        out = []
        n_pages = -(-length // self.page)
        for _ in range(n_aux):
            s = Seq()
            s.table = list(src.table[:n_pages])
            s.length = length
            for b in s.table:
                self.ref[b] += 1
            self.seqs.append(s)
            out.append(len(self.seqs) - 1)
        return out

    def append(self, seq_ids, n_tok, labels=None):
        """Append n_tok rows to each sequence in ``seq_ids`` (in that order).

        ``labels[i][t]`` is stored as the content of row t of sequence i when
        content tracking is on.
        """
        return self.prefill_batch(seq_ids, [n_tok] * len(seq_ids), labels)

    def prefill_batch(self, seq_ids, counts, labels=None):
        """Append counts[i] rows to sequence seq_ids[i], the sequences taken in
        order: the bookkeeping of a batched prefill, in which several agents'
        observation (Section 3.1) and thought (Section 3.5) rows arrive
        together.  All or nothing."""
        assert len(set(seq_ids)) == len(seq_ids), "a sequence may appear once per call"
        assert len(counts) == len(seq_ids) and all(n >= 0 for n in counts)
        seqs = [self.seqs[i] for i in seq_ids]
        assert all(s.alive for s in seqs)
        # all-or-nothing: the whole call's page need is checked first
        if sum(self._pages_needed(s, n) for s, n in zip(seqs, counts)) > len(self.free):
            raise OutOfBlocks()
        events = []
        p = self.page
        for idx, i in enumerate(seq_ids):
            s = self.seqs[i]
            for t in range(counts[idx]):
                off = s.length % p
                if off == 0:
                    s.table.append(self._pop())
                elif self.ref[s.table[-1]] > 1:
                    old = s.table[-1]
                    new = self._pop()
                    if self.content is not None:
                        self.content[new][:off] = self.content[old][:off]
                    self.ref[old] -= 1
                    s.table[-1] = new
                    events.append((old, new, off))
                if self.content is not None:
                    self.content[s.table[-1]][off] = None if labels is None else labels[idx][t]
                s.length += 1
        return events

    def merge(self, main, n_tok, labels=None):
        return self.append([main], n_tok, None if labels is None else [labels])

    def release(self, seq_id):
        s = self.seqs[seq_id]
        assert s.alive
        for b in s.table:
            self.ref[b] -= 1
            assert self.ref[b] >= 0
            if self.ref[b] == 0:
                self.free.append(b)
        s.alive = False
        s.table = []
        s.length = 0

    def read(self, seq_id):
        """Row labels of a sequence read through its block table."""
        s = self.seqs[seq_id]
        return [self.content[s.table[j // self.page]][j % self.page] for j in range(s.length)]
