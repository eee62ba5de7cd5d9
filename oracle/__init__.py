"""CPU oracle for fork-group attention -- TEST INFRASTRUCTURE ONLY.

Plain, slow, obviously-correct restatements of what the hot path computes:

* ``oracle.pool``       -- the paged block pool's allocation rules (fork = copy
  the block table and take a reference on every page; append with
  copy-on-write; release = drop references, freed pages go to the tail of a
  FIFO).  Integer results, compared bit-exactly.
* ``oracle.attention``  -- softmax attention of each branch's query over its
  materialised context (prefix ++ suffix) in float64; the merge prefill as a
  per-row loop over the causal prefix; the log-sum-exp combine of partials.

The paper (Second Thought, Sections 3.2-3.5) states the method at the level
of text buffers and a serving API; the attention-level reading it implies is:
branches share the KV of the snapshot H_t + R_t (Section 3.3), each decodes
over that prefix plus its own tokens, and the merge appends the harvested
thoughts after the existing context where the next turn reads them in order
(Section 3.5).  Sharing the prefix and splitting the softmax by log-sum-exp
are exact reorderings, so the oracle computes the unshared, unsplit
definition.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import this package.  The
CUDA library never links, loads or calls it, and this package imports
nothing from the CUDA side.
"""
