"""Seeded synthetic inputs for fork-group attention.

This module holds the shapes of the five agent-shaped workloads and the
seeded generators that draw their Q/K/V values and their length mixes.  It
holds none of the attention or allocator arithmetic: both the CUDA path and
the CPU oracle receive the tensors it produces, and neither imports the other.

Value recipe: K/V (and Q) are float32 N(0,1) draws from a torch generator
seeded per (workload, tag, layer), multiplied by the workload's value scale,
then rounded to bf16 (round-to-nearest-even).  Length mixes come from numpy's
PCG64 generator, which gives the same integers on every platform.
"""
from .configs import CONFIGS, Workload, get  # noqa: F401
from .gen import kv_rows, queries, seed_for, lengths_rng  # noqa: F401
