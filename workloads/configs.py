"""The five fork-group workloads, stated as shapes.

Section 3.3 of the paper forks four auxiliary branches off the main context;
all five share the prefix up to R_t.  Section 4.4 (timing and cost) says the
branch load is dominated by cached-prefix reads.  The paper prints no kernel
shapes, so the shapes below are the synthetic stand-ins for its SWE-Bench Pro
/ Terminal-Bench / tau-bench trajectories (about 23k-token main calls, about
64 branch tokens per turn, harvests of at most 4 x 5 atoms).
"""
from dataclasses import dataclass, field


@dataclass(frozen=True)
class Workload:
    name: str
    n_layers: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    n_blocks: int            # physical pages in the pool (each holds all layers)
    seed: int
    value_scale: float = 1.0  # N(0,1) draws are multiplied by this before bf16 rounding
    page_size: int = 16
    # structure
    n_tasks: int = 1          # independent fork groups
    n_aux: int = 4            # auxiliary branches per group (main is branch 0)
    prefix: tuple = ()        # per-task shared prefix length (filled by lengths())
    suffix: tuple = ()        # per-task tuple of per-branch suffix lengths
    steps: int = 0            # append+decode steps
    turns: int = 1
    merge_tokens: int = 0     # rows appended to main by st_merge each turn
    singletons: int = 0       # unforked decode-only sequences
    singleton_len: int = 0
    # pool capacities used by both the tests and the bench (launch configuration)
    limits: dict = field(default_factory=dict)

    @property
    def group(self):
        return self.n_q_heads // self.n_kv_heads

    @property
    def kv_bytes_per_token_layer(self):
        # K and V, bf16
        return self.n_kv_heads * self.head_dim * 2 * 2


def _tiny():
    return Workload(
        name="tiny_fork_group", n_layers=1, n_q_heads=8, n_kv_heads=2, head_dim=64,
        n_blocks=64, seed=0, value_scale=0.125, n_tasks=1,
        prefix=(512,), suffix=((0, 16, 33, 47, 64),), steps=0,
        limits=dict(max_seqs=8, max_decode_branches=5, max_splits=8, max_pages=64))


def _single_turn():
    return Workload(
        name="single_agent_turn", n_layers=1, n_q_heads=32, n_kv_heads=8, head_dim=128,
        n_blocks=1024, seed=1, n_tasks=1, prefix=(8192,),
        suffix=((256, 256, 256, 256, 256),), steps=256,
        limits=dict(max_seqs=8, max_decode_branches=5, max_splits=32, max_pages=1024))


def _batched():
    import numpy as np
    rng = np.random.default_rng(0)
    P = tuple(int(x) for x in rng.integers(4096, 32768, size=16, endpoint=True))
    S = tuple(tuple(int(x) for x in rng.integers(0, 1024, size=5, endpoint=True)) for _ in range(16))
    # 2 GiB of K+V for one layer: 32768 blocks of 16 tokens x 8 heads x 128 x bf16 x {K,V}
    return Workload(
        name="batched_agent_serving", n_layers=1, n_q_heads=32, n_kv_heads=8, head_dim=128,
        n_blocks=32768, seed=2, n_tasks=16, prefix=P, suffix=S, steps=1,
        limits=dict(max_seqs=96, max_decode_branches=80, max_splits=16, max_pages=2304))


def _long(n_aux=4):
    import numpy as np
    rng = np.random.default_rng(3)
    S = tuple(tuple(int(x) for x in rng.integers(0, 2048, size=n_aux + 1, endpoint=True)) for _ in range(4))
    # room for every suffix plus 256 decode steps per branch
    pages = sum(131072 // 16 + sum((s + 256 + 15) // 16 + 1 for s in row) for row in S)
    name = "long_trajectory_agent" if n_aux == 4 else f"long_trajectory_agent_{n_aux + 1}_branches"
    return Workload(
        name=name, n_layers=32, n_q_heads=64, n_kv_heads=8, head_dim=128, n_aux=n_aux,
        n_blocks=pages + 64, seed=3, n_tasks=4, prefix=(131072,) * 4, suffix=S, steps=1,
        limits=dict(max_seqs=4 * (n_aux + 1) + 4, max_decode_branches=4 * (n_aux + 1), max_splits=32,
                    max_pages=8192 + 160))


def long_with_branches(n_aux: int) -> Workload:
    """The long-trajectory workload with n_aux auxiliary branches per group
    (Section 3.2 lets the branch count vary): 1 + n_aux branches x 8 query
    heads per KV head are stacked on each shared page."""
    return _long(n_aux)


def _cycle():
    # per task: 16384 context; 5 turns x (fork, 512 steps, merge 2048, release)
    per_task = (16384 + 5 * (512 + 2048)) // 16 + 5 * 4 * (512 // 16 + 2) + 8
    singles = 64 * ((2048 + 512) // 16 + 1)
    return Workload(
        name="full_fork_decode_merge_cycle", n_layers=32, n_q_heads=32, n_kv_heads=8,
        head_dim=128, n_blocks=8 * per_task + singles + 256, seed=4, n_tasks=8,
        prefix=(16384,) * 8, suffix=((0, 0, 0, 0, 0),) * 8, steps=512, turns=5,
        merge_tokens=2048, singletons=64, singleton_len=2048,
        limits=dict(max_seqs=112, max_decode_branches=104, max_splits=16, max_pages=2048))


CONFIGS = {
    1: _tiny,
    2: _single_turn,
    3: _batched,
    4: _long,
    5: _cycle,
}


def get(i: int) -> Workload:
    return CONFIGS[i]()
