"""Fork-group decode benchmark: branch-steps/s and achieved HBM bandwidth.

Workload (default): the long-trajectory agent -- 4 independent fork groups,
each a 131072-token shared prefix with 1 main + 4 auxiliary branches holding
suffixes of up to 2048 tokens; 64 query / 8 KV heads, head_dim 128, 32
layers, bf16 KV, fp32 outputs.  One step = every branch appends one KV row
(all layers) and decodes one query (all layers): 20 branch-steps, about
71 GB of algorithmic KV reads, well beyond the 129 MB L2.

Multi-GPU: fork groups are independent, so N ranks run N replicas with no
data-path collective (weak scaling); the timing takes the max over ranks.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
"""
import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "fork-group decode branch-steps/s and achieved HBM GB/s vs GB300 peak (1 GPU)"
UNIT = "branch-steps/s"
PREFIX_CHUNK = 8192


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except OSError:
        return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}, "fallback"


def _dist(backend=None):
    """(rank, world, local rank).  One process per GPU under torchrun; NCCL on
    GPUs, gloo when asked (the CPU tests of the multi-rank path)."""
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    if ws <= 1:
        return 0, 1, 0
    import torch
    import torch.distributed as dist
    rank = int(os.environ["RANK"])
    local = int(os.environ.get("LOCAL_RANK", rank))
    backend = backend or ("nccl" if torch.cuda.is_available() else "gloo")
    if backend == "nccl":
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        dist.init_process_group("gloo")
    return rank, ws, local


def _allreduce_max(x, ws):
    """Max of a float over ranks (timings: the slowest rank sets the time)."""
    if ws <= 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons during the timed region."""
    FIELDS = ["clocks.sm", "clocks.max.sm", "power.draw", "clocks_event_reasons.hw_slowdown",
              "clocks_event_reasons.hw_thermal_slowdown", "clocks_event_reasons.sw_thermal_slowdown",
              "clocks_event_reasons.sw_power_cap"]

    def __init__(self, gpu):
        self.gpu = gpu
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), "--query-gpu=" + ",".join(self.FIELDS),
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
        except OSError:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.thread.join(timeout=2)
        sm, smax, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) != len(self.FIELDS):
                continue
            try:
                sm.append(float(parts[0]))
                smax = float(parts[1])
            except ValueError:
                continue
            for n, v in zip(names, parts[3:]):
                if v.lower() == "active":
                    reasons.add(n)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": smax,
                "reasons": sorted(reasons), "samples": len(sm)}


def _code_only(src):
    """C++ source without comments and whitespace (a comment edit is not a
    kernel change)."""
    import re
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", " ", src)
    return re.sub(r"\s+", "", src)


def _kernel_hash():
    h = hashlib.sha256()
    for f in ("attend_tc.cu", "ptx.cuh", "kernels.cuh"):
        with open(os.path.join(ROOT, "paper_2608_13667_gb300", "csrc", f)) as fh:
            h.update(_code_only(fh.read()).encode())
    return h.hexdigest()[:16]


def _ncu_traffic(kernel, workload):
    """dram bytes per launch from the committed ncu summary, if it was taken
    on the current kernel source and on this workload."""
    try:
        with open(os.path.join(ROOT, "profiles", "ncu_traffic.json")) as f:
            d = json.load(f)
    except OSError:
        return None
    e = d.get(kernel)
    if not e or e.get("source_hash") != _kernel_hash() or e.get("workload") != workload:
        return None
    return e.get("dram_bytes_per_launch")


# --------------------------------------------------------------------------- ours

def build_long_workload(w, dev, step_rows=0):
    """The workload's fork groups at full size in a pool with room for
    step_rows more rows per branch; returns (pool, branch handles)."""
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import kv_rows
    n_br = w.n_tasks * (w.n_aux + 1)
    extra = -(-step_rows // 16) + 1  # pages a branch may take for the steps
    limits = dict(w.limits)
    if step_rows:
        longest = max(p + max(s) for p, s in zip(w.prefix, w.suffix))
        limits["max_pages"] = max(limits.get("max_pages", 0), -(-longest // 16) + extra)
    pool = st.Pool(n_layers=w.n_layers, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads,
                   head_dim=w.head_dim, n_blocks=w.n_blocks + (n_br * extra if step_rows else 0), seed=w.seed,
                   device=dev, **limits)
    shape = lambda n: (w.n_layers, 1, n, w.n_kv_heads, w.head_dim)
    branches = []
    for t in range(w.n_tasks):
        m = pool.seq_create()
        for c0 in range(0, w.prefix[t], PREFIX_CHUNK):
            n = min(PREFIX_CHUNK, w.prefix[t] - c0)
            k, v = kv_rows(w, ("prefix", t, c0), n, device=dev)
            pool.append_kv([m], k.view(shape(n)), v.view(shape(n)))
            del k, v
        br = [m] + pool.fork(m, w.n_aux)
        for b, (h, s) in enumerate(zip(br, w.suffix[t])):
            if s:
                k, v = kv_rows(w, ("suffix", t, b), s, device=dev)
                pool.append_kv([h], k.view(shape(s)), v.view(shape(s)))
        branches += br
    torch.cuda.synchronize(dev)
    return pool, branches


def _workload(args):
    """The bench workload: config N, or the long-trajectory one with another
    branch count (--n-aux)."""
    from workloads import get
    from workloads.configs import long_with_branches
    if args.n_aux is None:
        return get(args.config)
    if args.config != 4:
        raise SystemExit("--n-aux applies to config 4 (long trajectory)")
    return long_with_branches(args.n_aux)


L2_BYTES = 126.5 * 2**20  # GB300 L2


def _l2_note(step_bytes):
    """How a step's working set relates to L2 (the timing rule: inputs larger
    than L2, or a flush between timed steps)."""
    if step_bytes > 4 * L2_BYTES:
        return f"inputs larger than L2 (~{step_bytes / 1e9:.1f} GB of KV per step)"
    return (f"KV of one step (~{step_bytes / 1e6:.0f} MB) fits in L2 and stays resident across steps, not "
            "flushed: a latency-bound configuration, reported as a latency, not as a roofline")


def run_ours(args, rank, ws, local):
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import kv_rows, queries
    w = _workload(args)
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    st.build()
    # rows each branch takes: warm-up and timed steps, the end-to-end run (at
    # most 12) and the latency record's two loops (5 + steps each)
    pool, br = build_long_workload(w, dev, step_rows=args.warmup + 3 * args.steps + 32)
    n_br = len(br)
    n_steps = args.warmup + args.steps
    # per-step inputs, resident in HBM before the timed region
    step_k, step_v, step_q = [], [], []
    for s in range(n_steps):
        k, v = kv_rows(w, ("step", s, rank), n_br, device=dev)
        step_k.append(k.view(w.n_layers, n_br, 1, w.n_kv_heads, w.head_dim))
        step_v.append(v.view(w.n_layers, n_br, 1, w.n_kv_heads, w.head_dim))
        step_q.append(queries(w, ("q", s, rank), n_br, device=dev))
    o = torch.empty((w.n_layers, n_br, w.n_q_heads, w.head_dim), dtype=torch.float32, device=dev)
    lse = torch.empty((w.n_layers, n_br, w.n_q_heads), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)

    def step(s):
        pool.append_kv(br, step_k[s], step_v[s])
        pool.decode_attn(br, step_q[s], o, lse)

    for s in range(args.warmup):
        step(s)
    pool.sync()
    pool.profile_read()  # drop warm-up counts
    pool.profile_enable(True)
    clocks = ClockSampler(local)
    _barrier(ws)
    torch.cuda.synchronize(dev)
    clocks.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for s in range(args.warmup, n_steps):
        step(s)
    e1.record(stream)
    torch.cuda.synchronize(dev)
    clk = clocks.stop()
    _barrier(ws)
    ms = e0.elapsed_time(e1)
    pool.sync()
    stats = pool.profile_read()
    pool.profile_enable(False)
    ms_max = _allreduce_max(ms, ws)

    # end-to-end through the public API with host buffers: H2D of the step's
    # q and new K/V rows from pinned memory, D2H of O and LSE, every step.  As
    # a serving loop would, the copies run on their own streams, double
    # buffered: step s+1's inputs go up and step s-1's outputs come down while
    # step s computes (events order each buffer's reuse).
    e2e_steps = max(2, min(args.steps, 10))
    e2e_warm = 2  # first use of the pinned buffers stays out of the timing
    n_host = min(e2e_steps, 4)  # distinct host input sets, used in turn
    hq = [step_q[s % n_steps].cpu().pin_memory() for s in range(n_host)]
    hk = [step_k[s % n_steps].cpu().pin_memory() for s in range(n_host)]
    hv = [step_v[s % n_steps].cpu().pin_memory() for s in range(n_host)]
    ho = [torch.empty(o.shape, dtype=o.dtype).pin_memory() for _ in range(2)]
    hl = [torch.empty(lse.shape, dtype=lse.dtype).pin_memory() for _ in range(2)]
    dq = [torch.empty_like(step_q[0]) for _ in range(2)]
    dk = [torch.empty_like(step_k[0]) for _ in range(2)]
    dv = [torch.empty_like(step_v[0]) for _ in range(2)]
    do = [o, torch.empty_like(o)]
    dl = [lse, torch.empty_like(lse)]
    up, down = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev = lambda: torch.cuda.Event()
    in_ready, in_free = [ev(), ev()], [ev(), ev()]
    out_ready, out_free = [ev(), ev()], [ev(), ev()]
    for b in range(2):  # all buffers free at the start
        in_free[b].record(stream)
        out_free[b].record(stream)

    def h2d(s):
        b = s % 2
        with torch.cuda.stream(up):
            up.wait_event(in_free[b])
            dq[b].copy_(hq[s % n_host], non_blocking=True)
            dk[b].copy_(hk[s % n_host], non_blocking=True)
            dv[b].copy_(hv[s % n_host], non_blocking=True)
            in_ready[b].record(up)

    def compute_and_d2h(s):
        b = s % 2
        stream.wait_event(in_ready[b])
        stream.wait_event(out_free[b])
        pool.append_kv(br, dk[b], dv[b])
        pool.decode_attn(br, dq[b], do[b], dl[b])
        in_free[b].record(stream)
        out_ready[b].record(stream)
        with torch.cuda.stream(down):
            down.wait_event(out_ready[b])
            ho[b].copy_(do[b], non_blocking=True)
            hl[b].copy_(dl[b], non_blocking=True)
            out_free[b].record(down)

    def e2e_run(n):
        h2d(0)
        for s in range(n):
            if s + 1 < n:
                h2d(s + 1)
            compute_and_d2h(s)
        torch.cuda.synchronize(dev)

    e2e_run(e2e_warm)
    _barrier(ws)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    e2e_run(e2e_steps)
    e2e_s = _allreduce_max(time.perf_counter() - t0, ws)
    h2d_bytes = hq[0].numel() * 2 + hk[0].numel() * 2 * 2
    d2h_bytes = ho[0].numel() * 4 + hl[0].numel() * 4

    res = {}
    if rank == 0:
        peaks, src = _peaks()
        dec = stats["decode_partial"]
        launches = sum(v["kernels"] for v in stats.values())  # device kernels, not calls
        avg_ms = dec["total_ms"] / max(1, dec["launches"])
        bytes_per_launch = dec["bytes"] / max(1, dec["launches"])
        achieved = bytes_per_launch / (avg_ms * 1e-3) / 1e9
        step_bytes = sum(v["bytes"] for v in stats.values()) / args.steps
        value = ws * n_br * args.steps / (ms_max * 1e-3)
        res = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms_max / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": w.name, "tasks": w.n_tasks, "branches_per_task": w.n_aux + 1,
                       "prefix_tokens": w.prefix[0], "suffix_tokens": [list(s) for s in w.suffix],
                       "layers": w.n_layers, "q_heads": w.n_q_heads, "kv_heads": w.n_kv_heads,
                       "head_dim": w.head_dim, "step": "append 1 KV row + decode, every branch, all layers",
                       "l2": _l2_note(step_bytes),
                       "parallelism": f"replicas x{ws}"},
            "hbm_gbs_step": step_bytes / (ms_max / args.steps * 1e-3) / 1e9,
            "roofline": {"kernel": "decode_partial", "bound": "hbm", "achieved": achieved,
                         "peak": peaks["hbm_gbs"], "peak_source": src, "unit": "GB/s",
                         "frac": achieved / peaks["hbm_gbs"], "frac_of_nominal_8tbs": achieved / 8000.0,
                         "bytes_per_launch": bytes_per_launch, "avg_launch_ms": avg_ms,
                         "traffic": _ncu_traffic("decode_partial", w.name)},
            "kernels": {k: {"launches": v["launches"], "device_kernels": v["kernels"], "ms": v["total_ms"]}
                        for k, v in stats.items() if v["launches"]},
            "gpu_launches": launches,
            "clocks": clk,
            "e2e": {"value": ws * n_br * e2e_steps / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d_bytes,
                    "d2h_bytes_per_step": d2h_bytes,
                    "copies": "pinned host buffers, H2D and D2H on their own streams, double-buffered, "
                              "overlapping the neighbouring steps' compute"},
        }
        if step_bytes < 0.5 * L2_BYTES:
            res["latency"] = _c_abi_latency(pool, br, step_k, step_v, step_q, o, lse, args.steps, dev)
    pool.close()
    if rank == 0:
        # the tensor-bound half of the path: the merge prefill, timed alone on a
        # fixed case in the same run
        mg = _merge_case(3, dev)
        peaks, src = _peaks()
        res["merge"] = {
            "kernel": "merge_prefill", "workload": MERGE_CASE,
            "ms": mg["merge_ms"], "launches": mg["merge_launches"],
            "roofline": {"bound": "tensor", "achieved": mg["merge_tflops"], "peak": peaks["bf16_tflops"],
                         "peak_source": src + " (bf16 burst: the kernel is timed alone)", "unit": "TFLOP/s",
                         "frac": mg["merge_tflops"] / peaks["bf16_tflops"],
                         "flops": "algorithmic: 4 D x causal keys x q heads x layers; P V runs for both bf16 "
                                  "terms of P, so the tensor cores execute 1.5x this"}}
    return res


def _c_abi_latency(pool, br, step_k, step_v, step_q, o, lse, n, dev):
    """A step of the latency case (a working set that stays in L2) timed through
    the C ABI alone, with arguments marshalled once and no per-kernel events:
    st_decode_step (one row appended per branch and the decode, the row
    written by the decode kernel), and st_append_kv then st_decode_attn.
    Returns microseconds per step for both."""
    import ctypes
    import torch
    import paper_2608_13667_gb300 as st
    L = st.lib()
    h = pool._h
    arr, n_br = st._seq_array(br)
    sp = pool._stream(None)
    vp = lambda t: ctypes.c_void_p(t.data_ptr())
    ks, vs, qs = [vp(t) for t in step_k], [vp(t) for t in step_v], [vp(t) for t in step_q]
    op, lp = vp(o), vp(lse)
    m = len(ks)

    def fused(s):
        return L.st_decode_step(h, arr, n_br, ks[s % m], vs[s % m], qs[s % m], op, lp, sp)

    def separate(s):
        return L.st_append_kv(h, arr, n_br, 1, ks[s % m], vs[s % m], sp) or \
            L.st_decode_attn(h, arr, n_br, qs[s % m], op, lp, sp)

    stream = torch.cuda.current_stream(dev)
    out = {}
    for name, call in (("st_decode_step", fused), ("st_append_kv + st_decode_attn", separate)):
        for s in range(5):
            if call(s):
                raise RuntimeError(L.st_last_error(h).decode())
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        t0 = time.perf_counter()
        e0.record(stream)
        for s in range(n):
            if call(s):
                raise RuntimeError(L.st_last_error(h).decode())
        e1.record(stream)
        torch.cuda.synchronize(dev)
        out[name] = {"us_per_step": e0.elapsed_time(e1) * 1e3 / n,
                     "host_us_per_step": (time.perf_counter() - t0) * 1e6 / n}
    pool.sync()
    return {"us_per_step": out["st_decode_step"]["us_per_step"], "steps": n, "calls": out,
            "how": "one row appended to every branch and the decode, per step, called from a ctypes loop with "
                   "arguments marshalled once and no per-kernel events; the step's pages stay in L2"}


# --------------------------------------------------------------------------- profiling case

def run_profile_small():
    """A small case of both attention paths for ncu captures: the long-trajectory
    decode with 4 layers (8.9 GB of KV per launch, beyond L2; three decode steps)
    and one merge of 2048 thought rows onto a 16896-token main context (32 q /
    8 kv heads, 4 layers).  Prints CUDA-event timings of the last decode and the
    merge."""
    import dataclasses
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import get, kv_rows, queries
    dev = torch.device("cuda", 0)
    st.build()
    w = dataclasses.replace(get(4), n_layers=4)
    pool, br = build_long_workload(w, dev)
    n = len(br)
    o = torch.empty((w.n_layers, n, w.n_q_heads, w.head_dim), dtype=torch.float32, device=dev)
    lse = torch.empty((w.n_layers, n, w.n_q_heads), dtype=torch.float32, device=dev)
    pool.profile_enable(True)
    for s in range(3):
        k, v = kv_rows(w, ("step", s), n, device=dev)
        shape = (w.n_layers, n, 1, w.n_kv_heads, w.head_dim)
        pool.append_kv(br, k.view(shape), v.view(shape))
        pool.decode_attn(br, queries(w, ("q", s), n, device=dev), o, lse)
    pool.sync()
    d = pool.profile_read()["decode_partial"]
    pool.close()
    del pool
    mg = _merge_case()
    print(json.dumps({"decode_ms_per_launch": d["total_ms"] / d["launches"],
                      "decode_gbs": d["bytes"] / d["total_ms"] / 1e6, **mg}))


MERGE_CASE = ("2048 thought rows merged onto a 16896-token main context (the full cycle's first merge), "
              "32 q / 8 kv heads, D 128, 4 layers")


def _merge_case(n_merges=3, dev=None):
    """Merges of 2048 thought rows onto a 16896-token main context (32 q / 8 kv
    heads, D 128, 4 layers): main is forked n_merges times and each fork takes
    one merge, so every launch does the same work.  Returns the CUDA-event
    timing of the fastest launch."""
    import dataclasses
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import get, kv_rows, queries
    dev = dev or torch.device("cuda", 0)
    st.build()
    w5 = dataclasses.replace(get(5), n_layers=4)
    p5 = st.Pool(n_layers=4, n_q_heads=w5.n_q_heads, n_kv_heads=w5.n_kv_heads, head_dim=w5.head_dim,
                 n_blocks=4096, seed=1, device=dev, max_seqs=8, max_pages=2048, max_decode_branches=8,
                 max_splits=16)
    m = p5.seq_create()
    for c0 in range(0, 16896, 8448):
        k, v = kv_rows(w5, ("ctx", c0), 8448, device=dev)
        p5.append_kv([m], k.view(4, 1, 8448, 8, 128), v.view(4, 1, 8448, 8, 128))
    forks = p5.fork(m, n_merges)
    k, v = kv_rows(w5, ("merge",), 2048, device=dev)
    q = queries(w5, ("mq",), 2048, device=dev)
    best = None
    for f in forks:
        p5.profile_enable(True)
        p5.merge(f, q, k, v)
        p5.sync()
        mg = p5.profile_read()["merge_prefill"]
        p5.profile_enable(False)
        if best is None or mg["total_ms"] < best["total_ms"]:
            best = mg
    p5.close()
    return {"merge_ms": best["total_ms"], "merge_tflops": best["flops"] / best["total_ms"] / 1e9,
            "merges": n_merges, "merge_launches": n_merges}


def run_profile_wide(n_aux=None):
    """The wide decode tile on a small case for ncu captures: the long-trajectory
    decode with 9 branches per group (72 stacked rows; another count with
    --n-aux, e.g. 16 for the paired tile's 136 rows) and 4 layers instead of
    32, three decode steps.  Prints the CUDA-event timing of the last one."""
    import dataclasses
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import kv_rows, queries
    from workloads.configs import long_with_branches
    dev = torch.device("cuda", 0)
    st.build()
    w = dataclasses.replace(long_with_branches(8 if n_aux is None else n_aux), n_layers=4)
    pool, br = build_long_workload(w, dev)
    n = len(br)
    o = torch.empty((w.n_layers, n, w.n_q_heads, w.head_dim), dtype=torch.float32, device=dev)
    lse = torch.empty((w.n_layers, n, w.n_q_heads), dtype=torch.float32, device=dev)
    for s in range(3):
        k, v = kv_rows(w, ("step", s), n, device=dev)
        shape = (w.n_layers, n, 1, w.n_kv_heads, w.head_dim)
        pool.append_kv(br, k.view(shape), v.view(shape))
        if s == 2:  # time the last step alone
            pool.sync()
            pool.profile_read()
            pool.profile_enable(True)
        pool.decode_attn(br, queries(w, ("q", s), n, device=dev), o, lse)
    pool.sync()
    d = pool.profile_read()["decode_partial"]
    pool.close()
    print(json.dumps({"workload": w.name, "layers": w.n_layers, "decode_ms": d["total_ms"] / d["launches"],
                      "decode_gbs": d["bytes"] / d["total_ms"] / 1e6}))


def run_turn():
    """One agent turn at the paper's shape, phase by phase: a main context of
    23040 tokens (32 layers, 32 q / 8 kv heads, D 128); fork 4 auxiliary
    branches; 64 steps in which main and branches append one row and decode
    (about the paper's branch tokens per turn); harvest the branches' token
    streams (synthetic ids with thought tags) on the device; merge the
    harvested rows into main; release the branches.  Three turns (the context
    grows by each merge); prints the phases of the last two."""
    import numpy as np
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import Workload, kv_rows, queries
    dev = torch.device("cuda", 0)
    st.build()
    w = Workload(name="agent_turn", n_layers=32, n_q_heads=32, n_kv_heads=8, head_dim=128, n_blocks=2048, seed=6)
    L, Hkv, D, n_aux, steps, ctx = w.n_layers, w.n_kv_heads, w.head_dim, 4, 64, 23040
    pool = st.Pool(n_layers=L, n_q_heads=w.n_q_heads, n_kv_heads=Hkv, head_dim=D, n_blocks=w.n_blocks,
                   seed=w.seed, device=dev, max_seqs=16, max_decode_branches=8, max_splits=32, max_pages=2048)
    main = pool.seq_create()
    for c0 in range(0, ctx, PREFIX_CHUNK):
        n = min(PREFIX_CHUNK, ctx - c0)
        k, v = kv_rows(w, ("ctx", c0), n, device=dev)
        pool.append_kv([main], k.view(L, 1, n, Hkv, D), v.view(L, 1, n, Hkv, D))
    nb = n_aux + 1
    sk, sv = kv_rows(w, ("step",), nb, device=dev)
    sk, sv = sk.view(L, nb, 1, Hkv, D), sv.view(L, nb, 1, Hkv, D)
    sq = queries(w, ("q",), nb, device=dev)
    o = torch.empty((L, nb, w.n_q_heads, D), dtype=torch.float32, device=dev)
    lse = torch.empty((L, nb, w.n_q_heads), dtype=torch.float32, device=dev)
    t_max = n_aux * steps
    mk, mv = kv_rows(w, ("merge",), t_max, device=dev)
    mq = queries(w, ("mq",), t_max, device=dev)
    rng = np.random.default_rng(6)   # the branches' generated ids: thought tags 7 / 8 among other ids
    s = rng.integers(100, 5000, size=(n_aux, steps)).astype(np.int32)
    r = rng.random((n_aux, steps))
    s[r < 0.06] = 7
    s[(r >= 0.06) & (r < 0.14)] = 8
    ds = torch.from_numpy(s).to(dev)
    dl = torch.full((n_aux,), steps, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)
    ev = lambda: torch.cuda.Event(enable_timing=True)
    turns = []
    for turn in range(3):
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        br = [main] + pool.fork(main, n_aux)
        t1 = time.perf_counter()
        e0, e1 = ev(), ev()
        e0.record(stream)
        for _ in range(steps):
            pool.append_kv(br, sk, sv)
            pool.decode_attn(br, sq, o, lse)
        e1.record(stream)
        torch.cuda.synchronize(dev)   # the observation arrives: the branches stop here
        th0 = time.perf_counter()
        ids, src, atoms = st.st_harvest(ds, dl, 7, 8, 5)   # reads the count back: the host sizes the merge
        T = int(ids.numel())
        th1 = time.perf_counter()
        qT, kT, vT = (x[:, :T].contiguous() for x in (mq, mk, mv))   # the thought rows' Q/K/V
        oT = torch.empty((L, T, w.n_q_heads, D), dtype=torch.float32, device=dev)
        lT = torch.empty((L, T, w.n_q_heads), dtype=torch.float32, device=dev)
        e2, e3 = ev(), ev()
        e2.record(stream)
        if T:
            pool.merge(main, qT, kT, vT, oT, lT)
        e3.record(stream)
        torch.cuda.synchronize(dev)
        t2 = time.perf_counter()
        for b in br[1:]:
            pool.release(b)
        t3 = time.perf_counter()
        turns.append({"context_tokens": pool.block_table(main)[1], "fork_us": (t1 - t0) * 1e6,
                      "decode_ms": e0.elapsed_time(e1), "decode_us_per_step": e0.elapsed_time(e1) / steps * 1e3,
                      "harvest_us_with_readback": (th1 - th0) * 1e6, "harvested_rows": T,
                      "merge_ms": e2.elapsed_time(e3), "release_us": (t3 - t2) * 1e6, "turn_ms": (t3 - t0) * 1e3})
    pool.sync()
    pool.close()
    print(json.dumps({"workload": "one agent turn: 23040-token main, 32 layers, 4 aux branches, 64 steps",
                      "turns": turns[1:]}))


def run_harvest():
    """The thought harvest (st_harvest) on token ids: 4 branches x 512 generated
    tokens (one turn's aux branches at the cycle's 512 steps) and 32 x 2048.
    Seeded streams with open/close tags at 6% / 8% of positions.  Prints the
    device time per call (200 calls back to back, CUDA events) and the latency
    of one call through the binding, including the read-back of the count."""
    import ctypes
    import numpy as np
    import torch
    import paper_2608_13667_gb300 as st
    st.build()
    L = st.lib()
    dev = torch.device("cuda", 0)
    stream = torch.cuda.current_stream(dev)
    res = {}
    for n_br, stride in ((4, 512), (32, 2048)):
        rng = np.random.default_rng(n_br)
        s = rng.integers(100, 5000, size=(n_br, stride)).astype(np.int32)
        r = rng.random((n_br, stride))
        s[r < 0.06] = 7
        s[(r >= 0.06) & (r < 0.14)] = 8
        ds = torch.from_numpy(s).to(dev)
        dl = torch.full((n_br,), stride, dtype=torch.int32, device=dev)
        ids = torch.empty(n_br * stride, dtype=torch.int32, device=dev)
        src = torch.empty_like(ids)
        atoms = torch.empty(n_br, dtype=torch.int32, device=dev)
        count = torch.empty(1, dtype=torch.int32, device=dev)
        args = (ctypes.c_void_p(ds.data_ptr()), stride, ctypes.c_void_p(dl.data_ptr()), n_br, 7, 8, 5,
                ctypes.c_void_p(ids.data_ptr()), ctypes.c_void_p(src.data_ptr()), ctypes.c_void_p(atoms.data_ptr()),
                ctypes.c_void_p(count.data_ptr()), ctypes.c_void_p(stream.cuda_stream))
        for _ in range(10):
            assert L.st_harvest(*args) == 0
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n = 200
        e0.record(stream)
        for _ in range(n):
            L.st_harvest(*args)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        dev_us = e0.elapsed_time(e1) / n * 1e3
        t0 = time.perf_counter()
        for _ in range(20):
            st.st_harvest(ds, dl, 7, 8, 5)
        lat_us = (time.perf_counter() - t0) / 20 * 1e6
        res[f"{n_br}x{stride}"] = {"device_us_per_call": dev_us, "latency_us_with_readback": lat_us,
                                   "harvested_tokens": int(count.item())}
    print(json.dumps({"workload": "thought harvest on token ids", **res}))


def run_prefill_batch():
    """Batched prefill on the batched-serving shape (1 layer, 32/8 heads, D 128):
    16 agents with contexts of 4096-32768 tokens each receive an observation of
    64-1024 rows (seeded).  One st_prefill_batch against one st_merge per agent
    on a second, identical set of agents.  Prints CUDA-event timings."""
    import numpy as np
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import get, kv_rows, queries
    dev = torch.device("cuda", 0)
    st.build()
    w = get(3)
    rng = np.random.default_rng(7)
    obs = [int(x) for x in rng.integers(64, 1024, size=w.n_tasks, endpoint=True)]
    pages = 2 * sum((p + n + 15) // 16 + 1 for p, n in zip(w.prefix, obs))
    pool = st.Pool(n_layers=w.n_layers, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads, head_dim=w.head_dim,
                   n_blocks=pages + 64, seed=w.seed, device=dev, max_seqs=2 * w.n_tasks + 3,
                   max_pages=max(w.prefix) // 16 + 80, max_decode_branches=8, max_splits=8)
    sets = []
    for rep in range(2):
        seqs = []
        for t_, p in enumerate(w.prefix):
            m = pool.seq_create()
            k, v = kv_rows(w, ("prefix", t_), p, device=dev)
            pool.append_kv([m], k.view(w.n_layers, 1, p, w.n_kv_heads, w.head_dim),
                           v.view(w.n_layers, 1, p, w.n_kv_heads, w.head_dim))
            seqs.append(m)
        sets.append(seqs)
    R = sum(obs)
    k, v = kv_rows(w, ("obs",), R, device=dev)
    q = queries(w, ("obs_q",), R, device=dev)
    # warm-up on a small extra sequence (first-launch setup stays out of the timings)
    x = pool.seq_create()
    pool.append_kv([x], k[:, :64].contiguous().view(w.n_layers, 1, 64, w.n_kv_heads, w.head_dim),
                   v[:, :64].contiguous().view(w.n_layers, 1, 64, w.n_kv_heads, w.head_dim))
    pool.merge(x, q[:, :16].contiguous(), k[:, :16].contiguous(), v[:, :16].contiguous())
    pool.prefill_batch([x], [16], q[:, :16].contiguous(), k[:, :16].contiguous(), v[:, :16].contiguous())
    keys = sum(n * p + n * (n + 1) / 2 for p, n in zip(w.prefix, obs))
    flops = 4.0 * w.head_dim * keys * w.n_q_heads * w.n_layers
    pool.sync()
    pool.profile_read()
    pool.profile_enable(True)
    pool.prefill_batch(sets[0], obs, q, k, v)
    pool.sync()
    b = pool.profile_read()
    off = 0
    for m, n in zip(sets[1], obs):
        pool.merge(m, q[:, off:off + n].contiguous(), k[:, off:off + n].contiguous(), v[:, off:off + n].contiguous())
        off += n
    pool.sync()
    s_ = pool.profile_read()
    pool.close()
    bm, sm_ = b["merge_prefill"], s_["merge_prefill"]
    ba, sa = b["append_kv"], s_["append_kv"]
    print(json.dumps({"agents": w.n_tasks, "rows": R, "tflop": flops / 1e12,
                      "batched": {"launches": bm["launches"], "prefill_ms": bm["total_ms"],
                                  "append_ms": ba["total_ms"], "tflops": flops / bm["total_ms"] / 1e9},
                      "per_agent": {"launches": sm_["launches"], "prefill_ms": sm_["total_ms"],
                                    "append_ms": sa["total_ms"], "tflops": flops / sm_["total_ms"] / 1e9}}))


def run_profile_merge():
    """Only the merge case of run_profile_small (about 1 GB on the device):
    three identical merge launches, for ncu captures of the merge kernel."""
    print(json.dumps(_merge_case()))


def run_cycle():
    """The full fork / decode / merge cycle (8 tasks x 16384-token contexts,
    32 layers, 32/8 heads): per turn, fork 4 branches per task, 512 steps in
    which main + branches + 64 unforked 2048-token sequences append one row
    and decode, merge 2048 thought rows into each main, release.  5 turns.
    Prints the time of the whole cycle and of its decode and merge parts."""
    import torch
    import paper_2608_13667_gb300 as st
    from workloads import get, kv_rows, queries
    w = get(5)
    dev = torch.device("cuda", 0)
    st.build()
    pool = st.Pool(n_layers=w.n_layers, n_q_heads=w.n_q_heads, n_kv_heads=w.n_kv_heads, head_dim=w.head_dim,
                   n_blocks=w.n_blocks, seed=w.seed, device=dev, **w.limits)
    L, Hkv, D = w.n_layers, w.n_kv_heads, w.head_dim
    mains = []
    for t in range(w.n_tasks):
        m = pool.seq_create()
        for c0 in range(0, w.prefix[t], PREFIX_CHUNK):
            n = min(PREFIX_CHUNK, w.prefix[t] - c0)
            k, v = kv_rows(w, ("prefix", t, c0), n, device=dev)
            pool.append_kv([m], k.view(L, 1, n, Hkv, D), v.view(L, 1, n, Hkv, D))
        mains.append(m)
    n_rows = w.n_tasks * (w.n_aux + 1) + w.singletons
    # step inputs drawn once and reused (values do not change the work)
    sk, sv = kv_rows(w, ("step",), n_rows, device=dev)
    sk, sv = sk.view(L, n_rows, 1, Hkv, D), sv.view(L, n_rows, 1, Hkv, D)
    sq = queries(w, ("q",), n_rows, device=dev)
    mk, mv = kv_rows(w, ("merge",), w.merge_tokens, device=dev)
    mq = queries(w, ("mq",), w.merge_tokens, device=dev)
    o = torch.empty((L, n_rows, w.n_q_heads, D), dtype=torch.float32, device=dev)
    lse = torch.empty((L, n_rows, w.n_q_heads), dtype=torch.float32, device=dev)
    mo = torch.empty((L, w.merge_tokens, w.n_q_heads, D), dtype=torch.float32, device=dev)
    ml = torch.empty((L, w.merge_tokens, w.n_q_heads), dtype=torch.float32, device=dev)
    torch.cuda.synchronize(dev)
    pool.profile_enable(True)
    t_fork = t_release = 0.0  # host time of the metadata-only calls (no GPU work)
    n_fork = n_release = 0
    t_all = time.perf_counter()
    for turn in range(w.turns):
        singles = [pool.seq_create() for _ in range(w.singletons)]
        for i in range(0, w.singletons, 8):
            k, v = kv_rows(w, ("single", turn, i), 8 * w.singleton_len, device=dev)
            pool.append_kv(singles[i:i + 8], k.view(L, 8, w.singleton_len, Hkv, D),
                           v.view(L, 8, w.singleton_len, Hkv, D))
        t0 = time.perf_counter()
        groups = [[m] + pool.fork(m, w.n_aux) for m in mains]
        t_fork += time.perf_counter() - t0
        n_fork += len(mains)
        rids = [r for g in groups for r in g] + singles
        for step in range(w.steps):
            pool.append_kv(rids, sk, sv)
            pool.decode_attn(rids, sq, o, lse)
        for m in mains:
            pool.merge(m, mq, mk, mv, mo, ml)
        t0 = time.perf_counter()
        for g in groups:
            for a in g[1:]:
                pool.release(a)
        t_release += time.perf_counter() - t0
        n_release += sum(len(g) - 1 for g in groups)
        for s_ in singles:
            pool.release(s_)
    torch.cuda.synchronize(dev)
    total = time.perf_counter() - t_all
    pool.sync()
    stats = pool.profile_read()
    dec, mer = stats["decode_partial"], stats["merge_prefill"]
    print(json.dumps({
        "workload": w.name, "seconds": total,
        "decode_steps": dec["launches"], "decode_ms_per_step": dec["total_ms"] / dec["launches"],
        "decode_gbs": dec["bytes"] / dec["total_ms"] / 1e6,
        "branch_steps_per_s": dec["launches"] * n_rows / total,
        "merges": mer["launches"], "merge_ms": mer["total_ms"] / mer["launches"],
        "merge_tflops": mer["flops"] / mer["total_ms"] / 1e9,
        "fork_us": t_fork / n_fork * 1e6, "fork_note": f"st_fork of {w.n_aux} branches off a main context, host time through the binding",
        "release_us": t_release / n_release * 1e6, "release_note": "st_release of one branch, host time through the binding",
        "kernels": {k: {"launches": v["launches"], "ms": v["total_ms"]} for k, v in stats.items() if v["launches"]}}))


# --------------------------------------------------------------------------- oracle

def _oracle_worker(w, dev_name, cmd_q, res_q, barrier):
    """A host-core worker of the oracle baseline.  Per round it receives a
    list of (layer, KV head) units of fork group 0, draws their inputs (not
    timed), waits at the barrier with the other workers, then runs the float64
    oracle (oracle.attention.decode, unchanged) on each unit's branches --
    every branch's query heads of that KV head over its materialised context,
    prefix ++ suffix -- and reports its start and end on the monotonic clock."""
    import torch
    torch.set_num_threads(1)
    from oracle import attention as A
    from workloads import kv_rows, queries
    dev = torch.device(dev_name)
    G = w.n_q_heads // w.n_kv_heads
    while True:
        units = cmd_q.get()
        if units is None:
            return
        jobs, drawn = [], {}
        for layer, g in units:
            if layer not in drawn:
                ks, vs = [], []
                for c0 in range(0, w.prefix[0], PREFIX_CHUNK):
                    n = min(PREFIX_CHUNK, w.prefix[0] - c0)
                    k, v = kv_rows(w, ("prefix", 0, c0), n, device=dev, layers=[layer])
                    ks.append(k[0].cpu())
                    vs.append(v[0].cpu())
                suf = []
                for b, n in enumerate(w.suffix[0]):
                    if n:
                        k, v = kv_rows(w, ("suffix", 0, b), n, device=dev, layers=[layer])
                        suf.append((k[0].cpu(), v[0].cpu()))
                    else:
                        suf.append(None)
                q = queries(w, ("q", 0, 0), w.n_aux + 1, device=dev, layers=[layer])[0].cpu()
                drawn = {layer: (torch.cat(ks), torch.cat(vs), suf, q)}
            pk, pv, suf, q = drawn[layer]
            for b in range(w.n_aux + 1):
                kc, vc = pk[:, g:g + 1], pv[:, g:g + 1]
                if suf[b] is not None:
                    kc = torch.cat([kc, suf[b][0][:, g:g + 1]])
                    vc = torch.cat([vc, suf[b][1][:, g:g + 1]])
                jobs.append((q[b, g * G:(g + 1) * G].clone(), kc.contiguous(), vc.contiguous()))
        drawn = {}
        barrier.wait()
        t0 = time.monotonic()
        for qh, kc, vc in jobs:
            A.decode(qh, kc, vc)
        t1 = time.monotonic()
        res_q.put((t0, t1, len(units)))


class ParallelOracle:
    """The float64 oracle on the host cores: one spawned worker process per
    core, each with one BLAS / torch thread, over (layer, KV head) units of
    one fork group.  A round's time is from the first worker's start to the
    last worker's end, all workers starting together after drawing their
    inputs."""

    def __init__(self, w, n_workers=None):
        import multiprocessing as mp
        import torch
        self.w = w
        self.n = max(1, min(n_workers or os.cpu_count() or 1, w.n_layers * w.n_kv_heads))
        ctx = mp.get_context("spawn")
        self.barrier = ctx.Barrier(self.n + 1)
        self.res = ctx.Queue()
        self.cmds = [ctx.Queue() for _ in range(self.n)]
        dev = "cuda" if torch.cuda.is_available() else "cpu"
        saved = {v: os.environ.get(v) for v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS", "MKL_NUM_THREADS")}
        os.environ.update({v: "1" for v in saved})
        try:
            self.procs = [ctx.Process(target=_oracle_worker, args=(w, dev, q, self.res, self.barrier), daemon=True)
                          for q in self.cmds]
            for p in self.procs:
                p.start()
        finally:
            for v, val in saved.items():
                if val is None:
                    os.environ.pop(v, None)
                else:
                    os.environ[v] = val
        self.next_unit = 0

    def round(self, units_per_worker):
        """Runs the next units_per_worker units on every worker; returns
        (seconds, branch-steps)."""
        w = self.w
        all_units = [(l, g) for l in range(w.n_layers) for g in range(w.n_kv_heads)]
        for q in self.cmds:
            mine = [all_units[(self.next_unit + i) % len(all_units)] for i in range(units_per_worker)]
            self.next_unit += units_per_worker
            q.put(mine)
        self.barrier.wait()
        t0, t1, n = [], [], 0
        for _ in self.procs:
            a, b, k = self.res.get()
            t0.append(a)
            t1.append(b)
            n += k
        return max(t1) - min(t0), n * (w.n_aux + 1) / (w.n_layers * w.n_kv_heads)

    def close(self):
        for q in self.cmds:
            q.put(None)
        for p in self.procs:
            p.join(timeout=30)


def cpu_baseline(w, n_workers=None):
    """The oracle on the host cores over a bounded sample of the step: 8
    layers of one fork group, every KV head, all its branches, spread over
    one worker per core."""
    po = ParallelOracle(w, n_workers)
    try:
        per = max(1, (min(8, w.n_layers) * w.n_kv_heads) // po.n)
        dt, units = po.round(per)
    finally:
        po.close()
    n_units = per * po.n
    layers = min(w.n_layers, -(-n_units // w.n_kv_heads))
    return {"value": units / dt, "unit": UNIT, "cores": po.n, "kind": "oracle",
            "sample": f"{n_units} (layer, KV head) units over {layers} of {w.n_layers} layers of 1 of "
                      f"{w.n_tasks} fork groups ({w.n_aux + 1} branches, {w.prefix[0]}-token prefix), float64 numpy, "
                      f"{po.n} worker processes with one thread each; {dt:.2f} s wall ({dt * po.n:.1f} core-s)"}


def run_reference(args, rank, ws, local):
    w = _workload(args)
    if rank != 0:
        return {}
    po = ParallelOracle(w, args.oracle_workers)
    try:
        for s in range(args.warmup):
            po.round(1)
        total_dt = total_units = 0.0
        for s in range(args.steps):
            dt, units = po.round(1)
            total_dt += dt
            total_units += units
    finally:
        po.close()
    value = total_units / total_dt
    sample = (f"each step: {po.n} (layer, KV head) units of 1 fork group ({w.n_aux + 1} branches, "
              f"{w.prefix[0]}-token prefix) of the {w.name} workload, float64 numpy oracle, one per worker "
              f"process ({po.n} processes, one thread each)")
    return {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": ws, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": total_dt / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": w.name, "sample": sample},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": po.n, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, default=4)
    ap.add_argument("--n-aux", type=int, default=None,
                    help="config 4 with this many auxiliary branches per group instead of 4")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--oracle-workers", type=int, default=None,
                    help="host worker processes of the oracle baseline (default: one per core)")
    ap.add_argument("--profile-small", action="store_true",
                    help="run the small decode + merge case used for ncu captures and exit")
    ap.add_argument("--profile-wide", action="store_true",
                    help="run the small 9-branch decode case (wide tile) used for ncu captures and exit")
    ap.add_argument("--turn", action="store_true",
                    help="time one agent turn (fork, 64 decode steps, harvest, merge, release) and exit")
    ap.add_argument("--harvest", action="store_true",
                    help="time the thought harvest (st_harvest) and exit")
    ap.add_argument("--prefill-batch", action="store_true",
                    help="time one batched prefill of 16 agents against one merge per agent and exit")
    ap.add_argument("--profile-merge", action="store_true",
                    help="run only the merge case of --profile-small (three identical launches) and exit")
    ap.add_argument("--cycle", action="store_true",
                    help="time the full fork/decode/merge cycle workload and exit")
    args = ap.parse_args()
    if args.profile_small:
        run_profile_small()
        return
    if args.profile_merge:
        run_profile_merge()
        return
    if args.prefill_batch:
        run_prefill_batch()
        return
    if args.harvest:
        run_harvest()
        return
    if args.turn:
        run_turn()
        return
    if args.profile_wide:
        run_profile_wide(args.n_aux)
        return
    if args.cycle:
        run_cycle()
        return
    rank, ws, local = _dist()
    if args.impl == "reference":
        res = run_reference(args, rank, ws, local)
    else:
        res = run_ours(args, rank, ws, local)
        if rank == 0 and ws == 1 and not args.no_cpu_baseline:
            import torch
            res["cpu_baseline"] = cpu_baseline(_workload(args), args.oracle_workers)
    if rank == 0:
        print(json.dumps(res), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
