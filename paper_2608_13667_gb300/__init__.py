"""Fork-group attention for Second Thought on GB300 (sm_103a).

A thin ctypes binding over libsecondthought.so (declared in include/st.h).
Every step of the path -- table refresh, KV append with copy-on-write,
shared-prefix decode partials, log-sum-exp combine, merge prefill -- runs in
the library's CUDA kernels; this module only checks shapes and passes device
pointers.  PyTorch supplies device memory and streams.

The functions named like the C entry points (st_fork, st_append_kv,
st_decode_attn, st_merge, st_release, ...) take a Pool as first argument;
Pool's methods do the same work.
"""
import ctypes
import os

from ._build import LIB, build  # noqa: F401

ST_OK, ST_ERR_INVALID, ST_ERR_OOM, ST_ERR_STATE, ST_ERR_CUDA, ST_ERR_TIMEOUT = range(6)
ST_FLAG_HOLD_LOADS = 1
ST_FLAG_FAIL_LAUNCH = 2
PAGE = 16


class STError(RuntimeError):
    def __init__(self, status, message):
        super().__init__(f"{message} (status {status})")
        self.status = status


class StConfig(ctypes.Structure):
    _fields_ = [
        ("n_layers", ctypes.c_int32),
        ("n_q_heads", ctypes.c_int32),
        ("n_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("page_size", ctypes.c_int32),
        ("max_seqs", ctypes.c_int32),
        ("max_pages", ctypes.c_int32),
        ("max_decode_branches", ctypes.c_int32),
        ("max_splits", ctypes.c_int32),
        ("flags", ctypes.c_int32),
        ("n_blocks", ctypes.c_int64),
        ("seed", ctypes.c_uint64),
    ]


class StKernelStat(ctypes.Structure):
    _fields_ = [
        ("name", ctypes.c_char * 32),
        ("launches", ctypes.c_int64),
        ("total_ms", ctypes.c_double),
        ("bytes", ctypes.c_double),
        ("flops", ctypes.c_double),
        ("kernels", ctypes.c_int64),
        ("overhead_bytes", ctypes.c_double),
    ]


_lib = None


def lib():
    """The loaded library.  Raises if it has not been built: there is no
    fallback path."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB):
        raise RuntimeError(f"{LIB} is missing; build it with paper_2608_13667_gb300.build()")
    L = ctypes.CDLL(LIB)
    P, I, I64, VP = ctypes.c_void_p, ctypes.c_int, ctypes.c_int64, ctypes.c_void_p
    i32p = ctypes.POINTER(ctypes.c_int32)
    i64p = ctypes.POINTER(ctypes.c_int64)
    sig = {
        "st_workspace_bytes": (ctypes.c_size_t, [ctypes.POINTER(StConfig)]),
        "st_pool_create": (I, [ctypes.POINTER(StConfig), VP, VP, VP, I, ctypes.POINTER(P)]),
        "st_pool_destroy": (I, [P]),
        "st_seq_create": (I, [P, i64p]),
        "st_fork": (I, [P, I64, I, i64p]),
        "st_fork_at": (I, [P, I64, I64, I, i64p]),
        "st_append_kv": (I, [P, i64p, I, I, VP, VP, VP]),
        "st_decode_attn": (I, [P, i64p, I, VP, VP, VP, VP]),
        "st_decode_plan": (I, [P, i64p, I, i32p, I, i32p, I, i32p, ctypes.POINTER(I), ctypes.POINTER(I)]),
        "st_decode_step": (I, [P, i64p, I, VP, VP, VP, VP, VP, VP]),
        "st_merge": (I, [P, I64, I, VP, VP, VP, VP, VP, VP]),
        "st_prefill_batch": (I, [P, i64p, I, i32p, VP, VP, VP, VP, VP, VP]),
        "st_release": (I, [P, I64]),
        "st_block_table": (I, [P, I64, i32p, I, ctypes.POINTER(I), ctypes.POINTER(I)]),
        "st_refcounts": (I, [P, i32p, I64]),
        "st_free_list": (I, [P, i32p, I64, i64p]),
        "st_sync": (I, [P, VP]),
        "st_profile_enable": (I, [P, I]),
        "st_profile_read": (I, [P, ctypes.POINTER(StKernelStat), I, ctypes.POINTER(I)]),
        "st_harvest": (I, [VP, I, VP, I, ctypes.c_int32, ctypes.c_int32, I, VP, VP, VP, VP, VP]),
        "st_decode_attn_noalloc": (I, [ctypes.POINTER(StConfig), VP, VP, i32p, I, i32p, I, VP, VP, VP, VP, VP]),
        "st_status_str": (ctypes.c_char_p, [I]),
        "st_last_error": (ctypes.c_char_p, [P]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib = L
    return L


def _seq_array(seqs):
    seqs = [int(s) for s in seqs]
    return (ctypes.c_int64 * max(1, len(seqs)))(*seqs), len(seqs)


class _SeqArrays:
    """The ctypes handle array of the last branch list passed, reused while the
    same handles come back (a decode loop passes the same list every step)."""

    def __init__(self):
        self._key = None
        self._val = None

    def __call__(self, seqs):
        key = tuple(seqs)
        if key != self._key:
            self._val = _seq_array(key)
            self._key = key
        return self._val


class Pool:
    """A KV block pool on one GPU (or metadata-only with device=None).

    KV storage (bf16 [L][n_blocks][Hkv][16][D] for K and for V) and the
    workspace are allocated here with PyTorch and owned by this object.
    """

    def __init__(self, n_layers, n_q_heads, n_kv_heads, head_dim, n_blocks, seed=0,
                 max_seqs=64, max_pages=None, max_decode_branches=16, max_splits=16,
                 device="cuda", flags=0):
        self._seqs = _SeqArrays()
        self.cfg = StConfig(
            n_layers=n_layers, n_q_heads=n_q_heads, n_kv_heads=n_kv_heads, head_dim=head_dim,
            page_size=PAGE, max_seqs=max_seqs,
            max_pages=int(max_pages if max_pages is not None else n_blocks),
            max_decode_branches=max_decode_branches, max_splits=max_splits, flags=flags,
            n_blocks=n_blocks, seed=seed)
        L = lib()
        self._h = ctypes.c_void_p()
        self.device = None
        self.k_pool = self.v_pool = self.workspace = None
        if device is None:
            st = L.st_pool_create(ctypes.byref(self.cfg), None, None, None, -1, ctypes.byref(self._h))
        else:
            import torch
            dev = torch.device(device)
            if dev.type != "cuda":
                raise ValueError("device must be a CUDA device (or None for a metadata-only pool)")
            if dev.index is None:
                dev = torch.device("cuda", torch.cuda.current_device())
            self.device = dev
            ws = L.st_workspace_bytes(ctypes.byref(self.cfg))
            if ws == 0:
                raise STError(ST_ERR_INVALID, "invalid pool configuration")
            shape = (n_layers, n_blocks, n_kv_heads, PAGE, head_dim)
            self.k_pool = torch.empty(shape, dtype=torch.bfloat16, device=dev)
            self.v_pool = torch.empty(shape, dtype=torch.bfloat16, device=dev)
            self.workspace = torch.empty(ws, dtype=torch.uint8, device=dev)
            st = L.st_pool_create(ctypes.byref(self.cfg), self.k_pool.data_ptr(), self.v_pool.data_ptr(),
                                  self.workspace.data_ptr(), dev.index, ctypes.byref(self._h))
        if st != ST_OK:
            raise STError(st, "st_pool_create: " + L.st_status_str(st).decode())

    # -- plumbing ---------------------------------------------------------
    def _check(self, st, what):
        if st != ST_OK:
            L = lib()
            msg = L.st_last_error(self._h).decode() if self._h else ""
            raise STError(st, f"{what}: {L.st_status_str(st).decode()}: {msg}")

    def _stream(self, stream):
        if self.device is None:
            return None
        if stream is None:
            # the current stream's handle, without building a Stream object
            import torch
            raw = getattr(torch._C, "_cuda_getCurrentRawStream", None)
            if raw is not None:
                return ctypes.c_void_p(raw(self.device.index))
            stream = torch.cuda.current_stream(self.device)
        return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))

    def _dev(self, t, dtype, shape, name):
        import torch
        if not isinstance(t, torch.Tensor):
            raise TypeError(f"{name} must be a torch tensor")
        if t.dtype != dtype or tuple(t.shape) != tuple(shape) or not t.is_contiguous() or t.device != self.device:
            raise ValueError(f"{name}: want contiguous {dtype} {tuple(shape)} on {self.device}, "
                             f"got {t.dtype} {tuple(t.shape)} on {t.device}")
        return ctypes.c_void_p(t.data_ptr())

    @property
    def group(self):
        return self.cfg.n_q_heads // self.cfg.n_kv_heads

    def close(self):
        if self._h:
            lib().st_pool_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- the five calls of the method ----------------------------------------
    def seq_create(self):
        out = ctypes.c_int64()
        self._check(lib().st_seq_create(self._h, ctypes.byref(out)), "st_seq_create")
        return out.value

    def fork(self, seq, n_aux=4):
        out = (ctypes.c_int64 * max(1, n_aux))()
        self._check(lib().st_fork(self._h, int(seq), n_aux, out), "st_fork")
        return [out[i] for i in range(n_aux)]

    def fork_at(self, seq, length, n_aux=4):
        out = (ctypes.c_int64 * max(1, n_aux))()
        self._check(lib().st_fork_at(self._h, int(seq), int(length), n_aux, out), "st_fork_at")
        return [out[i] for i in range(n_aux)]

    def append_kv(self, branches, k, v, stream=None):
        """k, v: bf16 [L][n_br][n_tok][Hkv][D] (a metadata-only pool takes
        k = v = None and n_tok passed as an int in k's place)."""
        arr, n = self._seqs(branches)
        c = self.cfg
        if self.device is None:
            n_tok = int(k)
            self._check(lib().st_append_kv(self._h, arr, n, n_tok, None, None, None), "st_append_kv")
            return
        import torch
        n_tok = k.shape[2] if k.dim() == 5 else -1
        shape = (c.n_layers, n, n_tok, c.n_kv_heads, c.head_dim)
        kp = self._dev(k, torch.bfloat16, shape, "k")
        vp = self._dev(v, torch.bfloat16, shape, "v")
        self._check(lib().st_append_kv(self._h, arr, n, n_tok, kp, vp, self._stream(stream)), "st_append_kv")

    def decode_attn(self, branches, q, o=None, lse=None, stream=None):
        """q: bf16 [L][n_br][Hq][D] -> (o fp32 [L][n_br][Hq][D], lse fp32 [L][n_br][Hq])."""
        import torch
        arr, n = self._seqs(branches)
        c = self.cfg
        qp = self._dev(q, torch.bfloat16, (c.n_layers, n, c.n_q_heads, c.head_dim), "q")
        if o is None:
            o = torch.empty((c.n_layers, n, c.n_q_heads, c.head_dim), dtype=torch.float32, device=self.device)
        if lse is None:
            lse = torch.empty((c.n_layers, n, c.n_q_heads), dtype=torch.float32, device=self.device)
        op = self._dev(o, torch.float32, (c.n_layers, n, c.n_q_heads, c.head_dim), "o")
        lp = self._dev(lse, torch.float32, (c.n_layers, n, c.n_q_heads), "lse")
        self._check(lib().st_decode_attn(self._h, arr, n, qp, op, lp, self._stream(stream)), "st_decode_attn")
        return o, lse

    def decode_step(self, branches, k, v, q, o=None, lse=None, stream=None):
        """One decode step: append one row per branch (k, v: bf16 [L][n_br][Hkv][D])
        and decode q (bf16 [L][n_br][Hq][D]) -> (o, lse), as st_append_kv then
        st_decode_attn."""
        import torch
        arr, n = self._seqs(branches)
        c = self.cfg
        kp = self._dev(k, torch.bfloat16, (c.n_layers, n, c.n_kv_heads, c.head_dim), "k")
        vp = self._dev(v, torch.bfloat16, (c.n_layers, n, c.n_kv_heads, c.head_dim), "v")
        qp = self._dev(q, torch.bfloat16, (c.n_layers, n, c.n_q_heads, c.head_dim), "q")
        if o is None:
            o = torch.empty((c.n_layers, n, c.n_q_heads, c.head_dim), dtype=torch.float32, device=self.device)
        if lse is None:
            lse = torch.empty((c.n_layers, n, c.n_q_heads), dtype=torch.float32, device=self.device)
        op = self._dev(o, torch.float32, (c.n_layers, n, c.n_q_heads, c.head_dim), "o")
        lp = self._dev(lse, torch.float32, (c.n_layers, n, c.n_q_heads), "lse")
        self._check(lib().st_decode_step(self._h, arr, n, kp, vp, qp, op, lp, self._stream(stream)),
                    "st_decode_step")
        return o, lse

    def decode_plan(self, branches):
        """The work decomposition st_decode_attn uses for these branches (host
        only, also on a metadata-only pool): (items, members, n_splits), items a
        list of dicts with the fields of include/st.h."""
        arr, n = _seq_array(branches)
        L = lib()
        ni, nm = ctypes.c_int(), ctypes.c_int()
        st = L.st_decode_plan(self._h, arr, n, None, 0, None, 0, None, ctypes.byref(ni), ctypes.byref(nm))
        if st != ST_OK and ni.value == 0:  # a rejected call (a plan has at least one item), not a size query
            self._check(st, "st_decode_plan")
        items = (ctypes.c_int32 * (8 * max(1, ni.value)))()
        members = (ctypes.c_int32 * max(1, nm.value))()
        n_splits = (ctypes.c_int32 * n)()
        self._check(L.st_decode_plan(self._h, arr, n, items, ni.value, members, nm.value, n_splits, ctypes.byref(ni),
                                     ctypes.byref(nm)), "st_decode_plan")
        names = ("owner", "page_begin", "n_pages", "n_tokens", "member_base", "n_members", "split", "flags")
        rows = [dict(zip(names, items[8 * k:8 * k + 8])) for k in range(ni.value)]
        return rows, list(members[:nm.value]), list(n_splits)

    def merge(self, main, q, k, v, o=None, lse=None, stream=None):
        """q: bf16 [L][T][Hq][D]; k, v: bf16 [L][T][Hkv][D] -> (o [L][T][Hq][D], lse [L][T][Hq])."""
        c = self.cfg
        if self.device is None:
            T = int(q)
            self._check(lib().st_merge(self._h, int(main), T, None, None, None, None, None, None), "st_merge")
            return None, None
        import torch
        T = q.shape[1]
        qp = self._dev(q, torch.bfloat16, (c.n_layers, T, c.n_q_heads, c.head_dim), "q")
        kp = self._dev(k, torch.bfloat16, (c.n_layers, T, c.n_kv_heads, c.head_dim), "k")
        vp = self._dev(v, torch.bfloat16, (c.n_layers, T, c.n_kv_heads, c.head_dim), "v")
        if o is None:
            o = torch.empty((c.n_layers, T, c.n_q_heads, c.head_dim), dtype=torch.float32, device=self.device)
        if lse is None:
            lse = torch.empty((c.n_layers, T, c.n_q_heads), dtype=torch.float32, device=self.device)
        op = self._dev(o, torch.float32, (c.n_layers, T, c.n_q_heads, c.head_dim), "o")
        lp = self._dev(lse, torch.float32, (c.n_layers, T, c.n_q_heads), "lse")
        self._check(lib().st_merge(self._h, int(main), T, qp, kp, vp, op, lp, self._stream(stream)), "st_merge")
        return o, lse

    def prefill_batch(self, seqs, n_tok, q, k, v, o=None, lse=None, stream=None):
        """n_tok[i] rows appended to seqs[i] and prefilled causally, all in one
        launch.  Rows packed in sequence order (R = sum(n_tok)):
        q: bf16 [L][R][Hq][D]; k, v: bf16 [L][R][Hkv][D] -> (o [L][R][Hq][D], lse [L][R][Hq]).
        On a metadata-only pool pass q = k = v = None."""
        c = self.cfg
        arr, n = _seq_array(seqs)
        counts = [int(x) for x in n_tok]
        if len(counts) != n:
            raise ValueError("n_tok needs one count per sequence")
        cnt = (ctypes.c_int32 * max(1, n))(*counts)
        if self.device is None:
            self._check(lib().st_prefill_batch(self._h, arr, n, cnt, None, None, None, None, None, None),
                        "st_prefill_batch")
            return None, None
        import torch
        R = sum(counts)
        qp = self._dev(q, torch.bfloat16, (c.n_layers, R, c.n_q_heads, c.head_dim), "q")
        kp = self._dev(k, torch.bfloat16, (c.n_layers, R, c.n_kv_heads, c.head_dim), "k")
        vp = self._dev(v, torch.bfloat16, (c.n_layers, R, c.n_kv_heads, c.head_dim), "v")
        if o is None:
            o = torch.empty((c.n_layers, R, c.n_q_heads, c.head_dim), dtype=torch.float32, device=self.device)
        if lse is None:
            lse = torch.empty((c.n_layers, R, c.n_q_heads), dtype=torch.float32, device=self.device)
        op = self._dev(o, torch.float32, (c.n_layers, R, c.n_q_heads, c.head_dim), "o")
        lp = self._dev(lse, torch.float32, (c.n_layers, R, c.n_q_heads), "lse")
        self._check(lib().st_prefill_batch(self._h, arr, n, cnt, qp, kp, vp, op, lp, self._stream(stream)),
                    "st_prefill_batch")
        return o, lse

    def release(self, seq):
        self._check(lib().st_release(self._h, int(seq)), "st_release")

    # -- introspection ---------------------------------------------------
    def block_table(self, seq):
        n_pages, n_tok = ctypes.c_int(), ctypes.c_int()
        self._check(lib().st_block_table(self._h, int(seq), None, 0, ctypes.byref(n_pages),
                                         ctypes.byref(n_tok)), "st_block_table")
        buf = (ctypes.c_int32 * max(1, n_pages.value))()
        self._check(lib().st_block_table(self._h, int(seq), buf, n_pages.value, None, None), "st_block_table")
        return [buf[i] for i in range(n_pages.value)], n_tok.value

    def refcounts(self):
        n = self.cfg.n_blocks
        buf = (ctypes.c_int32 * n)()
        self._check(lib().st_refcounts(self._h, buf, n), "st_refcounts")
        return list(buf)

    def free_list(self):
        n = ctypes.c_int64()
        self._check(lib().st_free_list(self._h, None, 0, ctypes.byref(n)), "st_free_list")
        buf = (ctypes.c_int32 * max(1, n.value))()
        self._check(lib().st_free_list(self._h, buf, n.value, None), "st_free_list")
        return [buf[i] for i in range(n.value)]

    def sync(self, stream=None):
        self._check(lib().st_sync(self._h, self._stream(stream)), "st_sync")

    def profile_enable(self, on=True):
        self._check(lib().st_profile_enable(self._h, 1 if on else 0), "st_profile_enable")

    def profile_read(self):
        buf = (StKernelStat * 16)()
        n = ctypes.c_int()
        self._check(lib().st_profile_read(self._h, buf, 16, ctypes.byref(n)), "st_profile_read")
        return {buf[i].name.decode(): dict(launches=buf[i].launches, total_ms=buf[i].total_ms,
                                           bytes=buf[i].bytes, flops=buf[i].flops, kernels=buf[i].kernels,
                                           overhead_bytes=buf[i].overhead_bytes)
                for i in range(n.value)}


# C-named entry points (argument marshalling only)
def st_pool_create(**kw):
    return Pool(**kw)


def st_seq_create(pool):
    return pool.seq_create()


def st_fork(pool, seq, n_aux=4):
    return pool.fork(seq, n_aux)


def st_fork_at(pool, seq, length, n_aux=4):
    return pool.fork_at(seq, length, n_aux)


def st_append_kv(pool, branches, k, v, stream=None):
    return pool.append_kv(branches, k, v, stream)


def st_decode_attn(pool, branches, q, o=None, lse=None, stream=None):
    return pool.decode_attn(branches, q, o, lse, stream)


def st_decode_step(pool, branches, k, v, q, o=None, lse=None, stream=None):
    return pool.decode_step(branches, k, v, q, o, lse, stream)


def st_merge(pool, main, q, k, v, o=None, lse=None, stream=None):
    return pool.merge(main, q, k, v, o, lse, stream)


def st_prefill_batch(pool, seqs, n_tok, q, k, v, o=None, lse=None, stream=None):
    return pool.prefill_batch(seqs, n_tok, q, k, v, o, lse, stream)


def st_release(pool, seq):
    return pool.release(seq)


def st_sync(pool, stream=None):
    return pool.sync(stream)


def st_harvest(streams, lens, open_id, close_id, cap=5, stream=None):
    """Thought harvest on the device (see include/st.h).  streams: int32
    [n_br, stride] CUDA tensor of generated token ids; lens: int32 [n_br] CUDA
    tensor.  Returns (ids [T], src [T], atoms [n_br]) as CUDA tensors; T is read
    back to the host to size the result."""
    import torch
    n_br, stride = streams.shape
    for t, name in ((streams, "streams"), (lens, "lens")):
        if t.dtype != torch.int32 or not t.is_cuda or not t.is_contiguous():
            raise ValueError(f"{name} must be a contiguous int32 CUDA tensor")
    out_ids = torch.empty(n_br * stride, dtype=torch.int32, device=streams.device)
    out_src = torch.empty_like(out_ids)
    atoms = torch.empty(n_br, dtype=torch.int32, device=streams.device)
    count = torch.empty(1, dtype=torch.int32, device=streams.device)
    if stream is None:
        stream = torch.cuda.current_stream(streams.device)
    st = lib().st_harvest(ctypes.c_void_p(streams.data_ptr()), stride, ctypes.c_void_p(lens.data_ptr()), n_br,
                          int(open_id), int(close_id), cap, ctypes.c_void_p(out_ids.data_ptr()),
                          ctypes.c_void_p(out_src.data_ptr()), ctypes.c_void_p(atoms.data_ptr()),
                          ctypes.c_void_p(count.data_ptr()), ctypes.c_void_p(stream.cuda_stream))
    if st != ST_OK:
        raise STError(st, "st_harvest: " + lib().st_status_str(st).decode())
    T = int(count.item())
    return out_ids[:T], out_src[:T], atoms


def st_decode_attn_noalloc(geom, k_pool, v_pool, page_tables, seq_len, q, o, lse, status=None, stream=None):
    """Allocation-free decode (see include/st.h): geom is a StConfig, k_pool/v_pool
    the bf16 KV tensors, page_tables a list of per-branch page-id lists (host),
    seq_len per-branch token counts, q/o/lse device tensors as for
    st_decode_attn, status a device int32 tensor of one element (made here if
    None) that holds the device-side outcome once the stream has passed the
    call.  Returns (status code of the call, status tensor)."""
    import torch
    n_br = len(seq_len)
    stride = max(1, max(len(t) for t in page_tables))
    table = (ctypes.c_int32 * (n_br * stride))()
    for i, t in enumerate(page_tables):
        for j, b in enumerate(t):
            table[i * stride + j] = b
    lens = (ctypes.c_int32 * n_br)(*[int(x) for x in seq_len])
    if status is None:
        status = torch.empty(1, dtype=torch.int32, device=q.device)
    if stream is None:
        stream = torch.cuda.current_stream(q.device)
    st = lib().st_decode_attn_noalloc(ctypes.byref(geom), ctypes.c_void_p(k_pool.data_ptr()),
                                      ctypes.c_void_p(v_pool.data_ptr()), table, stride, lens, n_br,
                                      ctypes.c_void_p(q.data_ptr()), ctypes.c_void_p(o.data_ptr()),
                                      ctypes.c_void_p(lse.data_ptr()), ctypes.c_void_p(status.data_ptr()),
                                      ctypes.c_void_p(stream.cuda_stream))
    return st, status
