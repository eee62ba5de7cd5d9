/*
 * st.h -- C ABI of the fork-group attention library (libsecondthought.so).
 *
 * Second Thought (arXiv 2608.13667) forks four auxiliary reasoning branches
 * off an agent's main context when a Thought phase ends (Section 3.2), lets
 * them decode while the main thread acts and waits (Section 3.1), and merges
 * their harvested thoughts back after the observation (Section 3.5).  Every
 * branch receives the same snapshot H_t + R_t, so the KV of that prefix is
 * shared by all decoding streams (Section 3.3); the branch load is therefore
 * dominated by cached-prefix reads (Section 4.4, timing and cost analyses).
 *
 * This library is the GPU side of that: a paged KV pool with refcounted
 * copy-on-write block tables (fork, release and the merge's bookkeeping touch
 * only metadata), a decode kernel that streams every shared prefix page once
 * for all branches x GQA heads of a fork group, per-branch suffix work, a
 * log-sum-exp combine, and a causal prefill for the merged thought rows.
 *
 * Conventions for every call:
 *  - Return value: ST_OK or an error code; a failing call changes no state.
 *    st_last_error() gives a one-line reason for the last failure.  The one
 *    exception is a CUDA call that fails after an append has changed the
 *    host tables (st_append_kv, st_merge, st_prefill_batch; or the table
 *    upload at the start of st_decode_attn): that call returns ST_ERR_CUDA
 *    and the pool is then unusable -- every later call on it returns
 *    ST_ERR_STATE except st_pool_destroy, st_last_error and the
 *    introspection calls (st_block_table, st_refcounts, st_free_list,
 *    st_decode_plan, st_profile_*), which report the host's view.
 *  - Device pointers are plain CUDA device addresses on the pool's device;
 *    the caller owns them (KV storage, workspace, inputs, outputs).
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls that
 *    take a stream enqueue work and return without waiting.  All calls on one
 *    pool must be ordered: use one stream, or order streams with events.
 *  - A pool is used from one host thread at a time.
 *  - Sequence handles (st_seq) are (generation << 32 | slot); a handle is
 *    invalid after st_release, and using it gives ST_ERR_INVALID.
 *  - bf16 tensors are IEEE bfloat16 bit patterns; fp32 outputs are float.
 *  - Attention is softmax(q k^T / sqrt(D)) v with the log-sum-exp returned in
 *    natural log (scale included); query head h reads KV head h / G with
 *    G = n_q_heads / n_kv_heads.
 */
#ifndef ST_H
#define ST_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define ST_API __attribute__((visibility("default")))
#else
#define ST_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  ST_OK = 0,
  ST_ERR_INVALID = 1, /* bad argument, stale handle, or a device-side bounds check fired */
  ST_ERR_OOM = 2,     /* pool pages or sequence slots exhausted; nothing changed */
  ST_ERR_STATE = 3,   /* operation not possible in the pool's current mode/state */
  ST_ERR_CUDA = 4,    /* a CUDA runtime call failed */
  ST_ERR_TIMEOUT = 5  /* a device-side wait ran past its limit (reported by st_sync) */
} st_status;

typedef int64_t st_seq;

/* Test hook for the device-timeout path: with this flag the decode kernel's
 * loader issues no copies, so its bounded waits (2 s) run out, the kernel
 * records ST_ERR_TIMEOUT in the device status word and returns without
 * faulting, and the next st_sync reports ST_ERR_TIMEOUT.  Outputs of such a
 * call are undefined.  Never set in normal use. */
#define ST_FLAG_HOLD_LOADS 1
/* Test hook for the CUDA-failure path: with this flag every kernel launch
 * the pool would make is skipped and reported as failed (ST_ERR_CUDA), as a
 * failing launch would be.  Never set in normal use. */
#define ST_FLAG_FAIL_LAUNCH 2
typedef struct st_pool st_pool;

/* Pool geometry and capacities.
 * KV storage layout (bf16, caller-allocated):
 *   k_pool, v_pool : [n_layers][n_blocks][n_kv_heads][page_size][head_dim]
 * so one page of one head is page_size*head_dim contiguous bf16 values. */
typedef struct {
  int32_t n_layers;
  int32_t n_q_heads;
  int32_t n_kv_heads;          /* must divide n_q_heads; G = n_q_heads / n_kv_heads <= 48 */
  int32_t head_dim;            /* 64 or 128 */
  int32_t page_size;           /* tokens per page; must be 16 */
  int32_t max_seqs;            /* live sequences at once (handle slots) */
  int32_t max_pages;           /* block-table capacity per sequence, in pages */
  int32_t max_decode_branches; /* branches per st_decode_attn call */
  int32_t max_splits;          /* partial results per (branch, head, layer) in one decode; 2..32 */
  int32_t flags;               /* ST_FLAG_* bits; 0 for normal use */
  int64_t n_blocks;            /* physical pages in the pool (each spans all layers and KV heads) */
  uint64_t seed;               /* seeds the free-list shuffle (splitmix64, Fisher-Yates) */
} st_config;

/* Bytes of device workspace st_pool_create needs for `cfg` (0 if cfg is invalid).
 * The workspace holds the device copy of the block tables, the staging area
 * for per-call plans, the decode partials and the device status word. */
ST_API size_t st_workspace_bytes(const st_config* cfg);

/* Create a pool over caller-owned storage.
 * k_pool, v_pool: device bf16 buffers in the layout above, 16-byte aligned.
 * workspace: device buffer of st_workspace_bytes(cfg) bytes, 256-byte aligned.
 * device: CUDA device ordinal of the buffers.  device = -1 creates a
 *   metadata-only pool (k_pool, v_pool and workspace must be NULL): fork,
 *   append and release then update tables and refcounts without touching any
 *   GPU, and attention calls return ST_ERR_STATE.
 * The free list starts as a Fisher-Yates shuffle of [0, n_blocks) driven by
 * splitmix64(seed): for i = n-1 down to 1, j = next() % (i+1), swap(i, j);
 * allocation pops the head, freed pages are pushed to the tail.
 * On success *out owns host memory and a pinned staging buffer; release it
 * with st_pool_destroy. */
ST_API st_status st_pool_create(const st_config* cfg, void* k_pool, void* v_pool, void* workspace,
                                int device, st_pool** out);

/* Free the pool's host state (waits for its outstanding work first).  The
 * caller's device buffers are not freed. */
ST_API st_status st_pool_destroy(st_pool* pool);

/* New empty sequence (a main thread).  ST_ERR_OOM when no slot is free. */
ST_API st_status st_seq_create(st_pool* pool, st_seq* out);

/* Fork (Section 3.2/3.3): create n_aux sequences whose block tables are copies
 * of `seq`'s, taking one reference on every page; no page is allocated and no
 * KV byte moves.  All-or-nothing: ST_ERR_OOM if fewer than n_aux slots are
 * free.  out_aux receives n_aux handles. */
ST_API st_status st_fork(st_pool* pool, st_seq seq, int n_aux, st_seq* out_aux);

/* Fork from an earlier point of `seq` (Table 2 of the paper: "w/o R_t" forks
 * before the just-finished thought, "fork onset" at the start of the turn):
 * the n_aux children see only seq's first `length` rows (0 <= length <=
 * seq's length).  They take the first ceil(length / page) table entries with
 * one reference each; a child's last page may still hold seq's rows past
 * `length`, which the child's first append copies away (copy-on-write of
 * rows [0, length % page)).  Otherwise as st_fork. */
ST_API st_status st_fork_at(st_pool* pool, st_seq seq, int64_t length, int n_aux, st_seq* out_aux);

/* Append n_tok KV rows to each of the n_br sequences in br (in that order;
 * each sequence at most once per call).
 * k, v: device bf16 [n_layers][n_br][n_tok][n_kv_heads][head_dim].
 * Row t of branch i lands at logical position len_i + t.  A fresh page is
 * taken when the position is page-aligned; a shared partial last page
 * (refcount > 1) is first copied (copy-on-write: new page, rows
 * [0, len % page) copied for every layer and head, one reference dropped on
 * the old page).  All-or-nothing: ST_ERR_OOM if the pool lacks the pages the
 * whole call needs.  On a metadata-only pool k and v must be NULL. */
ST_API st_status st_append_kv(st_pool* pool, const st_seq* br, int n_br, int n_tok, const void* k,
                              const void* v, void* stream);

/* Decode attention for one query per branch (Section 3.1: main and branches
 * decode concurrently).  Branches forked from a common sequence are grouped:
 * the pages they share are read once for the whole group, each branch's own
 * pages once for that branch, and the partial results are combined by
 * log-sum-exp.  The result equals softmax attention over each branch's full
 * context (every row appended to it or inherited at fork).
 * q:   device bf16 [n_layers][n_br][n_q_heads][head_dim]
 * o:   device fp32 [n_layers][n_br][n_q_heads][head_dim]
 * lse: device fp32 [n_layers][n_br][n_q_heads] (natural log)
 * Every branch must hold at least one row; n_br <= max_decode_branches;
 * a sequence may appear once. */
ST_API st_status st_decode_attn(st_pool* pool, const st_seq* br, int n_br, const void* q, float* o,
                                float* lse, void* stream);

/* One step of the decode loop (Section 3.1: each branch generates its own
 * tokens): append one KV row to each branch, then decode one query per
 * branch -- the same result, tables and page allocation as st_append_kv with
 * n_tok = 1 followed by st_decode_attn on the same branches, in fewer
 * launches: the decode kernel that reads a branch's last page writes the new
 * row into it first.  (When a branch's last page is shared and partly filled,
 * the step copies it with a separate append launch first.)
 * k, v: device bf16 [n_layers][n_br][n_kv_heads][head_dim], the new rows;
 * q, o, lse: as st_decode_attn.  Branches may be empty before the call.
 * Failures before the append change nothing; a failure after it (a CUDA
 * error, or a plan too large for one staging slot) leaves the pool unusable,
 * as for the other appending calls. */
ST_API st_status st_decode_step(st_pool* pool, const st_seq* br, int n_br, const void* k, const void* v,
                                const void* q, float* o, float* lse, void* stream);

/* The work decomposition st_decode_attn would use for these branches, without
 * launching anything (host only; also on a metadata-only pool, which plans for
 * 152 SMs with two decode CTAs each).  One item is a run of pages of one
 * block table read for a set of branches, one CTA per KV head and layer:
 * items:    int32 [item_cap][8] rows {owner, page_begin, n_pages, n_tokens,
 *           member_base, n_members, split, flags}: owner is the index in br
 *           of the branch whose block table the run is read from, pages
 *           [page_begin, page_begin + n_pages) of it, n_tokens valid keys,
 *           members[member_base .. + n_members) the branches (indices in br)
 *           whose query rows are stacked on it, split the partial slot it
 *           writes for each of them; flags bit 0: a sibling item of the same
 *           fork family reads the same pages (kept in L2), bit 1: the wide
 *           (M = 128) tile, for 65 to 128 stacked rows, bit 2: the paired
 *           tile (two M = 128 tiles of one CTA, for 129 to 256 stacked rows);
 *           neither: the narrow tile, up to 64 stacked rows.  Narrow items
 *           come first, then wide, then paired.
 * members:  int32 [member_cap]
 * n_splits: int32 [n_br], partial results per branch (each split index
 *           0 .. n_splits - 1 is written by exactly one item)
 * *n_items and *n_members receive the sizes the plan needs; ST_ERR_INVALID
 * (nothing written) when they exceed item_cap or member_cap. */
ST_API st_status st_decode_plan(st_pool* pool, const st_seq* br, int n_br, int32_t* items, int item_cap,
                                int32_t* members, int member_cap, int32_t* n_splits, int* n_items,
                                int* n_members);

/* Merge (Section 3.5): append the n_tok harvested thought rows to `main`
 * (same rules as st_append_kv) and run their causal prefill: thought row i
 * attends over main's rows [0, L0 + i] inclusive, L0 = main's length before
 * the call.  q: bf16 [n_layers][n_tok][n_q_heads][head_dim];
 * k, v: bf16 [n_layers][n_tok][n_kv_heads][head_dim];
 * o: fp32 [n_layers][n_tok][n_q_heads][head_dim]; lse: fp32 [n_layers][n_tok][n_q_heads].
 * n_tok = 0 (nothing harvested) is a no-op returning ST_OK.  On a
 * metadata-only pool all five pointers must be NULL (bookkeeping only). */
ST_API st_status st_merge(st_pool* pool, st_seq main, int n_tok, const void* q, const void* k,
                          const void* v, float* o, float* lse, void* stream);

/* Batched prefill across sequences (Section 3.1: the observation O_t is
 * appended to each agent's history, and Section 3.5: the harvested thoughts
 * after it; several agents' rows arrive together when many are served at
 * once).  For each i in order, n_tok[i] rows are appended to seqs[i] (same
 * rules as st_append_kv; the pages are taken as if the sequences were
 * appended one after another) and run through the causal prefill of
 * st_merge: row r of sequence i attends over its rows [0, L0_i + r], L0_i =
 * its length before the call.  One launch covers every sequence.
 * n_tok:  host int32 [n_seq], each >= 0 (0: the sequence is left unchanged)
 * rows are packed in sequence order, R = sum of n_tok:
 * q: bf16 [n_layers][R][n_q_heads][head_dim];
 * k, v: bf16 [n_layers][R][n_kv_heads][head_dim];
 * o: fp32 [n_layers][R][n_q_heads][head_dim]; lse: fp32 [n_layers][R][n_q_heads].
 * A sequence may appear once.  All or nothing on ST_ERR_OOM.  R = 0 is a
 * no-op.  On a metadata-only pool all five pointers must be NULL. */
ST_API st_status st_prefill_batch(st_pool* pool, const st_seq* seqs, int n_seq, const int32_t* n_tok,
                                  const void* q, const void* k, const void* v, float* o, float* lse,
                                  void* stream);

/* Thought harvest (Section 3.5): when the observation arrives, each branch's
 * generated token stream is cut at its last closed </thought>.  Completed
 * atoms (an open-tag token through the next close-tag token, tags included)
 * are kept -- the first `cap` per branch (the paper caps at 5) -- an
 * unfinished atom is dropped, a branch with no completed atom contributes
 * nothing, and the kept atoms are concatenated in branch order.  An open tag
 * inside an unfinished atom restarts it; a close tag outside an atom is
 * ignored.  The count T written to *out_count is the number of thought rows
 * to pass to st_merge (T = 0: nothing harvested, the turn is plain ReAct).
 * streams:  device int32 [n_br][stride], token ids generated by each branch
 * lens:     device int32 [n_br], tokens generated so far (clamped to stride)
 * out_ids:  device int32 [n_br * stride], harvested ids (first T valid)
 * out_src:  device int32 [n_br * stride] or NULL: b * stride + position of
 *           each harvested token in its branch's stream
 * out_atoms: device int32 [n_br] or NULL: atoms kept per branch
 * out_count: device int32 [1]
 * n_br <= 32, 0 <= cap <= 64, open_id != close_id.  Runs on `stream`; no pool
 * is needed. */
ST_API st_status st_harvest(const int32_t* streams, int stride, const int32_t* lens, int n_br,
                            int32_t open_id, int32_t close_id, int cap, int32_t* out_ids,
                            int32_t* out_src, int32_t* out_atoms, int32_t* out_count, void* stream);

/* Release (Section 3.5: in-flight branches are cancelled and discarded):
 * drop one reference per table entry in logical order; pages reaching zero
 * go to the tail of the free list.  The handle becomes invalid. */
ST_API st_status st_release(st_pool* pool, st_seq seq);

/* Introspection.  st_block_table copies up to `cap` physical page ids of
 * `seq` (logical order) into out and reports its page and token counts. */
ST_API st_status st_block_table(st_pool* pool, st_seq seq, int32_t* out, int cap, int* n_pages,
                                int* n_tokens);
/* Per-page refcounts, out[n_blocks]. */
ST_API st_status st_refcounts(st_pool* pool, int32_t* out, int64_t cap);
/* Free list in FIFO order (head first); *n receives its length. */
ST_API st_status st_free_list(st_pool* pool, int32_t* out, int64_t cap, int64_t* n);

/* Wait for the stream and report device-side errors raised since the last
 * st_sync (ST_ERR_TIMEOUT for a wait that ran out, ST_ERR_INVALID for a
 * failed bounds check, ST_ERR_CUDA for a kernel whose dynamic shared memory
 * was not 1024-byte aligned); the device status word is then cleared. */
ST_API st_status st_sync(st_pool* pool, void* stream);

/* Kernel accounting.  Launch counts are always kept; with timing enabled
 * (st_profile_enable(pool, 1)) each launch is bracketed by CUDA events on
 * its stream.  st_profile_read synchronises, fills up to cap records and
 * resets the counters. */
typedef struct {
  char name[32];
  int64_t launches;
  double total_ms;     /* summed event time (0 when timing was off) */
  double bytes;        /* algorithmic bytes the launches had to move */
  double flops;        /* algorithmic floating-point operations */
  int64_t kernels;     /* device kernels launched (a decode call with both tile
                          shapes launches two per call) */
  double overhead_bytes; /* bytes moved beyond the algorithmic ones: split-KV
                            partials (written by the decode, read by the
                            combine), second reads of a split fork family's
                            shared pages, copy-on-write rows */
} st_kernel_stat;
ST_API st_status st_profile_enable(st_pool* pool, int enable);
ST_API st_status st_profile_read(st_pool* pool, st_kernel_stat* out, int cap, int* n);

/* ---- Allocation-free decode ------------------------------------------------
 * The paper has no counterpart to this call; it exists for callers that
 * cannot allocate device memory: code running inside a host framework that
 * owns every device allocation and forbids new ones after start-up,
 * real-time serving loops that must not allocate on the hot path, and plugins
 * that are handed input and output pointers but no allocator.  Such callers
 * cannot supply the workspace st_pool_create needs, so this call takes only
 * inputs and outputs and allocates nothing (no cudaMalloc, no cudaFree, no
 * allocating library routine).  It runs the same kernels as st_decode_attn.
 *
 * Its scratch -- the per-call plan, a device copy of the page tables and the
 * split-KV partials -- lives in a static device array of
 * ST_NOALLOC_SCRATCH_BYTES (16 MiB) that every GPU loading the library holds
 * until the process exits.  The first call on a device looks up that array's
 * device address (once per device, with the device current); make that
 * first call before any stream capture.  Every call reuses the array, so
 * calls that overlap on the GPU (different streams without ordering) race.
 *
 * geom:        pool geometry (n_layers, n_q_heads, n_kv_heads, head_dim,
 *              page_size = 16, n_blocks); of the flags only ST_FLAG_HOLD_LOADS
 *              is honoured; other fields are ignored.
 * k_pool/v_pool: device bf16 [n_layers][n_blocks][n_kv_heads][16][head_dim]
 *              (the st_pool_create layout), 16-byte aligned.
 * page_table:  HOST int32 [n_br][table_stride], each branch's physical page
 *              ids in logical order; the first ceil(seq_len / 16) of each
 *              row must lie in [0, n_blocks) (checked; ST_ERR_INVALID).
 * seq_len:     HOST int32 [n_br], tokens in each branch's context (>= 1,
 *              ceil(len / 16) <= table_stride).
 * q, o, lse:   as st_decode_attn, on the current device.
 * status:      DEVICE int32 [1], caller-owned.  The call clears it on
 *              `stream` before its kernels run; once the stream has passed
 *              the call it holds ST_OK, ST_ERR_TIMEOUT (a device-side wait ran
 *              past its limit: o and lse are then undefined),
 *              ST_ERR_INVALID (a device-side bounds check fired) or
 *              ST_ERR_CUDA (the kernel's dynamic shared memory was not
 *              1024-byte aligned; nothing computed).  The return
 *              value covers only what the host can see when the call returns.
 * Branches whose tables start on the same physical page are treated as one
 * fork group: their common full pages are read once for the group (groups
 * of more than 64 / G branches are split into several).
 * Returns ST_ERR_INVALID for bad arguments or n_br > ST_NOALLOC_MAX_BRANCHES,
 * and ST_ERR_OOM when the call needs more than the static scratch:
 *   36.25 KiB of plan + 4*n_br*table_stride (rounded up to 256 bytes)
 *   + 4*n_layers*n_br*n_q_heads*16*(head_dim + 1) bytes > 16 MiB.
 * The work runs on `stream`. */
#define ST_NOALLOC_SCRATCH_BYTES (16u << 20)
#define ST_NOALLOC_MAX_BRANCHES 64
ST_API st_status st_decode_attn_noalloc(const st_config* geom, const void* k_pool, const void* v_pool,
                                        const int32_t* page_table, int table_stride,
                                        const int32_t* seq_len, int n_br, const void* q, float* o,
                                        float* lse, int32_t* status, void* stream);

ST_API const char* st_status_str(st_status s);
ST_API const char* st_last_error(st_pool* pool);

#ifdef __cplusplus
}
#endif

#endif /* ST_H */
