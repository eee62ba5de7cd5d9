// Parameter blocks and launchers of the device kernels.
//
//   table_update  -- refresh rows of the device block tables from the host's
//   append_kv     -- copy-on-write page copies + scatter of new K/V rows
//   attend_tc     -- paged decode partials (tcgen05, TMEM accumulators)
//   merge_pair    -- causal merge prefill, two query tiles per CTA (tcgen05)
//   lse_combine   -- log-sum-exp combine of decode partials
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace st {

constexpr int kPageTokens = 16;

// Device status word codes (mirrors st_status values).
constexpr int32_t kDevBadIndex = 1;
constexpr int32_t kDevBadSmem = 4;  // dynamic shared memory not where a kernel needs it
constexpr int32_t kDevTimeout = 5;

struct TableRun {
  int64_t dst;    // slot * max_pages + first entry
  int32_t count;  // entries
  int32_t src;    // offset into the values array
};

struct CowCopy {
  int32_t src_block;
  int32_t dst_block;
  int32_t rows;  // rows [0, rows) of every layer and KV head
  int32_t pad;
};

struct AppendBranch {
  int32_t slot;
  int32_t start;  // sequence length before this call
  int32_t row0;   // first of this branch's rows in the call's input
  int32_t n;      // rows appended to this branch
};

struct AppendParams {
  const __nv_bfloat16* k;  // [L][n_rows][Hkv][D]: branch b's rows are [row0, row0 + n)
  const __nv_bfloat16* v;
  __nv_bfloat16* k_pool;   // [L][n_blocks][Hkv][16][D]
  __nv_bfloat16* v_pool;
  const int32_t* table;    // [max_seqs][max_pages]
  const AppendBranch* branches;
  const CowCopy* cows;
  int32_t* status;
  int64_t n_blocks;
  int32_t n_cow, n_br, n_tok, L, Hkv, max_pages;
  int32_t n_rows;          // n_br * n_tok, or the sum of the branches' n
  int32_t ragged;          // 0: every branch takes n_tok rows (branch of row r is r / n_tok)
};

// One unit of decode work: a run of pages of one block table, read for a set
// of branches ("members") that all hold those pages.
struct AttnItem {
  int32_t slot;        // block-table row the page ids come from
  int32_t page_begin;  // first logical page
  int32_t n_pages;
  int32_t n_tokens;    // valid keys in the run (the last page may be partial)
  int32_t member_base; // index of the first member in the members array
  int32_t n_members;
  int32_t split;       // partial slot this item writes
  int32_t flags;       // kItemReread | kItemWide
};
// a sibling item (another subgroup of the fork group) reads the same pages
constexpr int32_t kItemReread = 1;
// more than 64 stacked rows: the M = 128 tile
constexpr int32_t kItemWide = 2;
// more than 128 stacked rows: two M = 128 tiles of one CTA sharing every K/V
// stage (the merge's paired tile, merge_tc.cu)
constexpr int32_t kItemPair = 4;
// a decode step's own item whose last key is the row the step appends: its
// loader writes that row into the pool before loading the page (st_decode_step)
constexpr int32_t kItemAppend = 8;

// One CTA of a batched merge / prefill: rows [row_base, row_base + 256) of
// one sequence's stacked (new row, head) rows.
struct MergeItem {
  int32_t slot;
  int32_t L0;      // the sequence's length before this call
  int32_t T;       // rows appended to it
  int32_t q_row0;  // its first row in the call's Q / O / LSE
  int32_t row_base;
  int32_t pad[3];
};

struct AttnParams {
  const __nv_bfloat16* q;  // [L][n_rows_q][Hq][D]
  float* out_o;            // decode: partials [L][n_br][Hq][max_splits][D]; merge: [L][n_rows_q][Hq][D]
  float* out_lse;          // decode: [L][n_br][Hq][max_splits];              merge: [L][n_rows_q][Hq]
  const int32_t* table;
  const AttnItem* items;   // decode only
  const int32_t* members;  // decode only: branch index (in the call) of each member
  int32_t* status;
  int64_t n_blocks;
  float scale_log2;        // log2(e) / sqrt(D)
  int32_t n_rows_q;        // decode: n_br; merge: rows in Q (T, or all sequences' rows)
  int32_t Hq, Hkv, G, L, max_pages, max_splits;
  int32_t slot, L0, T;     // merge only: main's slot, length before the append, thought rows
  int32_t hold_loads;      // test hook (ST_FLAG_HOLD_LOADS): the loader issues nothing
  int32_t item_base;       // decode: CTA x reads item item_base + x
  int32_t keep_l2;         // decode: the launch's pages fit in L2; load them evict-normal so they stay
  const MergeItem* mitems; // batched merge: CTA x takes mitems[x] (slot, L0, T above unused)
  // decode step (items flagged kItemAppend): the rows the step appends,
  // [L][n_br][Hkv][D], and the pools they go to
  const __nv_bfloat16* app_k;
  const __nv_bfloat16* app_v;
  __nv_bfloat16* k_pool;
  __nv_bfloat16* v_pool;
};

struct CombineParams {
  const float* part_o;
  const float* part_lse;
  float* o;                 // [L][n_br][Hq][D]
  float* lse;               // [L][n_br][Hq]
  const int32_t* n_splits;  // [n_br]
  int32_t n_br, Hq, L, max_splits;
};

// Small per-call plans travel inside the kernel parameters (no staging copy,
// no event): a kernel reads its plan from here when the pointer in its
// parameter block is null.
constexpr int kInlineItems = 64;
constexpr int kInlineMembers = 96;
constexpr int kInlineBranches = 64;
struct InlineDecodePlan {
  AttnItem items[kInlineItems];
  int32_t members[kInlineMembers];
  int32_t n_splits[kInlineBranches];
};
// the part of a small plan the combine reads (a smaller parameter block to launch)
struct InlineSplits {
  int32_t n_splits[kInlineBranches];
};
constexpr int kInlineAppendBranches = 32;
constexpr int kInlineCows = 32;
struct InlineAppendPlan {
  AppendBranch branches[kInlineAppendBranches];
  CowCopy cows[kInlineCows];
};

// Programmatic dependent launch.  The small kernels of a decode step (table
// update, append, decode partials, combine) are launched so that each may be
// scheduled while its predecessor in the stream is still running: it does
// its setup that touches no global memory (barrier init, tensor-memory
// allocation), then griddep_wait() blocks until the predecessor grid has
// completed and its writes are visible.  Every global-memory access of these
// kernels comes after that wait, so stream order holds for their data; the
// wait returns at once when the kernel was launched without the attribute.
// A dependent grid is launched only after every CTA of its predecessor has
// signalled (or exited), so a waiting grid never keeps its predecessor's
// CTAs off the SMs.
__device__ __forceinline__ void griddep_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void griddep_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
cudaError_t launch_chained(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                           Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

cudaError_t launch_table_update(int32_t* table, const TableRun* runs, const int32_t* values,
                                int n_runs, cudaStream_t s);
cudaError_t launch_append(const AppendParams& p, const InlineAppendPlan* inl, int D, cudaStream_t s);
cudaError_t launch_combine(const CombineParams& p, const InlineSplits* inl, int D, cudaStream_t s);
// Decode partials on tcgen05 (one CTA per item x KV head x layer; items from
// p.item_base on; wide: the M = 128 tile, for items flagged kItemWide).
cudaError_t launch_decode_tc(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttnParams& p,
                             const InlineDecodePlan* inl, int n_items, int D, bool wide, cudaStream_t s);
// Causal merge prefill on tcgen05, two 128-row query tiles per CTA sharing
// K/V (merge_tc.cu): one sequence (p.slot, p.L0, p.T; p.mitems null) or a
// batch of n_items work items (p.mitems), p.q -> p.out_o, p.out_lse.
cudaError_t launch_merge_tc(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttnParams& p, int n_items,
                            int D, cudaStream_t s);
// Decode partials of fork groups of 129 to 256 stacked rows on the same
// paired tile (one CTA per item x KV head x layer, items from p.item_base on,
// launched as a programmatic dependent like the other decode kernels).
cudaError_t launch_decode_pair(const CUtensorMap& kmap, const CUtensorMap& vmap, const AttnParams& p,
                               const InlineDecodePlan* inl, int n_items, int D, cudaStream_t s);
// CTAs of the tcgen05 decode kernel resident per SM (0 on error).
int decode_tc_ctas_per_sm(int D);

}  // namespace st
