// C ABI of the fork-group attention library (declared in include/st.h).
//
// The host side is authoritative: the block pool (block_pool.cpp) decides
// every allocation, and each call turns its decision into a small plan that
// the kernels of that call consume -- inside their parameter block when it is
// small (the common decode step), else copied to the device through a pinned
// staging ring.  Planning for st_decode_attn groups the branches of a
// call by fork family and finds the pages they share, so the kernels read a
// shared prefix page once per group (Section 3.3 of the paper).
#include <cudaTypedefs.h>

#include <algorithm>
#include <climits>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <initializer_list>
#include <map>
#include <tuple>
#include <new>
#include <string>

#include <nvtx3/nvToolsExt.h>
#include <vector>

#include "../../include/st.h"
#include "block_pool.h"
#include "kernels.cuh"

using namespace st;

namespace {

constexpr int kStageSlots = 8;
constexpr size_t kStageSlotBytes = 2u << 20;  // 2 MiB per plan
constexpr int kMaxAttnRows = 64;              // stacked query rows of the narrow decode tile
constexpr int kMaxGqa = 48;                   // query heads per KV head
constexpr int kMaxWideRows = 128;             // ... of the wide one
constexpr int kMaxPairRows = 256;             // ... and of the paired tile

enum KernelId { kKTable = 0, kKAppend, kKDecode, kKCombine, kKMerge, kNumKernels };
const char* const kKernelNames[kNumKernels] = {"table_update", "append_kv", "decode_partial",
                                              "lse_combine", "merge_prefill"};

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

struct WorkspaceLayout {
  size_t status = 0, tables = 0, staging = 0, part_o = 0, part_lse = 0, total = 0;
};

bool config_valid(const st_config* c, std::string* why) {
  auto bad = [&](const char* m) {
    if (why) *why = m;
    return false;
  };
  if (!c) return bad("config is NULL");
  if (c->n_layers < 1) return bad("n_layers must be >= 1");
  if (c->n_kv_heads < 1 || c->n_q_heads < 1 || c->n_q_heads % c->n_kv_heads != 0)
    return bad("n_kv_heads must divide n_q_heads");
  if (c->n_q_heads / c->n_kv_heads > kMaxGqa) return bad("n_q_heads / n_kv_heads must be <= 48");
  if (c->head_dim != 64 && c->head_dim != 128) return bad("head_dim must be 64 or 128");
  if (c->page_size != kPageTokens) return bad("page_size must be 16");
  if (c->max_seqs < 1) return bad("max_seqs must be >= 1");
  if (c->max_pages < 1) return bad("max_pages must be >= 1");
  if (c->max_decode_branches < 1) return bad("max_decode_branches must be >= 1");
  if (c->max_splits < 2 || c->max_splits > 32) return bad("max_splits must be in [2, 32]");
  if (c->n_blocks < 1 || c->n_blocks > (int64_t)INT32_MAX) return bad("n_blocks out of range");
  if ((int64_t)c->n_layers * c->n_blocks >= (int64_t)INT32_MAX)
    return bad("n_layers * n_blocks must be < 2^31");
  if ((int64_t)c->n_kv_heads * kPageTokens > 65535) return bad("too many KV heads");
  return true;
}

WorkspaceLayout layout_for(const st_config* c) {
  WorkspaceLayout w;
  size_t off = 0;
  w.status = off;
  off = align_up(off + 64, 256);
  w.tables = off;
  off = align_up(off + (size_t)c->max_seqs * c->max_pages * sizeof(int32_t), 256);
  w.staging = off;
  off = align_up(off + (size_t)kStageSlots * kStageSlotBytes, 256);
  const size_t n_part = (size_t)c->max_decode_branches * c->n_layers * c->n_q_heads * c->max_splits;
  w.part_o = off;
  off = align_up(off + n_part * c->head_dim * sizeof(float), 256);
  w.part_lse = off;
  off = align_up(off + n_part * sizeof(float), 256);
  w.total = off;
  return w;
}

struct KStat {
  int64_t launches = 0;  // calls of this kind
  int64_t kernels = 0;   // device kernels they launched
  double ms = 0, bytes = 0, flops = 0;
  double overhead_bytes = 0;  // moved beyond the algorithmic bytes (split-KV partials, sibling re-reads)
};

struct PendingTiming {
  int kid;
  cudaEvent_t e0, e1;
};

// Plan writer over one staging slot: sub-allocations are 16-byte aligned and
// addressed by the same offset on the host (pinned) and the device side.
struct Plan {
  uint8_t* h = nullptr;
  uint8_t* d = nullptr;
  size_t cap = 0, off = 0;
  template <class T>
  T* alloc(size_t n, const T** dev) {
    off = align_up(off, 16);
    if (off + n * sizeof(T) > cap) return nullptr;
    T* hp = reinterpret_cast<T*>(h + off);
    *dev = reinterpret_cast<const T*>(d + off);
    off += n * sizeof(T);
    return hp;
  }
};

// The decode work decomposition of one st_decode_attn call (host only; the
// same plan st_decode_plan reports), filled by plan_decode below.
struct DecodePlan {
  std::vector<AttnItem> items;
  std::vector<int32_t> members;   // the call's branch index of each item's members
  std::vector<int32_t> n_splits;  // partials per branch
  // algorithmic, whole launch: every KV page once per fork family and layer
  // (shared pages once for the family, own pages once for their branch) and
  // the queries
  double bytes = 0, flops = 0;
  double reread_bytes = 0;        // second and later reads of a split family's pages
  double part_bytes = 0;          // the split-KV partials (written here, read by the combine)
  // scratch of the planner, kept between calls so that a decode step
  // allocates nothing on the host once its sizes have been seen
  struct Group { int32_t mbase, nmem, pages, family, tile; bool split, reread; };
  std::vector<Group> groups;
  std::vector<int32_t> fam_of, fam_ids, by_fam, shared, own_pages, own_tokens, ns, item_family, order;
  std::vector<AttnItem> sorted;
};

}  // namespace

struct st_pool {
  st_config cfg{};
  BlockPool* pool = nullptr;
  bool meta_only = false;
  int device = -1;
  __nv_bfloat16* k_pool = nullptr;
  __nv_bfloat16* v_pool = nullptr;
  uint8_t* ws = nullptr;
  WorkspaceLayout lay;
  int32_t* d_status = nullptr;
  int32_t* d_tables = nullptr;
  float* d_part_o = nullptr;
  float* d_part_lse = nullptr;
  CUtensorMap kmap{}, vmap{};
  int sms = 0, decode_ctas_per_sm = 0;
  int64_t l2_bytes = 0;
  // staging ring
  uint8_t* h_stage = nullptr;
  cudaEvent_t stage_ev[kStageSlots] = {};
  bool stage_used[kStageSlots] = {};
  int stage_next = 0;
  uint32_t stage_held = 0;  // slots taken by a call that has not retired them yet
  // Set when a CUDA call failed after the host tables had changed: the device
  // copy may then disagree with them, so every later call is refused.
  bool broken = false;
  // accounting
  bool timing = false;
  KStat stats[kNumKernels];
  std::vector<PendingTiming> pending;
  std::vector<cudaEvent_t> spare_events;
  std::string err;
  // host scratch of the calls, reused call after call
  DecodePlan plan;
  std::vector<int> call_slots;
  std::vector<int32_t> call_counts;
  std::vector<AppendBranch> app_branches;
  std::vector<CowEvent> app_cows;
};

namespace {

st_status fail(st_pool* P, st_status s, const char* fmt, ...) {
  if (P) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    P->err = buf;
  }
  return s;
}

#define CUDA_TRY(P, call)                                                                     \
  do {                                                                                        \
    cudaError_t e_ = (call);                                                                  \
    if (e_ != cudaSuccess)                                                                    \
      return fail((P), ST_ERR_CUDA, "%s failed: %s", #call, cudaGetErrorString(e_));          \
  } while (0)

// Makes the pool's device current for the duration of a call.
struct DeviceGuard {
  int prev = -1;
  bool changed = false;
  explicit DeviceGuard(int dev) {
    if (dev < 0) return;
    if (cudaGetDevice(&prev) == cudaSuccess && prev != dev) {
      if (cudaSetDevice(dev) == cudaSuccess) changed = true;
    }
  }
  ~DeviceGuard() {
    if (changed) cudaSetDevice(prev);
  }
};

bool decode_handle(st_pool* P, st_seq h, int* slot) {
  const int64_t s = h & 0xffffffffll;
  const uint32_t gen = (uint32_t)((uint64_t)h >> 32);
  if (s < 0 || s >= P->pool->max_seqs()) return false;
  const SeqSlot& ss = P->pool->slot((int)s);
  if (!ss.live || ss.gen != gen) return false;
  *slot = (int)s;
  return true;
}

st_seq make_handle(st_pool* P, int slot) {
  return (st_seq)(((uint64_t)P->pool->slot(slot).gen << 32) | (uint32_t)slot);
}

cudaEvent_t take_event(st_pool* P) {
  if (!P->spare_events.empty()) {
    cudaEvent_t e = P->spare_events.back();
    P->spare_events.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  cudaEventCreate(&e);
  return e;
}

// Marks the pool unusable after a failure that left host and device state
// apart (a CUDA error once the host tables had changed).
st_status poison(st_pool* P, st_status s) {
  P->broken = true;
  P->err = "pool unusable after: " + P->err;
  return s;
}

// Every call that changes or reads pool state starts here.
st_status refuse_if_broken(st_pool* P) {
  if (!P->broken) return ST_OK;
  P->err = "the pool is unusable after an earlier CUDA failure; destroy it";
  return ST_ERR_STATE;
}

// Launch wrapper: counts the launch (and the n_kernels device kernels it
// makes), adds its algorithmic bytes/flops and the bytes it moves beyond
// them, and brackets it with events when timing is on.  With
// ST_FLAG_FAIL_LAUNCH the launch is not made and reported as failed.
template <class F>
st_status run_kernel(st_pool* P, int kid, double bytes, double flops, cudaStream_t s, F&& launch,
                     int n_kernels = 1, double overhead_bytes = 0) {
  cudaEvent_t e0 = nullptr, e1 = nullptr;
  if (P->timing) {
    e0 = take_event(P);
    cudaEventRecord(e0, s);
  }
  const cudaError_t e = (P->cfg.flags & ST_FLAG_FAIL_LAUNCH) ? cudaErrorLaunchFailure : launch();
  if (e != cudaSuccess)
    return fail(P, ST_ERR_CUDA, "%s launch failed: %s", kKernelNames[kid], cudaGetErrorString(e));
  if (P->timing) {
    e1 = take_event(P);
    cudaEventRecord(e1, s);
    P->pending.push_back({kid, e0, e1});
  }
  KStat& k = P->stats[kid];
  k.launches += 1;
  k.kernels += n_kernels;
  k.bytes += bytes;
  k.flops += flops;
  k.overhead_bytes += overhead_bytes;
  return ST_OK;
}

// Takes the next staging slot that no unfinished call holds, waiting for the
// work that last used it.  The slot stays held until retire_plan or
// drop_plan.
st_status acquire_plan(st_pool* P, Plan* plan, int* slot_out) {
  int i = P->stage_next;
  while (P->stage_held & (1u << i)) i = (i + 1) % kStageSlots;  // at most two are ever held
  P->stage_next = (i + 1) % kStageSlots;
  if (P->stage_used[i]) CUDA_TRY(P, cudaEventSynchronize(P->stage_ev[i]));
  P->stage_held |= 1u << i;
  plan->h = P->h_stage + (size_t)i * kStageSlotBytes;
  plan->d = P->ws + P->lay.staging + (size_t)i * kStageSlotBytes;
  plan->cap = kStageSlotBytes;
  plan->off = 0;
  *slot_out = i;
  return ST_OK;
}

st_status submit_plan(st_pool* P, const Plan& plan, cudaStream_t s) {
  if (plan.off) CUDA_TRY(P, cudaMemcpyAsync(plan.d, plan.h, plan.off, cudaMemcpyHostToDevice, s));
  return ST_OK;
}

st_status retire_plan(st_pool* P, int slot, cudaStream_t s) {
  P->stage_held &= ~(1u << slot);
  CUDA_TRY(P, cudaEventRecord(P->stage_ev[slot], s));
  P->stage_used[slot] = true;
  return ST_OK;
}

// Gives back a slot that was taken but never written to the device.
void drop_plan(st_pool* P, int slot) {
  if (slot >= 0) P->stage_held &= ~(1u << slot);
}

// Bytes a plan of these arrays takes in a staging slot (16-byte aligned parts).
size_t plan_bytes(std::initializer_list<size_t> parts) {
  size_t off = 0;
  for (size_t b : parts) off = align_up(off, 16) + b;
  return off;
}

// Refresh the device copy of every block-table range the host changed.
st_status flush_tables(st_pool* P, cudaStream_t s) {
  BlockPool& bp = *P->pool;
  int slot = 0;
  const int n = bp.max_seqs();
  while (slot < n) {
    Plan plan;
    int ps;
    bool any = false;
    for (int i = slot; i < n; ++i)
      if (bp.slot(i).live && bp.slot(i).dirty_hi > bp.slot(i).dirty_lo) {
        any = true;
        break;
      }
    if (!any) return ST_OK;
    st_status st = acquire_plan(P, &plan, &ps);
    if (st != ST_OK) return st;
    // runs first (bounded count), then values
    const int max_runs = 4096;
    const TableRun* d_runs;
    TableRun* runs = plan.alloc<TableRun>(max_runs, &d_runs);
    const size_t vals_cap = (plan.cap - plan.off - 64) / sizeof(int32_t);
    const int32_t* d_vals;
    int32_t* vals = plan.alloc<int32_t>(vals_cap, &d_vals);
    int n_runs = 0;
    size_t n_vals = 0;
    for (; slot < n && n_runs < max_runs; ++slot) {
      SeqSlot& ss = bp.slot_mut(slot);
      if (!ss.live || ss.dirty_hi <= ss.dirty_lo) continue;
      const size_t cnt = (size_t)(ss.dirty_hi - ss.dirty_lo);
      const size_t room = vals_cap - n_vals;
      if (room == 0) break;
      const size_t take = std::min(cnt, room);
      runs[n_runs] = TableRun{(int64_t)slot * bp.max_pages() + ss.dirty_lo, (int32_t)take, (int32_t)n_vals};
      std::memcpy(vals + n_vals, ss.table.data() + ss.dirty_lo, take * sizeof(int32_t));
      n_vals += take;
      ++n_runs;
      ss.dirty_lo += (int32_t)take;
      if (ss.dirty_lo < ss.dirty_hi) break;  // slot only partly uploaded: continue it next round
      ss.dirty_lo = ss.dirty_hi = 0;
    }
    st = submit_plan(P, plan, s);
    if (st != ST_OK) return st;
    int32_t* tbl = P->d_tables;
    st = run_kernel(P, kKTable, (double)n_vals * 8 + n_runs * 16, 0, s,
                    [&] { return launch_table_update(tbl, d_runs, d_vals, n_runs, s); });
    if (st != ST_OK) return st;
    st = retire_plan(P, ps, s);
    if (st != ST_OK) return st;
  }
  return ST_OK;
}

bool aligned(const void* p, size_t a) { return ((uintptr_t)p % a) == 0; }

// Validates and performs an append (shared by st_append_kv, st_merge and
// st_prefill_batch).  Appends counts[i] rows to slots[i], in order (the same
// page allocation as appending to each sequence in turn); k, v: [L][sum of
// counts][Hkv][D].  All or nothing: capacity, the plan's size and its staging
// slot are settled before any table changes; a CUDA failure after that
// leaves the pool unusable (every later call returns ST_ERR_STATE).
// With `deferred` non-null (a decode step of one row per branch), the rows
// are left to the decode kernels when the append needs no copy-on-write:
// *deferred is then set and no append kernel is launched.
st_status do_append_rows(st_pool* P, const int* slots, const int32_t* counts, int n_br, const void* k,
                         const void* v, cudaStream_t s, bool* deferred = nullptr) {
  if (deferred) *deferred = false;
  BlockPool& bp = *P->pool;
  int64_t need = 0, n_rows = 0;
  int cow_bound = 0;  // branches whose append may start with a copy-on-write
  bool uniform = true;
  for (int i = 0; i < n_br; ++i) {
    if (!bp.fits(slots[i], counts[i]))
      return fail(P, ST_ERR_OOM, "sequence would exceed max_pages (%d)", bp.max_pages());
    need += bp.pages_needed(slots[i], counts[i]);
    n_rows += counts[i];
    uniform = uniform && counts[i] == counts[0];
    const SeqSlot& ss = bp.slot(slots[i]);
    if (counts[i] > 0 && ss.len % kPageTokens != 0 && bp.refcounts()[ss.table.back()] > 1) ++cow_bound;
  }
  if (need > bp.free_count())
    return fail(P, ST_ERR_OOM, "pool has %lld free pages, call needs %lld",
                (long long)bp.free_count(), (long long)need);
  if (n_rows > INT32_MAX) return fail(P, ST_ERR_INVALID, "too many rows in one call");
  // Small plans travel in the kernel parameters, larger ones through a
  // staging slot.  Copy-on-writes can only be fewer than cow_bound (an
  // earlier branch's copy may leave a later one the last holder).
  const bool may_stage = n_rows > 0 && !(n_br <= kInlineAppendBranches && cow_bound <= kInlineCows);
  if (may_stage && plan_bytes({n_br * sizeof(AppendBranch), std::max(cow_bound, 1) * sizeof(CowCopy)}) >
                       kStageSlotBytes)
    return fail(P, ST_ERR_INVALID, "append of %d sequences does not fit one plan slot", n_br);
  Plan plan;
  int ps = -1;
  if (may_stage && !P->meta_only) {
    st_status st = acquire_plan(P, &plan, &ps);
    if (st != ST_OK) return st;
  }

  // ---- from here on the host tables change ----------------------------------
  std::vector<AppendBranch>& brs = P->app_branches;
  brs.resize(n_br);
  int32_t row0 = 0;
  for (int i = 0; i < n_br; ++i) {
    brs[i] = AppendBranch{slots[i], (int32_t)bp.slot(slots[i]).len, row0, counts[i]};
    row0 += counts[i];
  }
  std::vector<CowEvent>& cows = P->app_cows;
  cows.clear();
  if (uniform) {
    bp.append(slots, n_br, n_br ? counts[0] : 0, &cows);
  } else {
    for (int i = 0; i < n_br; ++i) bp.append(&slots[i], 1, counts[i], &cows);
  }
  if (P->meta_only || n_rows == 0) return ST_OK;

  st_status st = flush_tables(P, s);
  if (st != ST_OK) return poison(P, st);
  if (deferred && cows.empty()) {
    drop_plan(P, ps);
    *deferred = true;
    return ST_OK;
  }
  const bool inline_plan = n_br <= kInlineAppendBranches && cows.size() <= (size_t)kInlineCows;
  InlineAppendPlan inl;
  const AppendBranch* d_br = nullptr;
  const CowCopy* d_cow = nullptr;
  if (inline_plan) {
    drop_plan(P, ps);
    ps = -1;
    for (int i = 0; i < n_br; ++i) inl.branches[i] = brs[i];
    for (size_t i = 0; i < cows.size(); ++i)
      inl.cows[i] = CowCopy{cows[i].src_block, cows[i].dst_block, cows[i].rows, 0};
  } else {
    AppendBranch* br = plan.alloc<AppendBranch>(n_br, &d_br);
    CowCopy* cw = plan.alloc<CowCopy>(std::max<size_t>(cows.size(), 1), &d_cow);
    for (int i = 0; i < n_br; ++i) br[i] = brs[i];
    for (size_t i = 0; i < cows.size(); ++i)
      cw[i] = CowCopy{cows[i].src_block, cows[i].dst_block, cows[i].rows, 0};
    st = submit_plan(P, plan, s);
    if (st != ST_OK) return poison(P, st);
  }
  const st_config& c = P->cfg;
  AppendParams ap{};
  ap.k = static_cast<const __nv_bfloat16*>(k);
  ap.v = static_cast<const __nv_bfloat16*>(v);
  ap.k_pool = P->k_pool;
  ap.v_pool = P->v_pool;
  ap.table = P->d_tables;
  ap.branches = d_br;
  ap.cows = d_cow;
  ap.status = P->d_status;
  ap.n_blocks = c.n_blocks;
  ap.n_cow = (int32_t)cows.size();
  ap.n_br = n_br;
  ap.n_tok = uniform && n_br ? counts[0] : 0;
  ap.L = c.n_layers;
  ap.Hkv = c.n_kv_heads;
  ap.max_pages = c.max_pages;
  ap.n_rows = (int32_t)n_rows;
  ap.ragged = uniform ? 0 : 1;
  // algorithmic: the new rows read and written once; the copy-on-write rows
  // are the bookkeeping's own traffic
  const double row_bytes = (double)c.n_layers * c.n_kv_heads * c.head_dim * 2 * 2;
  double cow_rows = 0;
  for (auto& e : cows) cow_rows += e.rows;
  st = run_kernel(P, kKAppend, row_bytes * (double)n_rows * 2, 0, s,
                  [&] { return launch_append(ap, inline_plan ? &inl : nullptr, c.head_dim, s); }, 1,
                  row_bytes * cow_rows * 2);
  if (st != ST_OK) return poison(P, st);
  if (!inline_plan) {
    st = retire_plan(P, ps, s);
    if (st != ST_OK) return poison(P, st);
  }
  return ST_OK;
}

st_status do_append(st_pool* P, const int* slots, int n_br, int n_tok, const void* k, const void* v,
                    cudaStream_t s) {
  P->call_counts.assign(n_br, n_tok);
  return do_append_rows(P, slots, P->call_counts.data(), n_br, k, v, s);
}

// Longest common prefix (in pages) of two block tables.
int32_t lcp_pages(const std::vector<int32_t>& a, const std::vector<int32_t>& b) {
  const size_t n = std::min(a.size(), b.size());
  size_t i = 0;
  while (i < n && a[i] == b[i]) ++i;
  return (int32_t)i;
}

void split_even(int32_t n, int32_t k, int32_t c, int32_t* begin, int32_t* count) {
  const int32_t base = n / k, rem = n % k;
  *begin = c * base + std::min(c, rem);
  *count = base + (c < rem ? 1 : 0);
}

}  // namespace

extern "C" {

ST_API const char* st_status_str(st_status s) {
  switch (s) {
    case ST_OK: return "ok";
    case ST_ERR_INVALID: return "invalid argument";
    case ST_ERR_OOM: return "out of pool pages or sequence slots";
    case ST_ERR_STATE: return "operation not possible in this state";
    case ST_ERR_CUDA: return "CUDA error";
    case ST_ERR_TIMEOUT: return "device wait timed out";
  }
  return "unknown status";
}

ST_API const char* st_last_error(st_pool* pool) { return pool ? pool->err.c_str() : ""; }

ST_API size_t st_workspace_bytes(const st_config* cfg) {
  if (!config_valid(cfg, nullptr)) return 0;
  return layout_for(cfg).total;
}

ST_API st_status st_pool_create(const st_config* cfg, void* k_pool, void* v_pool, void* workspace,
                                int device, st_pool** out) {
  if (!out) return ST_ERR_INVALID;
  *out = nullptr;
  std::string why;
  if (!config_valid(cfg, &why)) return ST_ERR_INVALID;
  st_pool* P = new (std::nothrow) st_pool();
  if (!P) return ST_ERR_OOM;
  P->cfg = *cfg;
  P->device = device;
  P->meta_only = device < 0;
  if (P->meta_only) {
    if (k_pool || v_pool || workspace) {
      delete P;
      return ST_ERR_INVALID;
    }
  } else {
    if (!k_pool || !v_pool || !workspace || !aligned(k_pool, 16) || !aligned(v_pool, 16) ||
        !aligned(workspace, 256)) {
      delete P;
      return ST_ERR_INVALID;
    }
  }
  P->pool = new (std::nothrow)
      BlockPool(cfg->n_blocks, cfg->seed, cfg->page_size, cfg->max_seqs, cfg->max_pages);
  if (!P->pool) {
    delete P;
    return ST_ERR_OOM;
  }
  if (P->meta_only) {
    *out = P;
    return ST_OK;
  }

  auto bail = [&](st_status s) {
    st_pool_destroy(P);
    return s;
  };
  DeviceGuard guard(device);
  int cur = -1;
  if (cudaGetDevice(&cur) != cudaSuccess || cur != device) return bail(ST_ERR_CUDA);
  P->k_pool = static_cast<__nv_bfloat16*>(k_pool);
  P->v_pool = static_cast<__nv_bfloat16*>(v_pool);
  P->ws = static_cast<uint8_t*>(workspace);
  P->lay = layout_for(cfg);
  P->d_status = reinterpret_cast<int32_t*>(P->ws + P->lay.status);
  P->d_tables = reinterpret_cast<int32_t*>(P->ws + P->lay.tables);
  P->d_part_o = reinterpret_cast<float*>(P->ws + P->lay.part_o);
  P->d_part_lse = reinterpret_cast<float*>(P->ws + P->lay.part_lse);
  if (cudaMemset(P->ws, 0, P->lay.staging) != cudaSuccess) return bail(ST_ERR_CUDA);
  if (cudaDeviceGetAttribute(&P->sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess)
    return bail(ST_ERR_CUDA);
  {
    int l2 = 0;
    if (cudaDeviceGetAttribute(&l2, cudaDevAttrL2CacheSize, device) != cudaSuccess) return bail(ST_ERR_CUDA);
    P->l2_bytes = l2;
  }
  P->decode_ctas_per_sm = decode_tc_ctas_per_sm(cfg->head_dim);
  if (P->decode_ctas_per_sm < 1) return bail(ST_ERR_CUDA);
  if (cudaHostAlloc(reinterpret_cast<void**>(&P->h_stage), (size_t)kStageSlots * kStageSlotBytes,
                    cudaHostAllocDefault) != cudaSuccess)
    return bail(ST_ERR_CUDA);
  for (int i = 0; i < kStageSlots; ++i)
    if (cudaEventCreateWithFlags(&P->stage_ev[i], cudaEventDisableTiming) != cudaSuccess)
      return bail(ST_ERR_CUDA);

  // Tensor maps over the pools: dims (64, D/64, 16*Hkv, L*n_blocks), so one
  // box {64, 1, 16, 1} is 16 tokens x 64 dims of one head = 2 KiB, loaded
  // with the 128-byte swizzle.
  PFN_cuTensorMapEncodeTiled_v12000 encode = nullptr;
  cudaDriverEntryPointQueryResult qres;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&encode),
                                       12000, cudaEnableDefault, &qres) != cudaSuccess ||
      qres != cudaDriverEntryPointSuccess || !encode)
    return bail(ST_ERR_CUDA);
  const int D = cfg->head_dim;
  cuuint64_t dims[4] = {64, (cuuint64_t)(D / 64), (cuuint64_t)kPageTokens * cfg->n_kv_heads,
                        (cuuint64_t)cfg->n_layers * (cuuint64_t)cfg->n_blocks};
  cuuint64_t strides[3] = {128, (cuuint64_t)D * 2, (cuuint64_t)kPageTokens * cfg->n_kv_heads * D * 2};
  cuuint32_t box[4] = {64, 1, kPageTokens, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  for (int t = 0; t < 2; ++t) {
    CUresult r = encode(t == 0 ? &P->kmap : &P->vmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4,
                        t == 0 ? k_pool : v_pool, dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return bail(ST_ERR_CUDA);
  }
  *out = P;
  return ST_OK;
}

ST_API st_status st_pool_destroy(st_pool* P) {
  if (!P) return ST_ERR_INVALID;
  if (!P->meta_only) {
    DeviceGuard guard(P->device);
    for (int i = 0; i < kStageSlots; ++i)
      if (P->stage_ev[i]) {
        cudaEventSynchronize(P->stage_ev[i]);
        cudaEventDestroy(P->stage_ev[i]);
      }
    for (auto& t : P->pending) {
      cudaEventDestroy(t.e0);
      cudaEventDestroy(t.e1);
    }
    for (auto e : P->spare_events) cudaEventDestroy(e);
    if (P->h_stage) cudaFreeHost(P->h_stage);
  }
  delete P->pool;
  delete P;
  return ST_OK;
}

ST_API st_status st_seq_create(st_pool* P, st_seq* out) {
  if (!P || !out) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  const int s = P->pool->create_seq();
  if (s < 0) return fail(P, ST_ERR_OOM, "no free sequence slot (max_seqs = %d)", P->cfg.max_seqs);
  *out = make_handle(P, s);
  return ST_OK;
}

// NVTX range around each public call that issues work (no cost unless a
// profiler is attached), so that ncu / nsys can filter by call.
struct NvtxRange {
  explicit NvtxRange(const char* name) { nvtxRangePushA(name); }
  ~NvtxRange() { nvtxRangePop(); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

ST_API st_status st_fork(st_pool* P, st_seq seq, int n_aux, st_seq* out_aux) {
  NvtxRange range_("st_fork");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  int slot;
  if (!decode_handle(P, seq, &slot)) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
  return st_fork_at(P, seq, P->pool->slot(slot).len, n_aux, out_aux);
}

ST_API st_status st_fork_at(st_pool* P, st_seq seq, int64_t length, int n_aux, st_seq* out_aux) {
  NvtxRange range_("st_fork_at");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  int slot;
  if (!decode_handle(P, seq, &slot)) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
  if (n_aux < 0 || (n_aux > 0 && !out_aux)) return fail(P, ST_ERR_INVALID, "bad n_aux/out_aux");
  if (length < 0 || length > P->pool->slot(slot).len)
    return fail(P, ST_ERR_INVALID, "fork point %lld outside [0, %lld]", (long long)length,
                (long long)P->pool->slot(slot).len);
  if (n_aux == 0) return ST_OK;
  std::vector<int> slots(n_aux);
  if (!P->pool->fork_at(slot, length, n_aux, slots.data()))
    return fail(P, ST_ERR_OOM, "fewer than %d free sequence slots", n_aux);
  for (int i = 0; i < n_aux; ++i) out_aux[i] = make_handle(P, slots[i]);
  return ST_OK;
}

ST_API st_status st_release(st_pool* P, st_seq seq) {
  NvtxRange range_("st_release");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  int slot;
  if (!decode_handle(P, seq, &slot)) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
  P->pool->release(slot);
  return ST_OK;
}

ST_API st_status st_append_kv(st_pool* P, const st_seq* br, int n_br, int n_tok, const void* k,
                              const void* v, void* stream) {
  NvtxRange range_("st_append_kv");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  if (n_br < 0 || n_tok < 0 || (n_br > 0 && !br)) return fail(P, ST_ERR_INVALID, "bad n_br/n_tok");
  std::vector<int>& slots = P->call_slots;
  slots.resize(n_br);
  for (int i = 0; i < n_br; ++i) {
    if (!decode_handle(P, br[i], &slots[i])) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
    for (int j = 0; j < i; ++j)
      if (slots[j] == slots[i]) return fail(P, ST_ERR_INVALID, "sequence listed twice");
  }
  if (P->meta_only) {
    if (k || v) return fail(P, ST_ERR_INVALID, "metadata-only pool takes no KV data");
  } else if (n_br > 0 && n_tok > 0 && (!k || !v || !aligned(k, 16) || !aligned(v, 16))) {
    return fail(P, ST_ERR_INVALID, "k and v must be 16-byte aligned device pointers");
  }
  if (n_br == 0 || n_tok == 0) return ST_OK;
  DeviceGuard guard(P->device);
  return do_append(P, slots.data(), n_br, n_tok, k, v, static_cast<cudaStream_t>(stream));
}

namespace {

// Plans one st_decode_attn call.  Branches are grouped by fork family and
// the full pages every member of a group holds (the longest common prefix of
// their block tables) are read once for all of them; each branch's own pages
// are read for it alone.  Runs of pages are sized to the SM count (about 64
// waves of two CTAs per SM, at least 16 pages), the tile shape follows the
// stacked rows (narrow up to 64, wide up to 128, paired up to 256, balanced
// paired subgroups beyond), and the items come out narrow first, then wide,
// then paired, longest first within each.
void plan_decode(st_pool* P, const std::vector<int>& slots, DecodePlan* out) {
  BlockPool& bp = *P->pool;
  const st_config& c = P->cfg;
  const int G = c.n_q_heads / c.n_kv_heads;
  const int n_br = (int)slots.size();
  DecodePlan& d = *out;
  // ---- group by fork family, find the shared full pages --------------------
  // by_fam: the call's branch indices ordered by family (families in order of
  // first appearance, branches in call order within one)
  d.fam_ids.clear();
  d.fam_of.assign(n_br, 0);
  for (int i = 0; i < n_br; ++i) {
    const int32_t f = bp.slot(slots[i]).family;
    int k = 0;
    while (k < (int)d.fam_ids.size() && d.fam_ids[k] != f) ++k;
    if (k == (int)d.fam_ids.size()) d.fam_ids.push_back(f);
    d.fam_of[i] = k;
  }
  d.by_fam.clear();
  for (int k = 0; k < (int)d.fam_ids.size(); ++k)
    for (int i = 0; i < n_br; ++i)
      if (d.fam_of[i] == k) d.by_fam.push_back(i);
  d.shared.assign(n_br, 0);  // pages of branch i read through its group
  d.groups.clear();
  d.members.clear();
  for (int k = 0, f0 = 0; k < (int)d.fam_ids.size(); ++k) {
    int nm = 0;
    while (f0 + nm < n_br && d.fam_of[d.by_fam[f0 + nm]] == k) ++nm;
    const int32_t* mem = d.by_fam.data() + f0;
    f0 += nm;
    // one narrow tile (<= 64 stacked rows), else one wide tile (<= 128), else
    // one paired tile (<= 256), else paired subgroups
    const int rows = nm * G;
    const int tile = rows <= kMaxAttnRows ? 0 : rows <= kMaxWideRows ? 1 : 2;
    const int per_group = std::max(1, (tile == 0 ? kMaxAttnRows : tile == 1 ? kMaxWideRows : kMaxPairRows) / G);
    // full pages held by every member of mem[b0, b1)
    auto common_pages = [&](int b0, int b1) {
      const SeqSlot& lead = bp.slot(slots[mem[b0]]);
      int64_t min_len = lead.len;
      int32_t pages = (int32_t)lead.table.size();
      for (int x = b0 + 1; x < b1; ++x) {
        const SeqSlot& ss = bp.slot(slots[mem[x]]);
        pages = std::min(pages, lcp_pages(lead.table, ss.table));
        min_len = std::min<int64_t>(min_len, ss.len);
      }
      return std::min<int32_t>(pages, (int32_t)(min_len / kPageTokens));
    };
    // A family larger than one tile is split into ceil(m / per_group)
    // subgroups of near-equal size (40 at 32 per tile: 20 + 20), every one
    // of them over the family's common pages, so that sibling items cover
    // the same runs and can be scheduled together.
    const int n_sub = (nm + per_group - 1) / per_group;
    const int32_t fam_pages = n_sub > 1 ? common_pages(0, nm) : 0;
    for (int sg = 0; sg < n_sub; ++sg) {
      const int b0 = sg * nm / n_sub, b1 = (sg + 1) * nm / n_sub;
      if (n_sub == 1 && b1 - b0 < 2) continue;  // a lone sequence reads its pages as its own
      const int32_t pages = n_sub > 1 ? fam_pages : common_pages(b0, b1);
      if (pages < 1) continue;
      // the family's pages are counted (as algorithmic bytes) with its first subgroup
      d.groups.push_back(DecodePlan::Group{(int32_t)d.members.size(), b1 - b0, pages, d.fam_ids[k], tile,
                                           n_sub > 1, sg > 0});
      for (int x = b0; x < b1; ++x) {
        d.members.push_back(mem[x]);
        d.shared[mem[x]] = pages;
      }
    }
  }

  // ---- chunking -------------------------------------------------------------
  int64_t total_pages = 0;
  for (const auto& g : d.groups) total_pages += g.pages;
  d.own_pages.resize(n_br);
  d.own_tokens.resize(n_br);
  for (int i = 0; i < n_br; ++i) {
    const SeqSlot& ss = bp.slot(slots[i]);
    d.own_pages[i] = (int32_t)ss.table.size() - d.shared[i];
    d.own_tokens[i] = (int32_t)(ss.len - (int64_t)d.shared[i] * kPageTokens);
    total_pages += d.own_pages[i];
  }
  const int64_t units = total_pages * c.n_kv_heads * c.n_layers;
  // a metadata-only pool has no device: it plans for a GB300 (152 SMs, two decode CTAs each)
  const int64_t slots_per_wave = (int64_t)(P->sms > 0 ? P->sms : 152) * (P->decode_ctas_per_sm > 0 ? P->decode_ctas_per_sm : 2);
  const int64_t target_ctas = 64 * slots_per_wave;
  int64_t chunk = (units + target_ctas - 1) / target_ctas;
  chunk = std::max<int64_t>(16, (chunk + 3) / 4 * 4);
  // Many short runs: each CTA pays a fixed cost (barriers, TMEM, its Q rows,
  // the partial write-out) per run, so once there are 8 waves or more of
  // them, runs are at least 16 stages long (batched serving: +4%).
  if (units / chunk >= 8 * slots_per_wave) chunk = std::max<int64_t>(chunk, 64);
  // leave room for a branch's own runs, but never fewer than one run for the prefix
  const int max_prefix_chunks = std::max(1, c.max_splits - 2);
  // CTAs the runs of a given length make (the items below, times heads and layers)
  auto ctas_for = [&](int64_t ch) {
    int64_t n = 0;
    d.ns.assign(n_br, 0);
    for (const auto& g : d.groups) {
      const int64_t k = std::min<int64_t>(max_prefix_chunks, (g.pages + ch - 1) / ch);
      n += k;
      for (int x = 0; x < g.nmem; ++x) d.ns[d.members[g.mbase + x]] = (int32_t)k;
    }
    for (int i = 0; i < n_br; ++i)
      if (d.own_pages[i] > 0) n += std::min<int64_t>(c.max_splits - d.ns[i], (d.own_pages[i] + ch - 1) / ch);
    return n * c.n_kv_heads * c.n_layers;
  };
  // A small launch (a few waves) whose last wave is less than half full: longer
  // runs (whole 4-page stages at a time) until a wave disappears, since a wave
  // costs a CTA's whole latency however few CTAs are in it.
  {
    const int64_t n0 = ctas_for(chunk), waves = (n0 + slots_per_wave - 1) / slots_per_wave;
    if (waves <= 4 && n0 % slots_per_wave != 0 && n0 % slots_per_wave < slots_per_wave / 2) {
      for (int64_t ch = chunk + 4; ch <= chunk + 64; ch += 4) {
        if ((ctas_for(ch) + slots_per_wave - 1) / slots_per_wave < waves) {
          chunk = ch;
          break;
        }
      }
    }
  }

  std::vector<AttnItem>& items = d.items;
  items.clear();
  d.item_family.clear();  // fork family of a subgroup's item, for scheduling siblings together
  d.n_splits.assign(n_br, 0);
  double bytes = 0, flops = 0, reread = 0;
  const double page_bytes = (double)kPageTokens * c.head_dim * 2 * 2;  // K+V, one head
  for (const auto& g : d.groups) {
    const int32_t k = (int32_t)std::min<int64_t>(max_prefix_chunks, (g.pages + chunk - 1) / chunk);
    const int32_t lead = d.members[g.mbase];
    for (int32_t cidx = 0; cidx < k; ++cidx) {
      int32_t b, n;
      split_even(g.pages, k, cidx, &b, &n);
      items.push_back(AttnItem{slots[lead], b, n, n * kPageTokens, g.mbase, g.nmem, cidx,
                               (g.split ? kItemReread : 0) | (g.tile == 1 ? kItemWide : g.tile == 2 ? kItemPair : 0)});
      d.item_family.push_back(g.family);
      (g.reread ? reread : bytes) += n * page_bytes;
      flops += 4.0 * g.nmem * G * n * kPageTokens * c.head_dim;
    }
    for (int x = 0; x < g.nmem; ++x) d.n_splits[d.members[g.mbase + x]] = k;
  }
  for (int i = 0; i < n_br; ++i) {
    if (d.own_pages[i] <= 0) continue;
    const int32_t room = c.max_splits - d.n_splits[i];
    const int32_t k = (int32_t)std::min<int64_t>(room, (d.own_pages[i] + chunk - 1) / chunk);
    const int32_t mbase = (int32_t)d.members.size();
    d.members.push_back(i);
    for (int32_t cidx = 0; cidx < k; ++cidx) {
      int32_t b, n;
      split_even(d.own_pages[i], k, cidx, &b, &n);
      const int32_t tok = std::min<int32_t>(n * kPageTokens, d.own_tokens[i] - b * kPageTokens);
      items.push_back(AttnItem{slots[i], d.shared[i] + b, n, tok, mbase, 1, d.n_splits[i] + cidx, 0});
      d.item_family.push_back(-1);
      bytes += n * page_bytes;
      flops += 4.0 * G * tok * c.head_dim;
    }
    d.n_splits[i] += k;
  }
  // narrow items, then wide ones, then paired ones (up to three launches);
  // within each, longest runs first so the short ones fill the tail, and the
  // items of a split group's subgroups over the same pages next to each other
  // (same length, family and first page), so that the second read hits L2.
  // A stable order: an insertion sort for the usual few dozen items.
  {
    auto key = [&](int i) {
      const AttnItem& a = items[i];
      const bool rr = (a.flags & kItemReread) != 0;
      return std::make_tuple((a.flags & kItemPair) ? 2 : (a.flags & kItemWide) ? 1 : 0, -a.n_pages, rr ? 0 : 1,
                             rr ? d.item_family[i] : 0, rr ? a.page_begin : 0);
    };
    const int n_items = (int)items.size();
    d.order.resize(n_items);
    for (int i = 0; i < n_items; ++i) d.order[i] = i;
    auto less = [&](int a, int b) { return key(a) < key(b); };
    if (n_items <= 128) {
      for (int i = 1; i < n_items; ++i) {
        const int v = d.order[i];
        int j = i;
        while (j > 0 && less(v, d.order[j - 1])) {
          d.order[j] = d.order[j - 1];
          --j;
        }
        d.order[j] = v;
      }
    } else {
      std::stable_sort(d.order.begin(), d.order.end(), less);
    }
    d.sorted.resize(n_items);
    for (int i = 0; i < n_items; ++i) d.sorted[i] = items[d.order[i]];
    items.swap(d.sorted);
  }
  bytes *= (double)c.n_kv_heads * c.n_layers;
  reread *= (double)c.n_kv_heads * c.n_layers;
  flops *= (double)c.n_kv_heads * c.n_layers;
  const double q_bytes = (double)c.n_layers * n_br * c.n_q_heads * c.head_dim * 2;
  double part_rows = 0;
  for (const auto& it : items) part_rows += (double)it.n_members * G;
  part_rows *= (double)c.n_kv_heads * c.n_layers;
  d.bytes = bytes + q_bytes;
  d.flops = flops;
  d.reread_bytes = reread;
  d.part_bytes = part_rows * (c.head_dim + 1) * 4;
}

// The call's branches as pool slots: live, each listed once, and (unless the
// call appends a row to each first) non-empty.
st_status decode_slots(st_pool* P, const st_seq* br, int n_br, std::vector<int>* slots, bool appends = false) {
  if (n_br < 1 || !br) return fail(P, ST_ERR_INVALID, "need at least one branch");
  if (n_br > P->cfg.max_decode_branches)
    return fail(P, ST_ERR_INVALID, "n_br %d > max_decode_branches %d", n_br, P->cfg.max_decode_branches);
  slots->assign(n_br, 0);
  for (int i = 0; i < n_br; ++i) {
    if (!decode_handle(P, br[i], &(*slots)[i])) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
    if (!appends && P->pool->slot((*slots)[i]).len < 1) return fail(P, ST_ERR_INVALID, "decode over an empty sequence");
    for (int j = 0; j < i; ++j)
      if ((*slots)[j] == (*slots)[i]) return fail(P, ST_ERR_INVALID, "sequence listed twice");
  }
  return ST_OK;
}

}  // namespace

namespace {

// The decode of st_decode_attn and st_decode_step over validated slots.  With
// app_k / app_v (a decode step whose append was deferred), the item that
// reads each branch's last page also writes the step's new row into it.
st_status decode_impl(st_pool* P, const std::vector<int>& slots, const void* q, float* o, float* lse,
                      cudaStream_t s, const void* app_k, const void* app_v) {
  const int n_br = (int)slots.size();
  const st_config& c = P->cfg;
  const int G = c.n_q_heads / c.n_kv_heads;
  DecodePlan& dp = P->plan;
  plan_decode(P, slots, &dp);
  if (app_k) {
    // each branch's last page is its own (a shared partial page would have
    // been copied), so exactly one single-member item holds it
    int marked = 0;
    for (AttnItem& it : dp.items) {
      if (it.n_members != 1) continue;
      const SeqSlot& ss = P->pool->slot(slots[dp.members[it.member_base]]);
      if (it.page_begin + it.n_pages == (int32_t)ss.table.size()) {
        it.flags |= kItemAppend;
        ++marked;
      }
    }
    if (marked != n_br) return fail(P, ST_ERR_STATE, "decode step: %d of %d new rows placed", marked, n_br);
  }
  const std::vector<AttnItem>& items = dp.items;
  const std::vector<int32_t>& members = dp.members;
  const std::vector<int32_t>& n_splits = dp.n_splits;
  const double bytes = dp.bytes, flops = dp.flops, part_bytes = dp.part_bytes;
  // small plans travel in the kernel parameters; larger ones through staging
  const bool inline_plan = items.size() <= (size_t)kInlineItems && members.size() <= (size_t)kInlineMembers &&
                           n_br <= kInlineBranches;
  if (!inline_plan && plan_bytes({items.size() * sizeof(AttnItem), members.size() * sizeof(int32_t),
                                  n_br * sizeof(int32_t)}) > kStageSlotBytes)
    return fail(P, ST_ERR_INVALID, "decode plan of %d items does not fit one plan slot", (int)items.size());
  // device tables that missed an upload would disagree with the host's
  st_status st = flush_tables(P, s);
  if (st != ST_OK) return poison(P, st);

  InlineDecodePlan inl;
  const AttnItem* d_items = nullptr;
  const int32_t* d_members = nullptr;
  const int32_t* d_nsplit = nullptr;
  Plan plan;
  int ps = -1;
  if (inline_plan) {
    std::memcpy(inl.items, items.data(), items.size() * sizeof(AttnItem));
    std::memcpy(inl.members, members.data(), members.size() * sizeof(int32_t));
    std::memcpy(inl.n_splits, n_splits.data(), n_br * sizeof(int32_t));
  } else {
    st = acquire_plan(P, &plan, &ps);
    if (st != ST_OK) return st;
    AttnItem* hi = plan.alloc<AttnItem>(items.size(), &d_items);
    int32_t* hm = plan.alloc<int32_t>(members.size(), &d_members);
    int32_t* hn = plan.alloc<int32_t>(n_br, &d_nsplit);
    std::memcpy(hi, items.data(), items.size() * sizeof(AttnItem));
    std::memcpy(hm, members.data(), members.size() * sizeof(int32_t));
    std::memcpy(hn, n_splits.data(), n_br * sizeof(int32_t));
    st = submit_plan(P, plan, s);
    if (st != ST_OK) {
      drop_plan(P, ps);
      return st;
    }
  }

  AttnParams ap{};
  ap.q = static_cast<const __nv_bfloat16*>(q);
  ap.out_o = P->d_part_o;
  ap.out_lse = P->d_part_lse;
  ap.table = P->d_tables;
  ap.items = d_items;
  ap.members = d_members;
  ap.status = P->d_status;
  ap.n_blocks = c.n_blocks;
  ap.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c.head_dim));
  ap.n_rows_q = n_br;
  ap.Hq = c.n_q_heads;
  ap.Hkv = c.n_kv_heads;
  ap.G = G;
  ap.L = c.n_layers;
  ap.max_pages = c.max_pages;
  ap.max_splits = c.max_splits;
  ap.hold_loads = (c.flags & ST_FLAG_HOLD_LOADS) ? 1 : 0;
  ap.app_k = static_cast<const __nv_bfloat16*>(app_k);
  ap.app_v = static_cast<const __nv_bfloat16*>(app_v);
  ap.k_pool = P->k_pool;
  ap.v_pool = P->v_pool;
  // a launch whose pages take less than half of L2 is one agent's step or a
  // few: the next step reads the same pages, so they stay in L2
  ap.keep_l2 = bytes < 0.5 * (double)P->l2_bytes ? 1 : 0;
  const int n_items = (int)items.size();
  int n_narrow = 0, n_wide = 0;
  while (n_narrow < n_items && !(items[n_narrow].flags & (kItemWide | kItemPair))) ++n_narrow;
  while (n_narrow + n_wide < n_items && (items[n_narrow + n_wide].flags & kItemWide)) ++n_wide;
  const int n_pair = n_items - n_narrow - n_wide;
  st = run_kernel(P, kKDecode, bytes, flops, s, [&] {
    const InlineDecodePlan* ip = inline_plan ? &inl : nullptr;
    cudaError_t e = launch_decode_tc(P->kmap, P->vmap, ap, ip, n_narrow, c.head_dim, false, s);
    if (e != cudaSuccess) return e;
    AttnParams aw = ap;
    aw.item_base = n_narrow;
    e = launch_decode_tc(P->kmap, P->vmap, aw, ip, n_wide, c.head_dim, true, s);
    if (e != cudaSuccess) return e;
    aw.item_base = n_narrow + n_wide;
    return launch_decode_pair(P->kmap, P->vmap, aw, ip, n_pair, c.head_dim, s);
  }, (n_narrow > 0 ? 1 : 0) + (n_wide > 0 ? 1 : 0) + (n_pair > 0 ? 1 : 0),
                  dp.reread_bytes + part_bytes);
  if (st != ST_OK) {
    if (ps >= 0) retire_plan(P, ps, s);  // its copy may still be in flight
    return st;
  }

  CombineParams cp{};
  cp.part_o = P->d_part_o;
  cp.part_lse = P->d_part_lse;
  cp.o = o;
  cp.lse = lse;
  cp.n_splits = d_nsplit;
  cp.n_br = n_br;
  cp.Hq = c.n_q_heads;
  cp.L = c.n_layers;
  cp.max_splits = c.max_splits;
  // algorithmic: O and LSE written once; the partials it reads are the split's own traffic
  const double cbytes = (double)c.n_layers * n_br * c.n_q_heads * (c.head_dim + 1) * 4;
  InlineSplits isp;
  if (inline_plan) std::memcpy(isp.n_splits, n_splits.data(), n_br * sizeof(int32_t));
  st = run_kernel(P, kKCombine, cbytes, 0, s,
                  [&] { return launch_combine(cp, inline_plan ? &isp : nullptr, c.head_dim, s); }, 1, part_bytes);
  if (st != ST_OK) {
    if (ps >= 0) retire_plan(P, ps, s);  // its copy may still be in flight
    return st;
  }
  return inline_plan ? ST_OK : retire_plan(P, ps, s);
}

}  // namespace

ST_API st_status st_decode_attn(st_pool* P, const st_seq* br, int n_br, const void* q, float* o,
                                float* lse, void* stream) {
  NvtxRange range_("st_decode_attn");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  if (P->meta_only) return fail(P, ST_ERR_STATE, "metadata-only pool has no KV storage");
  if (!q || !o || !lse || !aligned(q, 16) || !aligned(o, 16) || !aligned(lse, 4))
    return fail(P, ST_ERR_INVALID, "q/o/lse must be aligned device pointers");
  std::vector<int>& slots = P->call_slots;
  st_status vs = decode_slots(P, br, n_br, &slots);
  if (vs != ST_OK) return vs;
  DeviceGuard guard(P->device);
  return decode_impl(P, slots, q, o, lse, static_cast<cudaStream_t>(stream), nullptr, nullptr);
}

ST_API st_status st_decode_step(st_pool* P, const st_seq* br, int n_br, const void* k, const void* v,
                                const void* q, float* o, float* lse, void* stream) {
  NvtxRange range_("st_decode_step");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  if (P->meta_only) return fail(P, ST_ERR_STATE, "metadata-only pool has no KV storage");
  if (!k || !v || !q || !o || !lse || !aligned(k, 16) || !aligned(v, 16) || !aligned(q, 16) || !aligned(o, 16) ||
      !aligned(lse, 4))
    return fail(P, ST_ERR_INVALID, "k/v/q/o/lse must be aligned device pointers");
  std::vector<int>& slots = P->call_slots;
  st_status st = decode_slots(P, br, n_br, &slots, /*appends=*/true);
  if (st != ST_OK) return st;
  DeviceGuard guard(P->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  P->call_counts.assign(n_br, 1);
  bool deferred = false;
  st = do_append_rows(P, slots.data(), P->call_counts.data(), n_br, k, v, s, &deferred);
  if (st != ST_OK) return st;
  // the rows are in the host tables now: a failure from here on leaves the
  // device behind them
  st = decode_impl(P, slots, q, o, lse, s, deferred ? k : nullptr, deferred ? v : nullptr);
  return st == ST_OK ? ST_OK : poison(P, st);
}

ST_API st_status st_decode_plan(st_pool* P, const st_seq* br, int n_br, int32_t* items, int item_cap,
                                int32_t* members, int member_cap, int32_t* n_splits, int* n_items,
                                int* n_members) {
  if (!P) return ST_ERR_INVALID;
  std::vector<int>& slots = P->call_slots;
  st_status vs = decode_slots(P, br, n_br, &slots);
  if (vs != ST_OK) return vs;
  DecodePlan& dp = P->plan;
  plan_decode(P, slots, &dp);
  if (n_items) *n_items = (int)dp.items.size();
  if (n_members) *n_members = (int)dp.members.size();
  if (!items || !members || !n_splits || (int)dp.items.size() > item_cap || (int)dp.members.size() > member_cap)
    return fail(P, ST_ERR_INVALID, "the plan needs %d items and %d members", (int)dp.items.size(),
                (int)dp.members.size());
  for (size_t k = 0; k < dp.items.size(); ++k) {
    const AttnItem& a = dp.items[k];
    int owner = 0;
    while (slots[owner] != a.slot) ++owner;  // every slot of the plan is one of the call's branches
    int32_t* row = items + 8 * k;
    row[0] = owner;
    row[1] = a.page_begin;
    row[2] = a.n_pages;
    row[3] = a.n_tokens;
    row[4] = a.member_base;
    row[5] = a.n_members;
    row[6] = a.split;
    row[7] = a.flags;
  }
  std::memcpy(members, dp.members.data(), dp.members.size() * sizeof(int32_t));
  std::memcpy(n_splits, dp.n_splits.data(), (size_t)n_br * sizeof(int32_t));
  return ST_OK;
}

ST_API st_status st_merge(st_pool* P, st_seq main, int n_tok, const void* q, const void* k,
                          const void* v, float* o, float* lse, void* stream) {
  NvtxRange range_("st_merge");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  int slot;
  if (!decode_handle(P, main, &slot)) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
  if (n_tok < 0) return fail(P, ST_ERR_INVALID, "n_tok < 0");
  if (n_tok == 0) return ST_OK;  // nothing harvested: plain ReAct continues
  if (P->meta_only) {
    if (q || k || v || o || lse) return fail(P, ST_ERR_INVALID, "metadata-only pool takes no data");
    return do_append(P, &slot, 1, n_tok, nullptr, nullptr, nullptr);
  }
  if (!q || !k || !v || !o || !lse || !aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) ||
      !aligned(o, 16) || !aligned(lse, 4))
    return fail(P, ST_ERR_INVALID, "q/k/v/o/lse must be aligned device pointers");
  const st_config& c = P->cfg;
  const int64_t L0 = P->pool->slot(slot).len;
  DeviceGuard guard(P->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  st_status st = do_append(P, &slot, 1, n_tok, k, v, s);
  if (st != ST_OK) return st;
  const int G = c.n_q_heads / c.n_kv_heads;
  AttnParams ap{};
  ap.q = static_cast<const __nv_bfloat16*>(q);
  ap.out_o = o;
  ap.out_lse = lse;
  ap.table = P->d_tables;
  ap.status = P->d_status;
  ap.n_blocks = c.n_blocks;
  ap.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c.head_dim));
  ap.n_rows_q = n_tok;
  ap.Hq = c.n_q_heads;
  ap.Hkv = c.n_kv_heads;
  ap.G = G;
  ap.L = c.n_layers;
  ap.max_pages = c.max_pages;
  ap.max_splits = c.max_splits;
  ap.slot = slot;
  ap.L0 = (int32_t)L0;
  ap.T = n_tok;
  ap.hold_loads = (c.flags & ST_FLAG_HOLD_LOADS) ? 1 : 0;
  // algorithmic: main's KV once per (layer, head) + Q + O/LSE; flops: causal
  const double kv_bytes = (double)(L0 + n_tok) * c.n_kv_heads * c.head_dim * 2 * 2 * c.n_layers;
  const double io_bytes = (double)c.n_layers * n_tok * c.n_q_heads * (c.head_dim * 2 + c.head_dim * 4 + 4);
  const double keys = (double)n_tok * L0 + (double)n_tok * (n_tok + 1) / 2;
  const double flops = 4.0 * c.head_dim * keys * c.n_q_heads * c.n_layers;
  st = run_kernel(P, kKMerge, kv_bytes + io_bytes, flops, s,
                  [&] { return launch_merge_tc(P->kmap, P->vmap, ap, 0, c.head_dim, s); });
  return st == ST_OK ? ST_OK : poison(P, st);  // the rows are in, their prefill is not
}

ST_API st_status st_prefill_batch(st_pool* P, const st_seq* seqs, int n_seq, const int32_t* n_tok,
                                  const void* q, const void* k, const void* v, float* o, float* lse,
                                  void* stream) {
  NvtxRange range_("st_prefill_batch");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  if (n_seq < 0 || (n_seq > 0 && (!seqs || !n_tok))) return fail(P, ST_ERR_INVALID, "bad n_seq/seqs/n_tok");
  std::vector<int> slots;
  std::vector<int32_t> counts;
  std::vector<int> all(n_seq);
  int64_t R = 0;
  for (int i = 0; i < n_seq; ++i) {
    if (!decode_handle(P, seqs[i], &all[i])) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
    for (int j = 0; j < i; ++j)
      if (all[j] == all[i]) return fail(P, ST_ERR_INVALID, "sequence listed twice");
    if (n_tok[i] < 0) return fail(P, ST_ERR_INVALID, "n_tok[%d] < 0", i);
    if (n_tok[i] > 0) {
      slots.push_back(all[i]);
      counts.push_back(n_tok[i]);
      R += n_tok[i];
    }
  }
  if (R > INT32_MAX) return fail(P, ST_ERR_INVALID, "too many rows in one call");
  const st_config& c = P->cfg;
  const int G = c.n_q_heads / c.n_kv_heads;
  // work items: each sequence's stacked (row, head) rows in tiles of 256
  int64_t n_items64 = 0;
  for (size_t i = 0; i < slots.size(); ++i) n_items64 += ((int64_t)counts[i] * G + 255) / 256;
  if (plan_bytes({(size_t)n_items64 * sizeof(MergeItem)}) > kStageSlotBytes)
    return fail(P, ST_ERR_INVALID, "prefill of %lld row tiles does not fit one plan slot", (long long)n_items64);
  if (P->meta_only) {
    if (q || k || v || o || lse) return fail(P, ST_ERR_INVALID, "metadata-only pool takes no data");
    return do_append_rows(P, slots.data(), counts.data(), (int)slots.size(), nullptr, nullptr, nullptr);
  }
  if (R == 0) return ST_OK;
  if (!q || !k || !v || !o || !lse || !aligned(q, 16) || !aligned(k, 16) || !aligned(v, 16) ||
      !aligned(o, 16) || !aligned(lse, 4))
    return fail(P, ST_ERR_INVALID, "q/k/v/o/lse must be aligned device pointers");
  std::vector<int32_t> L0(slots.size());
  for (size_t i = 0; i < slots.size(); ++i) L0[i] = (int32_t)P->pool->slot(slots[i]).len;
  DeviceGuard guard(P->device);
  cudaStream_t s = static_cast<cudaStream_t>(stream);

  std::vector<MergeItem> items;
  double kv_bytes = 0, io_bytes = 0, keys = 0;
  int32_t q_row0 = 0;
  for (size_t i = 0; i < slots.size(); ++i) {
    const int64_t rows = (int64_t)counts[i] * G;
    for (int64_t rb = 0; rb < rows; rb += 256)
      items.push_back(MergeItem{slots[i], L0[i], counts[i], q_row0, (int32_t)rb, {0, 0, 0}});
    kv_bytes += (double)(L0[i] + counts[i]) * c.n_kv_heads * c.head_dim * 2 * 2 * c.n_layers;
    keys += (double)counts[i] * L0[i] + (double)counts[i] * (counts[i] + 1) / 2;
    q_row0 += counts[i];
  }
  // longest first (an item's work grows with the keys its rows see, L0 plus
  // its first token), so that the launch ends on short items, not on the
  // last tiles of a long context
  std::stable_sort(items.begin(), items.end(), [&](const MergeItem& x, const MergeItem& y) {
    return (int64_t)x.L0 + x.row_base / G > (int64_t)y.L0 + y.row_base / G;
  });
  io_bytes = (double)c.n_layers * R * c.n_q_heads * (c.head_dim * 2 + c.head_dim * 4 + 4);
  const double flops = 4.0 * c.head_dim * keys * c.n_q_heads * c.n_layers;
  Plan plan;
  int ps = -1;
  st_status st = acquire_plan(P, &plan, &ps);
  if (st != ST_OK) return st;
  st = do_append_rows(P, slots.data(), counts.data(), (int)slots.size(), k, v, s);
  if (st != ST_OK) {
    drop_plan(P, ps);  // nothing was written to it
    return st;
  }
  const MergeItem* d_items = nullptr;
  MergeItem* hi = plan.alloc<MergeItem>(items.size(), &d_items);
  std::memcpy(hi, items.data(), items.size() * sizeof(MergeItem));
  st = submit_plan(P, plan, s);
  if (st != ST_OK) return poison(P, st);
  AttnParams ap{};
  ap.q = static_cast<const __nv_bfloat16*>(q);
  ap.out_o = o;
  ap.out_lse = lse;
  ap.table = P->d_tables;
  ap.status = P->d_status;
  ap.n_blocks = c.n_blocks;
  ap.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c.head_dim));
  ap.n_rows_q = (int32_t)R;
  ap.Hq = c.n_q_heads;
  ap.Hkv = c.n_kv_heads;
  ap.G = G;
  ap.L = c.n_layers;
  ap.max_pages = c.max_pages;
  ap.max_splits = c.max_splits;
  ap.mitems = d_items;
  ap.hold_loads = (c.flags & ST_FLAG_HOLD_LOADS) ? 1 : 0;
  const int n_items = (int)items.size();
  st = run_kernel(P, kKMerge, kv_bytes + io_bytes, flops, s,
                  [&] { return launch_merge_tc(P->kmap, P->vmap, ap, n_items, c.head_dim, s); });
  const st_status rs = retire_plan(P, ps, s);
  if (st != ST_OK) return poison(P, st);
  return rs == ST_OK ? ST_OK : poison(P, rs);
}

ST_API st_status st_block_table(st_pool* P, st_seq seq, int32_t* out, int cap, int* n_pages,
                                int* n_tokens) {
  if (!P) return ST_ERR_INVALID;
  int slot;
  if (!decode_handle(P, seq, &slot)) return fail(P, ST_ERR_INVALID, "stale or unknown handle");
  const SeqSlot& ss = P->pool->slot(slot);
  if (n_pages) *n_pages = (int)ss.table.size();
  if (n_tokens) *n_tokens = (int)ss.len;
  if (out && cap > 0) {
    const int n = std::min<int>(cap, (int)ss.table.size());
    std::memcpy(out, ss.table.data(), n * sizeof(int32_t));
  }
  return ST_OK;
}

ST_API st_status st_refcounts(st_pool* P, int32_t* out, int64_t cap) {
  if (!P || !out) return ST_ERR_INVALID;
  const auto& r = P->pool->refcounts();
  const int64_t n = std::min<int64_t>(cap, (int64_t)r.size());
  std::memcpy(out, r.data(), n * sizeof(int32_t));
  return ST_OK;
}

ST_API st_status st_free_list(st_pool* P, int32_t* out, int64_t cap, int64_t* n) {
  if (!P) return ST_ERR_INVALID;
  std::vector<int32_t> fl;
  P->pool->free_list(&fl);
  if (n) *n = (int64_t)fl.size();
  if (out && cap > 0) std::memcpy(out, fl.data(), std::min<int64_t>(cap, (int64_t)fl.size()) * sizeof(int32_t));
  return ST_OK;
}

ST_API st_status st_sync(st_pool* P, void* stream) {
  NvtxRange range_("st_sync");
  if (!P) return ST_ERR_INVALID;
  if (st_status b_ = refuse_if_broken(P)) return b_;
  if (P->meta_only) return ST_OK;
  DeviceGuard guard(P->device);
  CUDA_TRY(P, cudaStreamSynchronize(static_cast<cudaStream_t>(stream)));
  int32_t code = 0;
  CUDA_TRY(P, cudaMemcpy(&code, P->d_status, sizeof code, cudaMemcpyDeviceToHost));
  if (code != 0) {
    CUDA_TRY(P, cudaMemset(P->d_status, 0, sizeof code));
    if (code == kDevTimeout) return fail(P, ST_ERR_TIMEOUT, "a device-side wait ran past its limit");
    if (code == kDevBadSmem) return fail(P, ST_ERR_CUDA, "a kernel's dynamic shared memory was not 1024-byte aligned");
    return fail(P, ST_ERR_INVALID, "a device-side bounds check failed (code %d)", code);
  }
  return ST_OK;
}

ST_API st_status st_profile_enable(st_pool* P, int enable) {
  if (!P) return ST_ERR_INVALID;
  P->timing = enable != 0 && !P->meta_only;
  return ST_OK;
}

ST_API st_status st_profile_read(st_pool* P, st_kernel_stat* out, int cap, int* n) {
  if (!P) return ST_ERR_INVALID;
  if (!P->meta_only) {
    DeviceGuard guard(P->device);
    for (auto& t : P->pending) {
      CUDA_TRY(P, cudaEventSynchronize(t.e1));
      float ms = 0;
      CUDA_TRY(P, cudaEventElapsedTime(&ms, t.e0, t.e1));
      P->stats[t.kid].ms += ms;
      P->spare_events.push_back(t.e0);
      P->spare_events.push_back(t.e1);
    }
    P->pending.clear();
  }
  int k = 0;
  for (int i = 0; i < kNumKernels; ++i) {
    if (k < cap && out) {
      std::memset(&out[k], 0, sizeof(st_kernel_stat));
      std::snprintf(out[k].name, sizeof out[k].name, "%s", kKernelNames[i]);
      out[k].launches = P->stats[i].launches;
      out[k].total_ms = P->stats[i].ms;
      out[k].bytes = P->stats[i].bytes;
      out[k].flops = P->stats[i].flops;
      out[k].kernels = P->stats[i].kernels;
      out[k].overhead_bytes = P->stats[i].overhead_bytes;
      ++k;
    }
    P->stats[i] = KStat{};
  }
  if (n) *n = k;
  return ST_OK;
}

}  // extern "C"
