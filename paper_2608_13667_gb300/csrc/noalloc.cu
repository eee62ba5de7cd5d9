// st_decode_attn_noalloc: decode attention over caller-owned paged KV that
// allocates no memory at all.
//
// Some callers cannot call cudaMalloc: code that runs inside a host
// framework which owns every device allocation and forbids new ones after
// start-up, real-time serving loops that must not allocate on the hot path,
// and plugins that are handed input and output pointers but no allocator.
// They cannot provide the workspace st_pool_create needs, so this entry
// point takes only inputs and outputs and keeps its scratch -- the per-call
// plan, a device copy of the page tables and the split-KV partials -- in the
// file-scope array below.  The kernels are the same ones st_decode_attn
// launches; only where the plan and the partials live differs.
//
// The array is ST_NOALLOC_SCRATCH_BYTES (16 MiB) per device and stays
// allocated on every GPU that loads the library until the process exits.
// Every call reuses it: calls that overlap on the GPU (different streams
// without ordering) race on it.  Nothing in it needs to start at zero: the
// plan and the page-table copy are uploaded whole by each call, and every
// partial slot the combine reads is written by that call's decode.  Device
// errors (a wait that ran out, a page id out of range) go to the caller's
// status word, which the call clears first.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstring>
#include <mutex>

#include "../../include/st.h"
#include "kernels.cuh"

using namespace st;

namespace {

constexpr size_t kScratchBytes = ST_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxBranches = ST_NOALLOC_MAX_BRANCHES;
constexpr int kMaxItems = 1024;
constexpr int kSplitStride = 16;  // partial slots per (layer, branch, head)
constexpr int kMaxRows = 64;      // stacked query rows per CTA (the narrow tile)
constexpr int kMaxGqa = 48;       // query heads per KV head, as for a pool
constexpr int kMaxDevices = 64;

static __device__ __align__(256) unsigned char g_noalloc_scratch[kScratchBytes];

// Per device, set up once (std::call_once, so two host threads making their
// first call together are safe): the device address of the array -- in host
// code the array's name is only a host-side stand-in, so the address comes
// from cudaGetSymbolAddress with that device current -- and the launch
// geometry the planner sizes runs by.
struct DeviceSetup {
  std::once_flag once;
  st_status status = ST_ERR_CUDA;
  void* scratch = nullptr;
  int sms = 0;
  int ctas_per_sm[2] = {};  // [head_dim == 128]
};
DeviceSetup g_dev[kMaxDevices];

size_t up256(size_t x) { return (x + 255) / 256 * 256; }

const DeviceSetup* setup_device(int dev) {
  if (dev < 0 || dev >= kMaxDevices) return nullptr;
  DeviceSetup& d = g_dev[dev];
  std::call_once(d.once, [&] {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return;
    if (cudaDeviceGetAttribute(&d.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return;
    d.ctas_per_sm[1] = decode_tc_ctas_per_sm(128);
    d.ctas_per_sm[0] = decode_tc_ctas_per_sm(64);
    if (d.ctas_per_sm[0] < 1 || d.ctas_per_sm[1] < 1) return;
    d.scratch = p;
    d.status = ST_OK;
  });
  return &d;
}

PFN_cuTensorMapEncodeTiled_v12000 lookup_encode() {
  PFN_cuTensorMapEncodeTiled_v12000 f = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", reinterpret_cast<void**>(&f), 12000,
                                       cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess)
    return nullptr;
  return f;
}

bool encode_map(CUtensorMap* map, const void* base, const st_config& c) {
  static const PFN_cuTensorMapEncodeTiled_v12000 encode = lookup_encode();  // initialised once, thread-safe
  if (!encode) return false;
  const int D = c.head_dim;
  cuuint64_t dims[4] = {64, (cuuint64_t)(D / 64), (cuuint64_t)kPageTokens * c.n_kv_heads,
                        (cuuint64_t)c.n_layers * (cuuint64_t)c.n_blocks};
  cuuint64_t strides[3] = {128, (cuuint64_t)D * 2, (cuuint64_t)kPageTokens * c.n_kv_heads * D * 2};
  cuuint32_t box[4] = {64, 1, kPageTokens, 1};
  cuuint32_t estr[4] = {1, 1, 1, 1};
  return encode(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base), dims, strides, box,
                estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

void split_even(int32_t n, int32_t k, int32_t c, int32_t* begin, int32_t* count) {
  const int32_t base = n / k, rem = n % k;
  *begin = c * base + std::min(c, rem);
  *count = base + (c < rem ? 1 : 0);
}

// Host-side plan, kept on the stack (fixed maximum sizes).
struct NoallocPlan {
  AttnItem items[kMaxItems];
  int32_t members[kMaxItems];
  int32_t n_splits[kMaxBranches];
};

}  // namespace

extern "C" ST_API st_status st_decode_attn_noalloc(const st_config* geom, const void* k_pool,
                                                   const void* v_pool, const int32_t* page_table,
                                                   int table_stride, const int32_t* seq_len, int n_br,
                                                   const void* q, float* o, float* lse, int32_t* status,
                                                   void* stream) {
  if (!geom || !k_pool || !v_pool || !page_table || !seq_len || !q || !o || !lse || !status)
    return ST_ERR_INVALID;
  const st_config& c = *geom;
  if (c.n_layers < 1 || c.n_kv_heads < 1 || c.n_q_heads % c.n_kv_heads != 0 ||
      c.n_q_heads / c.n_kv_heads > kMaxGqa || (c.head_dim != 64 && c.head_dim != 128) ||
      c.page_size != kPageTokens || c.n_blocks < 1 || (int64_t)c.n_layers * c.n_blocks >= INT32_MAX)
    return ST_ERR_INVALID;
  if (n_br < 1 || n_br > kMaxBranches || table_stride < 1) return ST_ERR_INVALID;
  if (((uintptr_t)k_pool | (uintptr_t)v_pool | (uintptr_t)q | (uintptr_t)o) % 16 != 0 ||
      ((uintptr_t)lse | (uintptr_t)status) % 4 != 0)
    return ST_ERR_INVALID;
  const int G = c.n_q_heads / c.n_kv_heads;
  for (int i = 0; i < n_br; ++i) {
    if (seq_len[i] < 1 || (int64_t)(seq_len[i] + kPageTokens - 1) / kPageTokens > table_stride)
      return ST_ERR_INVALID;
    const int32_t* t = page_table + (size_t)i * table_stride;
    for (int32_t p = 0; p < (seq_len[i] + kPageTokens - 1) / kPageTokens; ++p)
      if (t[p] < 0 || t[p] >= c.n_blocks) return ST_ERR_INVALID;
  }

  // scratch layout and its limit
  const size_t off_plan = 0;
  const size_t off_table = up256(off_plan + sizeof(NoallocPlan));
  const size_t off_part_o = up256(off_table + (size_t)n_br * table_stride * sizeof(int32_t));
  const size_t n_part = (size_t)c.n_layers * n_br * c.n_q_heads * kSplitStride;
  const size_t off_part_lse = up256(off_part_o + n_part * c.head_dim * sizeof(float));
  const size_t need = up256(off_part_lse + n_part * sizeof(float));
  if (need > kScratchBytes) return ST_ERR_OOM;  // beyond the static scratch: see the header

  int dev = -1;
  if (cudaGetDevice(&dev) != cudaSuccess) return ST_ERR_CUDA;
  const DeviceSetup* ds = setup_device(dev);
  if (!ds) return ST_ERR_INVALID;
  if (ds->status != ST_OK) return ds->status;
  unsigned char* scratch = static_cast<unsigned char*>(ds->scratch);

  // ---- plan: fork groups = branches whose tables start on the same page ----
  NoallocPlan plan;
  int32_t shared[kMaxBranches] = {};
  int32_t n_items = 0, n_members = 0;
  int64_t total_pages = 0;
  bool grouped[kMaxBranches] = {};
  struct Grp { int32_t first, count, pages; int32_t mem[kMaxRows]; };
  Grp groups[kMaxBranches];
  int n_groups = 0;
  const int per_group = std::max(1, kMaxRows / G);
  for (int i = 0; i < n_br; ++i) {
    if (grouped[i] || seq_len[i] < kPageTokens) continue;
    const int32_t* ti = page_table + (size_t)i * table_stride;
    Grp g{};
    g.mem[g.count++] = i;
    grouped[i] = true;
    int32_t min_len = seq_len[i];
    for (int j = i + 1; j < n_br && g.count < per_group; ++j) {
      if (grouped[j] || seq_len[j] < kPageTokens) continue;
      if (page_table[(size_t)j * table_stride] != ti[0]) continue;
      g.mem[g.count++] = j;
      grouped[j] = true;
      min_len = std::min(min_len, seq_len[j]);
    }
    if (g.count < 2) continue;
    int32_t pages = min_len / kPageTokens;
    for (int m = 1; m < g.count; ++m) {
      const int32_t* tj = page_table + (size_t)g.mem[m] * table_stride;
      int32_t p = 0;
      while (p < pages && tj[p] == ti[p]) ++p;
      pages = p;
    }
    if (pages < 1) continue;
    g.pages = pages;
    for (int m = 0; m < g.count; ++m) shared[g.mem[m]] = pages;
    groups[n_groups++] = g;
    total_pages += pages;
  }
  int32_t own_pages[kMaxBranches], own_tokens[kMaxBranches];
  for (int i = 0; i < n_br; ++i) {
    own_pages[i] = (seq_len[i] + kPageTokens - 1) / kPageTokens - shared[i];
    own_tokens[i] = seq_len[i] - shared[i] * kPageTokens;
    total_pages += own_pages[i];
    plan.n_splits[i] = 0;
  }
  const int64_t units = total_pages * c.n_kv_heads * c.n_layers;
  const int64_t target = (int64_t)32 * ds->sms * ds->ctas_per_sm[c.head_dim == 128];
  int64_t chunk = std::max<int64_t>(16, ((units + target - 1) / target + 3) / 4 * 4);
  for (int gi = 0; gi < n_groups; ++gi) {
    const Grp& g = groups[gi];
    const int32_t k = (int32_t)std::min<int64_t>(kSplitStride - 2, (g.pages + chunk - 1) / chunk);
    const int32_t mbase = n_members;
    for (int m = 0; m < g.count; ++m) plan.members[n_members++] = g.mem[m];
    for (int32_t ci = 0; ci < k; ++ci) {
      int32_t b, n;
      split_even(g.pages, k, ci, &b, &n);
      plan.items[n_items++] = AttnItem{g.mem[0], b, n, n * kPageTokens, mbase, g.count, ci, 0};
    }
    for (int m = 0; m < g.count; ++m) plan.n_splits[g.mem[m]] = k;
  }
  for (int i = 0; i < n_br; ++i) {
    if (own_pages[i] <= 0) continue;
    const int32_t room = kSplitStride - plan.n_splits[i];
    const int32_t k = (int32_t)std::min<int64_t>(room, (own_pages[i] + chunk - 1) / chunk);
    const int32_t mbase = n_members;
    plan.members[n_members++] = i;
    for (int32_t ci = 0; ci < k; ++ci) {
      int32_t b, n;
      split_even(own_pages[i], k, ci, &b, &n);
      const int32_t tok = std::min<int32_t>(n * kPageTokens, own_tokens[i] - b * kPageTokens);
      plan.items[n_items++] = AttnItem{i, shared[i] + b, n, tok, mbase, 1, plan.n_splits[i] + ci, 0};
    }
    plan.n_splits[i] += k;
  }

  CUtensorMap kmap, vmap;
  if (!encode_map(&kmap, k_pool, c) || !encode_map(&vmap, v_pool, c)) return ST_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // pageable host sources: the copies have consumed them when these calls return
  if (cudaMemsetAsync(status, 0, sizeof(int32_t), s) != cudaSuccess ||
      cudaMemcpyAsync(scratch + off_plan, &plan, sizeof plan, cudaMemcpyHostToDevice, s) != cudaSuccess ||
      cudaMemcpyAsync(scratch + off_table, page_table, (size_t)n_br * table_stride * sizeof(int32_t),
                      cudaMemcpyHostToDevice, s) != cudaSuccess)
    return ST_ERR_CUDA;

  NoallocPlan* dplan = reinterpret_cast<NoallocPlan*>(scratch + off_plan);
  AttnParams ap{};
  ap.q = static_cast<const __nv_bfloat16*>(q);
  ap.out_o = reinterpret_cast<float*>(scratch + off_part_o);
  ap.out_lse = reinterpret_cast<float*>(scratch + off_part_lse);
  ap.table = reinterpret_cast<const int32_t*>(scratch + off_table);
  ap.items = dplan->items;
  ap.members = dplan->members;
  ap.status = status;
  ap.n_blocks = c.n_blocks;
  ap.scale_log2 = (float)(1.4426950408889634 / std::sqrt((double)c.head_dim));
  ap.n_rows_q = n_br;
  ap.Hq = c.n_q_heads;
  ap.Hkv = c.n_kv_heads;
  ap.G = G;
  ap.L = c.n_layers;
  ap.max_pages = table_stride;
  ap.max_splits = kSplitStride;
  ap.hold_loads = (c.flags & ST_FLAG_HOLD_LOADS) ? 1 : 0;
  if (launch_decode_tc(kmap, vmap, ap, nullptr, n_items, c.head_dim, false, s) != cudaSuccess) return ST_ERR_CUDA;
  CombineParams cp{};
  cp.part_o = ap.out_o;
  cp.part_lse = ap.out_lse;
  cp.o = o;
  cp.lse = lse;
  cp.n_splits = dplan->n_splits;
  cp.n_br = n_br;
  cp.Hq = c.n_q_heads;
  cp.L = c.n_layers;
  cp.max_splits = kSplitStride;
  if (launch_combine(cp, nullptr, c.head_dim, s) != cudaSuccess) return ST_ERR_CUDA;
  return ST_OK;
}
