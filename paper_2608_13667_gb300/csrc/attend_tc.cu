// Fork-group decode partials on the 5th-generation tensor cores (tcgen05,
// accumulators in tensor memory).  The merge prefill is in merge_tc.cu.
//
// Section 3.3 of the paper: every branch receives the snapshot H_t + R_t, so
// the prefix KV is shared by all decoding streams; Section 4.4: branch load
// is dominated by those cached-prefix reads.  A decode CTA owns one run of
// pages of one KV head of one layer and stacks every query row that reads
// it -- for a shared prefix all branches of the fork group x the G query
// heads of the KV head (<= 64 rows) -- so each prefix page crosses HBM once
// per group.
//
// Two tile shapes (Section 3.2 lets the branch count vary, so the stacked
// row count n_b G does):
//   narrow  S at M = 64, up to 64 rows (the paper's 1 + 4 branches at
//           G <= 12); P goes to shared memory over the stage's consumed K
//           slot, its two bf16 terms stacked as the 128 A rows of one P V
//   wide    M = 128, up to 128 rows; P stays in TMEM over its own scores and
//           P V reads it from there (no P in shared memory, so two CTAs still
//           fit an SM).
// A group of 129 to 256 rows runs on the merge kernel's paired tile
// (merge_tc.cu); a larger one is split into paired subgroups whose items over
// the same pages run next to each other, so the second read of a page comes
// from L2.
//
// CTA layout (192 threads, 2 CTAs per SM):
//   warps 0..3  softmax (only those with rows run).  Narrow: row r's scores
//               sit in TMEM lane 32 (r / 16) + r % 16, and threads t and
//               t + 16 of a warp share row t, each with half of the stage's
//               keys (16-lane TMEM loads with a column split); thread t owns
//               the lane of the row's O_hi, thread t + 16 the lane 16 higher,
//               which holds O_lo.  Wide: thread r owns row r = TMEM lane r.
//               A thread loads its part of its Q row into shared memory;
//               per stage it reads its
//               scores from TMEM, masks keys past the run, keeps a running max
//               (narrow: combined with its partner by one shuffle) that is
//               raised only when a score exceeds it by more than 2^8 (O in
//               TMEM is then rescaled in place), and writes P = 2^(s - m) as
//               two bf16 terms.  At the end it normalises O out of TMEM: a
//               split-KV partial with its log-sum-exp.
//   warp 4      loader: page ids from the block table (32 per read, one batch
//               ahead), one 2 KiB TMA copy per (page, 64-wide half of D, K|V)
//               into a ring of stages, per-stage mbarriers with byte counts;
//               a stage's copies are issued by the warp's lanes together.
//               Narrow: one ring of three stages, a stage's K and V slots
//               freed together after its P V.  Wide: K and V have their own
//               rings of two slots and barriers; a K slot is freed by the
//               commit after S_j, a V slot after P_j V_j.
//               A decode step (st_decode_step): the narrow item that holds a
//               branch's last page first stores the step's new K and V row of
//               its (layer, KV head) into that page, then a proxy fence makes
//               the store visible to the page's TMA copies.  Only that CTA
//               reads the page (a branch's last page is its own), so no
//               separate append launch is needed.
//   warp 5      TMEM owner; lane 0 issues   S = Q K^T  (M, N=64 keys)
//               and O += P V (M = 128, N=D) and commits them to mbarriers.  S is
//               double-buffered in TMEM: S_{j+1} is issued before P_j V_j when
//               its data has landed, so the softmax of stage j+1 overlaps the
//               tensor work of stage j.
//               A rescale of O first waits for the commit of P_{j-1} V_{j-1}.
//
// The kernel is launched as a programmatic dependent of the append before it
// in the stream: the TMEM allocation comes before griddepcontrol.wait, every
// global-memory access after it.
//
// Shared-memory operands use the 128-byte swizzle (8-row x 128-byte atoms):
//   Q  [D/64][rows][64]       K-major A (SBO 1024)
//   K  [D/64][keys][64]       K-major B (SBO 1024)
//   P  [128][keys]            narrow: K-major A (SBO 1024), written over K:
//                             P_hi of row r at A row 32 (r / 16) + r % 16,
//                             P_lo at the A row 16 higher
//                             wide: in TMEM, the 16 score columns of keys
//                             [16 k, 16 k + 16) holding P_hi and P_lo of them
//   V  [D/64][keys][64]       MN-major B (LBO = one D-half, SBO 1024)
// The narrow P V reads 128 A rows of which only those of real rows are
// written; the others read whatever is in shared memory and only produce
// accumulator rows that nobody reads (each output row depends on its own A
// row only).  V rows of keys that are not valid (past the run,
// or in pages a short last stage did not load) are zeroed before P V, so
// stale shared or pool memory cannot turn 0 * x into NaN in a real row.
#include <math.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace st {

namespace {

constexpr int kLoadWarp = 4, kMmaWarp = 5;
constexpr int kThreads = 6 * 32;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kTmemS = 0, kTmemO = 128;  // S buffers at 0 and 64
constexpr float kRescaleThreshold = 8.f;  // log2 units
constexpr float kLn2 = 0.69314718055994530942f;
constexpr int kMaxDevices = 64;

constexpr int cmax(int a, int b) { return a > b ? a : b; }

template <int D, bool kWide>
struct TcCfg {
  static constexpr int kHalves = D / 64;
  static constexpr int kKeys = 64;                     // keys per stage
  static constexpr int kPagesPerStage = kKeys / kPageTokens;
  // Wide: P lives in TMEM, so a K slot is free once S_j has been computed and
  // K and V slots recycle separately (K and V barrier rings).  Narrow: P goes
  // over K_j, the two are released together after P_j V_j (one ring of
  // stages).
  static constexpr int kStages = kWide ? 2 : 3;         // K slots
  static constexpr int kVStages = kWide ? 2 : kStages;  // V slots
  static constexpr bool kSplitKV = kWide;
  // S at M = 64 for <= 64 stacked rows: score rows sit in TMEM lanes 0..15
  // of each warp's 32-lane quarter (row r at lane 32 (r / 16) + r % 16);
  // M = 128 for up to 128 rows (row r at lane r)
  static constexpr int kM = kWide ? 128 : 64;
  static constexpr int kRowsPerWarp = kM / 4;
  static constexpr int kQRows = kWide ? 128 : 64;      // Q rows stored
  static constexpr int kQHalfBytes = kQRows * 128;
  static constexpr int kQBytes = kHalves * kQHalfBytes;
  static constexpr int kKVHalfBytes = kKeys * 128;
  // P as two bf16 terms (P = P_hi + P_lo, both against the same V): the
  // rounding of a single bf16 P does not average out when a row sees few
  // keys or its weights are peaked.  Narrow: the two terms are the A rows of
  // one M = 128 product O += [P_hi; P_lo] V, written over the K slot --
  // P_hi of row r at A row 32 (r / 16) + r % 16 (the lane of r's scores),
  // P_lo at A row 32 (r / 16) + 16 + r % 16, the lanes M = 64 leaves free in
  // each warp's quarter -- so the accumulator holds O_hi of row r in one lane
  // and O_lo in the lane 16 above it, summed at the end.
  static constexpr int kMo = 128;                                  // M of P V
  static constexpr int kPBytes = kWide ? 0 : kMo * 128;           // the A rows of P V
  static constexpr int kKSlotBytes = cmax(kHalves * kKVHalfBytes, kPBytes);
  static constexpr int kVSlotBytes = kHalves * kKVHalfBytes;
  // the K slots, then the V slots
  static constexpr int kKRingBytes = kStages * kKSlotBytes;
  static constexpr int kRingBytes = kKRingBytes + kVStages * kVSlotBytes;
  static constexpr int kBarOffset = kQBytes + kRingBytes;
  // no alignment slack: two narrow CTAs of 64 rows fill an SM's shared
  // memory, so the kernel requires the dynamic shared memory to start on a
  // 1024-byte boundary (it does when a kernel has no static shared memory;
  // the kernel checks and reports ST_ERR_CUDA otherwise)
  static constexpr int kSmemBytes = kBarOffset + 256;
};

template <int D, bool kWide, bool kElect>
__global__ void __launch_bounds__(kThreads, 2)
    attend_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                     const AttnParams p, const __grid_constant__ InlineDecodePlan inl) {
  using C = TcCfg<D, kWide>;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if (smem_addr(smem_raw) & 1023u) {  // the 128-byte swizzle needs 1024-byte aligned operands
    griddep_wait();
    if (threadIdx.x == 0) atomicCAS(p.status, 0, kDevBadSmem);
    return;
  }
  uint8_t* base = smem_raw;
  uint8_t* q_s = base;
  uint8_t* ring = base + C::kQBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::kBarOffset);
  uint64_t* full = bars;                 // [kStages] K (and, narrow, V) landed
  uint64_t* empty = bars + C::kStages;   // [kStages] K (and, narrow, V) slot free
  // K slot s and V slot s (narrow: the K and V of stage s)
  auto k_slot = [&](int s) { return ring + s * C::kKSlotBytes; };
  auto v_slot = [&](int s) { return ring + C::kKRingBytes + s * C::kVSlotBytes; };
  uint64_t* s_full = bars + 2 * C::kStages;   // [2] per S buffer
  uint64_t* p_full = s_full + 2;              // [2] per S buffer
  uint64_t* o_ready = s_full + 4;             // one phase per P V
  uint64_t* o_final = s_full + 5;
  uint64_t* q_ready = s_full + 6;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(s_full + 7);
  uint64_t* v_full = s_full + 8;               // [kVStages] wide: V landed
  uint64_t* v_empty = v_full + C::kVStages;    // [kVStages] wide: V slot free

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int kvh = blockIdx.y;
  const int layer = blockIdx.z;
  const int G = p.G;
  // the tensor-memory allocation touches no global memory: ahead of the wait
  // for the previous kernel in the stream (the append that wrote the pages)
  if (warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
  griddep_wait();
  griddep_launch_dependents();

  // ---- what this CTA reads and for whom ------------------------------------------
  const int32_t* members = p.members ? p.members : inl.members;
  const int item_idx = p.item_base + blockIdx.x;
  const AttnItem item = p.items ? p.items[item_idx] : inl.items[item_idx];
  const int slot = item.slot;
  const int page_begin = item.page_begin;
  const int n_pages = item.n_pages;
  const int n_valid_keys = item.n_tokens;
  const int n_rows = item.n_members * G;
  const int n_tiles = (n_pages + C::kPagesPerStage - 1) / C::kPagesPerStage;
  const int n_sw = (n_rows + C::kRowsPerWarp - 1) / C::kRowsPerWarp;  // softmax warps with rows
  const int n_swt = n_sw * 32;

  if (threadIdx.x == 0) {
    for (int s = 0; s < C::kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    if (C::kSplitKV) {
      for (int s = 0; s < C::kVStages; ++s) {
        mbar_init(&v_full[s], 1);
        mbar_init(&v_empty[s], 1);
      }
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(&s_full[b], 1);
      mbar_init(&p_full[b], n_swt);
    }
    mbar_init(o_ready, 1);
    mbar_init(o_final, 1);
    mbar_init(q_ready, n_swt);
    fence_mbar_init();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  // ---- loader --------------------------------------------------------------------
  if (warp == kLoadWarp) {
    if (!kWide && (item.flags & kItemAppend)) {
      // a decode step: this run's last key is the row the step appends.  The
      // warp writes this (layer, KV head)'s K and V of it into the pool (16
      // bytes per lane) before anything else, so the row is stored even if a
      // wait of this CTA runs out later, and makes the writes visible to the
      // TMA copy that loads the page.
      const int last = n_valid_keys - 1;  // key within the run
      const int blk = p.table[(int64_t)slot * p.max_pages + page_begin + last / kPageTokens];
      constexpr int kChunks = D / 8;
      if (lane < 2 * kChunks) {
        if ((uint64_t)blk >= (uint64_t)p.n_blocks) {
          atomicCAS(p.status, 0, kDevBadIndex);
        } else {
          const bool is_v = lane >= kChunks;
          const int c = lane % kChunks;
          const int64_t src = (((int64_t)layer * p.n_rows_q + members[item.member_base]) * p.Hkv + kvh) * D + c * 8;
          const int64_t dst =
              ((((int64_t)layer * p.n_blocks + blk) * p.Hkv + kvh) * kPageTokens + last % kPageTokens) * D + c * 8;
          *reinterpret_cast<uint4*>((is_v ? p.v_pool : p.k_pool) + dst) =
              *reinterpret_cast<const uint4*>((is_v ? p.app_v : p.app_k) + src);
          fence_proxy_async_global();
        }
      }
      __syncwarp();
    }
    if (p.hold_loads) return;  // test hook: nothing arrives, the other roles' waits run out
    if (lane == 0) {
      prefetch_tensormap(&kmap);
      prefetch_tensormap(&vmap);
    }
    // a page is streamed once, unless a sibling item (the group's other
    // subgroup, scheduled next to this one) reads it too, or the whole launch
    // fits in L2 (one agent's step, read again by the next step): then keep it
    const uint64_t policy =
        (p.keep_l2 || (item.flags & kItemReread)) ? l2_policy_evict_normal() : l2_policy_evict_first();
    const int32_t* ids = p.table + (int64_t)slot * p.max_pages + page_begin;
    int base_id = 0;
    int cur = lane < n_pages ? ids[lane] : 0;
    int nxt = 32 + lane < n_pages ? ids[32 + lane] : 0;
    // waits for the slot of stage j in a ring of `depth` slots to be
    // released (lane 0 waits)
    auto slot_free = [&](uint64_t* ring_empty, int depth, int j) -> bool {
      int w = 1;
      if (j >= depth && lane == 0) w = mbar_wait(&ring_empty[j % depth], ((j / depth) - 1) & 1) ? 1 : 0;
      return __shfl_sync(0xffffffffu, w, 0) != 0;
    };
    // pages of stage j (j increasing): the count and the TMA page coordinates
    auto stage_pages = [&](int j, int* c3) -> int {
      const int page0 = j * C::kPagesPerStage;
      if (page0 >= base_id + 32) {
        base_id += 32;
        cur = nxt;
        nxt = base_id + 32 + lane < n_pages ? ids[base_id + 32 + lane] : 0;
      }
      const int np = min(C::kPagesPerStage, n_pages - page0);
#pragma unroll
      for (int q = 0; q < C::kPagesPerStage; ++q) {
        int b = __shfl_sync(0xffffffffu, cur, (page0 - base_id + q) & 31);
        if (q < np && (uint64_t)b >= (uint64_t)p.n_blocks) {
          if (lane == 0) atomicCAS(p.status, 0, kDevBadIndex);
          b = 0;
        }
        c3[q] = layer * (int)p.n_blocks + b;
      }
      return np;
    };
    // wide: np pages of one operand into a slot, completing on bar, one copy
    // per lane (lane = D/64 q + h), after lane 0's expect-tx
    const uint32_t page_bytes = (uint32_t)(C::kHalves * kPageTokens * 128);
    auto issue = [&](const CUtensorMap* map, uint8_t* dst, uint64_t* bar, const int* c3, int np) {
      __syncwarp();
      const int q = lane / C::kHalves, h = lane % C::kHalves;
      int cq = c3[0];
#pragma unroll
      for (int i = 1; i < C::kPagesPerStage; ++i)
        if (q == i) cq = c3[i];
      if (lane < C::kHalves * np)
        tma_load_4d(dst + h * C::kKVHalfBytes + q * kPageTokens * 128, map, bar, 0, h, kvh * kPageTokens, cq,
                    policy);
    };
    int jk = 0, jv = 0;  // stages whose K and V copies have been issued
    bool ok = true;
    for (; jk < n_tiles; ++jk) {
      const int s = jk % C::kStages;
      if (!slot_free(empty, C::kStages, jk)) {
        ok = false;
        break;
      }
      uint8_t* kst = k_slot(s);
      if constexpr (C::kSplitKV) {
        int c3[C::kPagesPerStage];
        const int np = stage_pages(jk, c3);
        if (lane == 0) mbar_arrive_expect_tx(&full[s], np * page_bytes);
        issue(&kmap, kst, &full[s], c3, np);
        // the K slot was released by S_j-kStages, the V slot waits for P_j-kVStages V_j-kVStages
        const int sv = jk % C::kVStages;
        if (!slot_free(v_empty, C::kVStages, jk)) {
          ok = false;
          ++jk;  // K_j is in flight
          break;
        }
        if (lane == 0) mbar_arrive_expect_tx(&v_full[sv], np * page_bytes);
        issue(&vmap, v_slot(sv), &v_full[sv], c3, np);
        jv = jk + 1;
      } else {
        uint8_t* vst = v_slot(s);
        const int page0 = jk * C::kPagesPerStage;
        if (page0 >= base_id + 32) {
          base_id += 32;
          cur = nxt;
          nxt = base_id + 32 + lane < n_pages ? ids[base_id + 32 + lane] : 0;
        }
        const int np = min(C::kPagesPerStage, n_pages - page0);
        if (lane == 0) mbar_arrive_expect_tx(&full[s], 2 * np * page_bytes);
        __syncwarp();
        // one copy per lane (lane = 2 D/64 q + (V ? D/64 : 0) + h): a single
        // thread issuing them one after another is what limits the stage rate
        constexpr int kPerPage = 2 * C::kHalves;
        const int q = lane / kPerPage, r = lane % kPerPage;
        const int h = r % C::kHalves;
        const bool is_v = r >= C::kHalves;
        int b = __shfl_sync(0xffffffffu, cur, (page0 - base_id + (q < C::kPagesPerStage ? q : 0)) & 31);
        if (lane < kPerPage * np) {
          if ((uint64_t)b >= (uint64_t)p.n_blocks) {
            atomicCAS(p.status, 0, kDevBadIndex);
            b = 0;
          }
          tma_load_4d((is_v ? vst : kst) + h * C::kKVHalfBytes + q * kPageTokens * 128, is_v ? &vmap : &kmap,
                      &full[s], 0, h, kvh * kPageTokens, layer * (int)p.n_blocks + b, policy);
        }
      }
    }
    if (!ok && lane == 0) {
      atomicCAS(p.status, 0, kDevTimeout);
      // wait (bounded) for this CTA's copies still in flight before it exits
      for (int t = max(0, jk - C::kStages); t < jk; ++t) mbar_wait(&full[t % C::kStages], (t / C::kStages) & 1);
      if constexpr (C::kSplitKV)
        for (int t = max(0, jv - C::kVStages); t < jv; ++t)
          mbar_wait(&v_full[t % C::kVStages], (t / C::kVStages) & 1);
    }
    return;
  }

  // ---- MMA issuer ----------------------------------------------------------------
  // One lane runs the issue loop; in the kElect form (small launches whose
  // pages stay in L2, where a step is a chain of latencies) the whole warp
  // runs it with warp-uniform operands and an elected lane issues, which
  // shortens each hand-off but costs the streaming launches issue slots.
  if (warp == kMmaWarp) {
    auto wait = [&](uint64_t* bar, uint32_t parity) {
      return kElect ? __all_sync(0xffffffffu, mbar_wait(bar, parity)) : mbar_wait(bar, parity);
    };
    auto landed = [&](uint64_t* bar, uint32_t parity) {
      return kElect ? __all_sync(0xffffffffu, mbar_try_wait(bar, parity)) : mbar_try_wait(bar, parity);
    };
    auto mma_ss = [&](uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
      if constexpr (kElect) tc_mma_bf16_elect(d, a, b, idesc, acc);
      else tc_mma_bf16(d, a, b, idesc, acc);
    };
    auto mma_ts = [&](uint32_t d, uint32_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
      if constexpr (kElect) tc_mma_bf16_tmem_a_elect(d, a, b, idesc, acc);
      else tc_mma_bf16_tmem_a(d, a, b, idesc, acc);
    };
    auto commit = [&](uint64_t* bar) {
      if constexpr (kElect) tc_commit_elect(bar);
      else tc_commit(bar);
    };
    if (kElect || lane == 0) {
      constexpr uint32_t idesc_s = tc_idesc_bf16(C::kM, C::kKeys, 0, 0);
      constexpr uint32_t idesc_o = tc_idesc_bf16(C::kMo, D, 0, 1);
      // Shared-memory descriptors are built once: the start field holds
      // address / 16 (below 2^14 in shared memory), so the descriptor of an
      // operand shifted by b bytes is the base descriptor + b / 16.
      const uint64_t q_desc = tc_desc_sw128(smem_addr(q_s), 16, 1024);
      const uint64_t k_desc0 = tc_desc_sw128(smem_addr(ring), 16, 1024);
      const uint64_t v_desc0 = tc_desc_sw128(smem_addr(ring + C::kKRingBytes), C::kKVHalfBytes, 1024);
      bool ok = wait(q_ready, 0);
      tc_fence_after_sync();
      // S_j = Q K_j^T into S buffer j & 1
      auto issue_s = [&](int j) -> bool {
        const int s = j % C::kStages;
        if (!wait(&full[s], (j / C::kStages) & 1)) return false;
        tc_fence_after_sync();
        const uint64_t kd = k_desc0 + (uint64_t)((s * C::kKSlotBytes) >> 4);
#pragma unroll
        for (int h = 0; h < C::kHalves; ++h)
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_ss(tmem + kTmemS + (j & 1) * C::kKeys, q_desc + (uint64_t)((h * C::kQHalfBytes + kk * 32) >> 4),
                   kd + (uint64_t)((h * C::kKVHalfBytes + kk * 32) >> 4), idesc_s, (h | kk) != 0);
        commit(&s_full[j & 1]);
        if constexpr (C::kSplitKV) commit(&empty[s]);  // K_j has been read
        return true;
      };
      if (ok) ok = issue_s(0);
      for (int j = 0; ok && j < n_tiles; ++j) {
        // S buffer (j+1)&1 was last read by the softmax of stage j-1, whose P
        // this thread has already waited for.  Issue S_{j+1} ahead of P_j V_j
        // only when its data has already landed, so that a slow load never
        // delays P_j V_j.
        const int jn = j + 1;
        bool early = false;
        if (jn < n_tiles && landed(&full[jn % C::kStages], (jn / C::kStages) & 1)) {
          if (!issue_s(jn)) {
            ok = false;
            break;
          }
          early = true;
        }
        if (!wait(&p_full[j & 1], (j >> 1) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const int s = j % C::kStages, sv = j % C::kVStages;
        const uint64_t kd = k_desc0 + (uint64_t)((s * C::kKSlotBytes) >> 4);
        const uint64_t vd0 = v_desc0 + (uint64_t)((sv * C::kVSlotBytes) >> 4);
        if constexpr (kWide) {
          if (!wait(&v_full[sv], (j / C::kVStages) & 1)) {
            ok = false;
            break;
          }
          tc_fence_after_sync();
          // P_hi, P_lo of keys [16 ks, 16 ks + 16) in the 16 TMEM columns of their scores
          const uint32_t p_tm = tmem + kTmemS + (j & 1) * C::kKeys;
#pragma unroll
          for (int ks = 0; ks < C::kKeys / 16; ++ks) {
            const uint64_t vd = vd0 + (uint64_t)((ks * 16 * 128) >> 4);
            mma_ts(tmem + kTmemO, p_tm + ks * 16, vd, idesc_o, (j > 0 || ks > 0) ? 1u : 0u);
            mma_ts(tmem + kTmemO, p_tm + ks * 16 + 8, vd, idesc_o, 1u);
          }
        } else {
          // [P_hi; P_lo] V: one M = 128 product per 16 keys for both terms
#pragma unroll
          for (int ks = 0; ks < C::kKeys / 16; ++ks)
            mma_ss(tmem + kTmemO, kd + (uint64_t)((ks * 32) >> 4), vd0 + (uint64_t)((ks * 16 * 128) >> 4), idesc_o,
                   (j > 0 || ks > 0) ? 1u : 0u);
        }
        commit(C::kSplitKV ? &v_empty[sv] : &empty[s]);
        commit(o_ready);
        if (jn < n_tiles && !early && !issue_s(jn)) {
          ok = false;
          break;
        }
      }
      commit(o_final);
      if (!ok && lane == 0) atomicCAS(p.status, 0, kDevTimeout);
    }
    __syncwarp();
    named_barrier_sync(1, n_swt + 32);
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
    return;
  }
  if (warp >= n_sw) return;

  // ---- softmax warps ---------------------------------------------------------------
  // Narrow: threads t and t + 16 of a warp share row t and half of the
  // stage's keys each, the row max and sum combined with one shuffle; thread
  // t owns the TMEM lane of O_hi (P_hi V) of the row, thread t + 16 the lane
  // of O_lo (P_lo V).  Wide: one thread per row.
  constexpr bool kPair = !kWide;
  constexpr int kKpt = C::kKeys / (kPair ? 2 : 1);  // keys per thread per stage
  const int tid = threadIdx.x;                      // 0 .. n_swt-1, for cooperative loops
  const int half = kPair ? (lane >> 4) : 0;
  const int r = kPair ? warp * 16 + (lane & 15) : threadIdx.x;  // this thread's row
  const uint32_t t_lane = tmem + ((uint32_t)(warp * 32) << 16);
  const bool valid = r < n_rows;
  int qrow = 0, head = 0;
  if (valid) {
    qrow = members[item.member_base + r / G];
    head = kvh * G + r % G;
  }
  if (r < C::kQRows) {
    const uint4* src = reinterpret_cast<const uint4*>(p.q + (((int64_t)layer * p.n_rows_q + qrow) * p.Hq + head) * D);
    constexpr int kChunks = D / 8 / (kPair ? 2 : 1);  // 16-byte chunks of the row this thread writes
#pragma unroll
    for (int cc = 0; cc < kChunks; ++cc) {
      const int c = half * kChunks + cc;
      const uint4 v = valid ? src[c] : make_uint4(0u, 0u, 0u, 0u);
      *reinterpret_cast<uint4*>(q_s + (c >> 3) * C::kQHalfBytes + r * 128 + (((c & 7) ^ (r & 7)) << 4)) = v;
    }
    fence_proxy_async_smem();
  }
  mbar_arrive(q_ready);

  // columns [32 k, 32 k + 32) of this thread's O lane
  auto o_load = [&](int k, float* o) { tmem_ld32(t_lane + kTmemO + k * 32, o); };
  auto o_store = [&](int k, const float* o) { tmem_st32(t_lane + kTmemO + k * 32, o); };

  const float sl2 = p.scale_log2;
  float m_used = -1e30f, l = 0.f;  // l: this thread's share of the row sum
  bool ok = true;
  for (int j = 0; j < n_tiles; ++j) {
    const int s = j % C::kStages;
    if (!__all_sync(0xffffffffu, mbar_wait(&s_full[j & 1], (j >> 1) & 1))) {
      ok = false;
      break;
    }
    tc_fence_after_sync();
    // raw scores q.k of this thread's keys; the softmax works in the log2
    // domain, x = s * sl2
    float sc[kKpt];
    static_assert(C::kKeys == 64, "64 keys per stage");
    if constexpr (kPair) tmem_ld16x2_32<32>(t_lane + kTmemS + (j & 1) * C::kKeys, sc);
    else tmem_ld64(t_lane + kTmemS + (j & 1) * C::kKeys, sc);
    const int key0 = j * C::kKeys;
    const int kbase = half * kKpt;  // this thread's first key within the stage
    const int np = min(C::kPagesPerStage, n_pages - j * C::kPagesPerStage);
    const int loaded = np * kPageTokens;
    if (key0 + C::kKeys > n_valid_keys || loaded < C::kKeys) {
#pragma unroll
      for (int c = 0; c < kKpt; ++c)
        if (kbase + c >= loaded || key0 + kbase + c >= n_valid_keys) sc[c] = -INFINITY;
    }
    // 8 independent max chains, then a tree (short dependency chains)
    float mx8[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) mx8[i] = sc[i];
#pragma unroll
    for (int c = 8; c < kKpt; ++c) mx8[c & 7] = fmaxf(mx8[c & 7], sc[c]);
    float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                     fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
    if constexpr (kPair) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 16));
    const float m_new = fmaxf(m_used, mx * sl2);  // sl2 > 0: max commutes with the scale
    const bool need = valid && m_new > m_used + kRescaleThreshold;
    if (__any_sync(0xffffffffu, need)) {
      const float alpha = need ? ex2(m_used - m_new) : 1.f;
      if (j > 0) {
        // P_{j-1} V_{j-1} must have landed in O (P_j V_j cannot start before
        // this thread's P_j, so the parity below is unambiguous)
        if (!__all_sync(0xffffffffu, mbar_wait(o_ready, (j - 1) & 1))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
#pragma unroll 1
        for (int k = 0; k < D / 32; ++k) {
          float o[32];
          o_load(k, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          o_store(k, o);
        }
      }
      l *= alpha;
      if (need) m_used = m_new;
    }
    uint8_t* kslot = k_slot(s);  // narrow: S_j has been consumed, P_j goes over K_j
    if constexpr (kWide) {
      // P_hi, P_lo of keys [16 k, 16 k + 16) over the 16 TMEM columns of their
      // scores (all read above).  The store is warp-wide: rows past the
      // item's take 2^-inf = 0.
      const uint32_t p_tm = t_lane + kTmemS + (j & 1) * C::kKeys;
      const float mo = valid ? m_used : INFINITY;
      float rs[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int kq = 0; kq < C::kKeys / 16; ++kq) {
        uint32_t pk[16];
#pragma unroll
        for (int c = 0; c < 16; c += 2) {
          const float a = ex2(fmaf(sc[kq * 16 + c], sl2, -mo)), b = ex2(fmaf(sc[kq * 16 + c + 1], sl2, -mo));
          rs[(c >> 1) & 7] += a + b;
          const uint32_t hi = pack_bf16(a, b);
          pk[c / 2] = hi;
          pk[8 + c / 2] = pack_bf16(a - __uint_as_float(hi << 16), b - __uint_as_float(hi & 0xffff0000u));
        }
        tmem_st16u_nowait(p_tm + kq * 16, pk);
      }
      tmem_wait_st();
      l += ((rs[0] + rs[1]) + (rs[2] + rs[3])) + ((rs[4] + rs[5]) + (rs[6] + rs[7]));
    } else if (valid) {
      uint32_t pk[kKpt / 2];
      uint32_t pl[kKpt / 2];
      float rs[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int c = 0; c < kKpt; c += 2) {
        const float a = ex2(fmaf(sc[c], sl2, -m_used)), b = ex2(fmaf(sc[c + 1], sl2, -m_used));
        rs[(c >> 1) & 7] += a + b;
        const uint32_t hi = pack_bf16(a, b);
        pk[c / 2] = hi;
        // remainders below the bf16 rounding of a and b
        pl[c / 2] = pack_bf16(a - __uint_as_float(hi << 16), b - __uint_as_float(hi & 0xffff0000u));
      }
      l += ((rs[0] + rs[1]) + (rs[2] + rs[3])) + ((rs[4] + rs[5]) + (rs[6] + rs[7]));
      // A rows of P_hi and P_lo: 32 w + t and 32 w + 16 + t (both = t mod 8)
      const int a_hi = warp * 32 + (lane & 15);
#pragma unroll
      for (int cc = 0; cc < kKpt / 8; ++cc) {
        const int c = half * (kKpt / 8) + cc;  // 16-byte chunk of the P row (8 keys)
        const uint32_t off = a_hi * 128 + ((c ^ (a_hi & 7)) << 4);
        *reinterpret_cast<uint4*>(kslot + off) = make_uint4(pk[4 * cc], pk[4 * cc + 1], pk[4 * cc + 2], pk[4 * cc + 3]);
        *reinterpret_cast<uint4*>(kslot + 16 * 128 + off) =
            make_uint4(pl[4 * cc], pl[4 * cc + 1], pl[4 * cc + 2], pl[4 * cc + 3]);
      }
    }
    if (key0 + C::kKeys > n_valid_keys || loaded < C::kKeys) {
      // zero the V rows of keys that are not valid, once V_j has landed
      // (narrow: with K_j, from which S_j was computed)
      const int sv = j % C::kVStages;
      if (!__all_sync(0xffffffffu, C::kSplitKV ? mbar_wait(&v_full[sv], (j / C::kVStages) & 1)
                                               : mbar_wait(&full[s], (j / C::kStages) & 1))) {
        ok = false;
        break;
      }
      uint8_t* vslot = v_slot(sv);
      for (int t = tid; t < C::kKeys * C::kHalves; t += n_swt) {
        const int c = t % C::kKeys, h = t / C::kKeys;
        if (c >= loaded || key0 + c >= n_valid_keys) {
#pragma unroll
          for (int x = 0; x < 8; ++x)
            *reinterpret_cast<uint4*>(vslot + h * C::kKVHalfBytes + c * 128 + x * 16) = make_uint4(0u, 0u, 0u, 0u);
        }
      }
    }
    fence_proxy_async_smem();
    tc_fence_before_sync();
    mbar_arrive(&p_full[j & 1]);
  }
  if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_final, 0));
  tc_fence_after_sync();
  if (ok) {
    if constexpr (kPair) l += __shfl_xor_sync(0xffffffffu, l, 16);  // the row's full sum
    const float inv = 1.f / l;
    float* dst = nullptr;
    float* dst_lse = nullptr;
    if (valid) {
      const int64_t idx = (((int64_t)layer * p.n_rows_q + qrow) * p.Hq + head) * p.max_splits + item.split;
      dst = p.out_o + idx * D;
      if (half == 0) dst_lse = p.out_lse + idx;
    }
    if constexpr (kPair) {
      // O = O_hi + O_lo: thread t writes columns [0, D/2) of the row, thread
      // t + 16 columns [D/2, D); one shuffle per column pair swaps the halves
      // each needs from the other's lane
#pragma unroll 1
      for (int k = 0; k < D / 64; ++k) {
        float a[32], b[32];
        o_load(k, a);           // columns [32 k, 32 k + 32)
        o_load(k + D / 64, b);  // columns [D/2 + 32 k, D/2 + 32 k + 32)
#pragma unroll
        for (int i = 0; i < 32; ++i) {
          const float other = __shfl_xor_sync(0xffffffffu, half ? a[i] : b[i], 16);
          a[i] = (half ? b[i] : a[i]) + other;
        }
        if (dst) {
          float* d = dst + half * (D / 2) + k * 32;
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            *reinterpret_cast<float4*>(d + i) = make_float4(a[i] * inv, a[i + 1] * inv, a[i + 2] * inv, a[i + 3] * inv);
        }
      }
    } else {
#pragma unroll 1
      for (int k = 0; k < D / 32; ++k) {
        float o[32];
        o_load(k, o);
        if (dst) {
#pragma unroll
          for (int i = 0; i < 32; i += 4)
            *reinterpret_cast<float4*>(dst + k * 32 + i) =
                make_float4(o[i] * inv, o[i + 1] * inv, o[i + 2] * inv, o[i + 3] * inv);
        }
      }
    }
    if (dst_lse) *dst_lse = (m_used + log2f(l)) * kLn2;
  } else if (lane == 0) {
    atomicCAS(p.status, 0, kDevTimeout);
  }
  tc_fence_before_sync();
  named_barrier_sync(1, n_swt + 32);
}

template <int D, bool kWide, bool kElect>
cudaError_t launch_tc_t(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p,
                        const InlineDecodePlan& inl, int n_ctas, cudaStream_t s) {
  using C = TcCfg<D, kWide>;
  // the shared-memory opt-in is a per-device function attribute
  static bool configured[kMaxDevices] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    e = cudaFuncSetAttribute(attend_tc_kernel<D, kWide, kElect>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  dim3 grid(n_ctas, p.Hkv, p.L);
  return launch_chained(attend_tc_kernel<D, kWide, kElect>, grid, dim3(kThreads), C::kSmemBytes, s, km, vm, p,
                        inl);
}

template <int D>
int decode_ctas_per_sm_t() {
  using C = TcCfg<D, false>;
  if (cudaFuncSetAttribute(attend_tc_kernel<D, false, false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           C::kSmemBytes) != cudaSuccess)
    return 0;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attend_tc_kernel<D, false, false>, kThreads, C::kSmemBytes) !=
      cudaSuccess)
    return 0;
  return n < 2 ? n : 2;  // two CTAs' TMEM (2 x 256 columns) fill an SM
}

}  // namespace

cudaError_t launch_decode_tc(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p,
                             const InlineDecodePlan* inl, int n_items, int D, bool wide, cudaStream_t s) {
  static const InlineDecodePlan kNone{};
  const InlineDecodePlan& ip = inl ? *inl : kNone;
  if (n_items <= 0) return cudaSuccess;
  // the narrow tile of a launch whose pages stay in L2 takes the elected issue
  const bool elect = !wide && p.keep_l2;
  if (D == 128) {
    if (wide) return launch_tc_t<128, true, false>(km, vm, p, ip, n_items, s);
    return elect ? launch_tc_t<128, false, true>(km, vm, p, ip, n_items, s)
                 : launch_tc_t<128, false, false>(km, vm, p, ip, n_items, s);
  }
  if (D == 64) {
    if (wide) return launch_tc_t<64, true, false>(km, vm, p, ip, n_items, s);
    return elect ? launch_tc_t<64, false, true>(km, vm, p, ip, n_items, s)
                 : launch_tc_t<64, false, false>(km, vm, p, ip, n_items, s);
  }
  return cudaErrorInvalidValue;
}

int decode_tc_ctas_per_sm(int D) {
  if (D == 128) return decode_ctas_per_sm_t<128>();
  if (D == 64) return decode_ctas_per_sm_t<64>();
  return 0;
}

}  // namespace st
