// Merge prefill on the tcgen05 tensor cores: two 128-row query tiles per CTA
// that share every K/V stage (one CTA per SM).
//
// Section 3.5 of the paper: the harvested thoughts are appended after main's
// context and read in order, so thought row i of a merge of T rows attends
// to main's keys [0, L0 + i].  The (thought row, query head) pairs of one KV
// head are stacked G per token; a CTA takes 256 consecutive stacked rows as
// tile A (the first 128) and tile B (the next 128) and walks main's pages up
// to the causal limit of its last row, 128 keys per stage.  Both tiles read
// each K/V stage from shared memory.  A batched prefill (several sequences'
// new rows in one launch) gives each CTA its own (sequence, L0, T, row tile)
// through a work list.
//
// CTA layout (352 threads, one CTA per SM, all 512 TMEM columns):
//   warps 0..3  softmax of tile A, warps 4..7 softmax of tile B: thread r of
//               a tile owns its row r = TMEM lane r (warp w reads lanes
//               32 (w % 4) ..).  It stages its Q row in shared memory; per
//               stage it reads its 128 scores, masks keys past the stage's
//               pages and past its causal limit, keeps a running max raised
//               only when a score exceeds it by more than 2^8 (O in TMEM is
//               then rescaled in place), and writes P = 2^(s - m) as two bf16
//               terms (P_hi + P_lo, exact to about 16 bits) into TMEM over its
//               own scores.  At the end it normalises O.
//   warp 8      K loader, warp 9 V loader: page ids from the block table (32
//               per read, one batch ahead), one 2 KiB TMA copy per (page,
//               64-wide half of D) into separate K and V rings.
//   warp 10     TMEM owner and MMA issuer (the whole warp runs the loop with
//               warp-uniform operands, an elected lane issues), per stage j
//               and tile t = A, B,
//                 O_t += P_t(j-1) V_{j-1}   (A = P_hi, P_lo from TMEM, M 128, N D)
//                 S_t(j) = Q_t K_j^T        (M 128, N 128)
//               so that the softmax of one tile overlaps the MMAs of the
//               other.
//
// TMEM columns: tile t (0 = A, 1 = B) has S at 256 t (128 columns; the 16
// columns of keys [16 k, 16 k + 16) then hold P_hi and P_lo of those keys as
// bf16 pairs) and O at 256 t + 128.  S_t(j + 1) overwrites P_t(j)
// only after O_t += P_t(j) V_j, which the same thread issued first; and the
// commit that announces S_t(j) also covers O_t += P_t(j-1) V_{j-1}, so the
// softmax may rescale O_t as soon as it sees S_t(j).
//
// Synchronisation (every wait bounded; a wait that runs out sets the status
// word and the CTA winds down):
//   k_full / k_empty, v_full / v_empty   ring slots (TMA bytes / MMA commit)
//   s_full[t]      S_t of the stage is complete                 (MMA commit)
//   p_full[t][h]   P_t of keys [64 h, 64 h + 64) is in TMEM     (128 arrivals)
//   o_final        every MMA of the CTA has completed
// S_t(j + 1) is issued only after p_full[t][1] of stage j, so each barrier is
// at most one phase ahead of its waiters.  The MMAs of the first half of P
// run while the softmax computes the second.
//
// Shared-memory operands use the 128-byte swizzle (8-row x 128-byte atoms):
//   Q_t [D/64][128 rows][64]   K-major A (SBO 1024)
//   K   [D/64][128 keys][64]   K-major B (SBO 1024)
//   V   [D/64][128 keys][64]   MN-major B (LBO = one D-half, SBO 1024)
// V rows of keys that are not valid (past main's end, or in pages a short
// last stage did not load) are zeroed by tile A's threads before P V, so that
// stale shared or pool memory cannot turn 0 * x into NaN in a real row.
#include <math.h>

#include <type_traits>

#include "kernels.cuh"
#include "ptx.cuh"

namespace st {

namespace {

constexpr int kTileRows = 128;
constexpr int kKeys = 128;  // keys per stage
constexpr int kPagesPerStage = kKeys / kPageTokens;
constexpr int kKLoadWarp = 8, kVLoadWarp = 9, kMmaWarp = 10;
constexpr int kThreads = 11 * 32;
constexpr int kSoftThreads = 8 * 32;
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kTmemTile = 256, kTmemO = 128;  // per-tile column base, O offset within it
constexpr float kRescaleThreshold = 8.f;           // log2 units
constexpr float kLn2 = 0.69314718055994530942f;

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

template <int D>
struct PairCfg {
  static constexpr int kHalves = D / 64;
  static constexpr int kQHalfBytes = kTileRows * 128;
  static constexpr int kQTileBytes = kHalves * kQHalfBytes;
  static constexpr int kKVHalfBytes = kKeys * 128;
  static constexpr int kSlotBytes = kHalves * kKVHalfBytes;
  static constexpr int kKStages = D == 128 ? 3 : 4;
  static constexpr int kVStages = D == 128 ? 2 : 4;
  static constexpr int kQOff = 0;
  static constexpr int kKOff = kQOff + 2 * kQTileBytes;
  static constexpr int kVOff = kKOff + kKStages * kSlotBytes;
  static constexpr int kBarOff = kVOff + kVStages * kSlotBytes;
  static constexpr int kSmemBytes = 1024 + kBarOff + 256;
  static_assert(kSmemBytes <= 227 * 1024, "shared memory of one CTA");
};

template <int D, bool kDecode>
__global__ void __launch_bounds__(kThreads, 1)
    merge_pair_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                      const AttnParams p, const __grid_constant__ InlineDecodePlan inl) {
  using C = PairCfg<D>;
  constexpr int kKS = C::kKStages, kVS = C::kVStages;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* base = smem_raw + ((1024u - (raw & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + C::kBarOff);
  uint64_t* k_full = bars;
  uint64_t* k_empty = k_full + kKS;
  uint64_t* v_full = k_empty + kKS;
  uint64_t* v_empty = v_full + kVS;
  uint64_t* s_full = v_empty + kVS;  // [2 tiles]
  uint64_t* p_full = s_full + 2;     // [2 tiles][2 key halves]
  uint64_t* o_final = p_full + 4;
  uint64_t* q_ready = o_final + 1;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(q_ready + 1);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int kvh = blockIdx.y;
  const int layer = blockIdx.z;
  const int G = p.G;

  // Decode: launched as a programmatic dependent of the kernel before it in
  // the stream; the tensor-memory allocation touches no global memory, every
  // global access comes after the wait.
  if constexpr (kDecode) {
    if (warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
    griddep_wait();
    griddep_launch_dependents();
  }
  // one merge: its row tiles, the last ones (most keys) first; a batch: one
  // work item per CTA (the host orders those longest first); a decode: one
  // run of pages of a fork group (at most 256 stacked rows) per CTA, every
  // row over all of the run's keys
  int slot = p.slot, L0 = p.L0, T = p.T, q_row0 = 0, row_base = (gridDim.x - 1 - blockIdx.x) * 2 * kTileRows;
  int page_begin = 0, n_rows, n_pages, n_valid_keys;
  AttnItem item{};
  const int32_t* members = nullptr;
  if constexpr (kDecode) {
    members = p.members ? p.members : inl.members;
    item = p.items ? p.items[p.item_base + blockIdx.x] : inl.items[p.item_base + blockIdx.x];
    slot = item.slot;
    page_begin = item.page_begin;
    row_base = 0;
    n_rows = min(2 * kTileRows, item.n_members * G);
    n_pages = item.n_pages;
    n_valid_keys = item.n_tokens;
  } else {
    if (p.mitems) {
      const MergeItem mi = p.mitems[blockIdx.x];
      slot = mi.slot;
      L0 = mi.L0;
      T = mi.T;
      q_row0 = mi.q_row0;
      row_base = mi.row_base;
    }
    n_rows = min(2 * kTileRows, T * G - row_base);
    const int t_last = (row_base + n_rows - 1) / G;
    n_pages = (L0 + t_last + 1 + kPageTokens - 1) / kPageTokens;
    n_valid_keys = L0 + T;
  }
  const int n_tiles = (n_pages + kPagesPerStage - 1) / kPagesPerStage;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kKS; ++s) {
      mbar_init(&k_full[s], 1);
      mbar_init(&k_empty[s], 1);
    }
    for (int s = 0; s < kVS; ++s) {
      mbar_init(&v_full[s], 1);
      mbar_init(&v_empty[s], 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(&s_full[t], 1);
      mbar_init(&p_full[2 * t], kTileRows);
      mbar_init(&p_full[2 * t + 1], kTileRows);
    }
    mbar_init(o_final, 1);
    mbar_init(q_ready, kSoftThreads);
    fence_mbar_init();
  }
  if (!kDecode && warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  // ---- loaders -------------------------------------------------------------------
  if (warp == kKLoadWarp || warp == kVLoadWarp) {
    if (p.hold_loads) return;  // test hook: nothing arrives, the other roles' waits run out
    const bool is_k = warp == kKLoadWarp;
    const CUtensorMap* map = is_k ? &kmap : &vmap;
    uint64_t* full = is_k ? k_full : v_full;
    uint64_t* empty = is_k ? k_empty : v_empty;
    const int n_st = is_k ? kKS : kVS;
    uint8_t* ring = base + (is_k ? C::kKOff : C::kVOff);
    if (lane == 0) prefetch_tensormap(map);
    // merge: every CTA of one (layer, KV head) walks the same pages, keep them
    // in L2; decode: a page is streamed once, unless a sibling subgroup's CTA
    // reads it too or the whole launch fits in L2
    const uint64_t policy = !kDecode ? l2_policy_evict_last()
                            : (p.keep_l2 || (item.flags & kItemReread)) ? l2_policy_evict_normal()
                                                                         : l2_policy_evict_first();
    const int32_t* ids = p.table + (int64_t)slot * p.max_pages + page_begin;
    int base_id = 0;
    int cur = lane < n_pages ? ids[lane] : 0;
    int nxt = 32 + lane < n_pages ? ids[32 + lane] : 0;
    int j = 0;
    bool ok = true;
    for (; j < n_tiles; ++j) {
      const int s = j % n_st;
      if (j >= n_st) {
        int w = 1;
        if (lane == 0) w = mbar_wait(&empty[s], ((j / n_st) - 1) & 1) ? 1 : 0;
        w = __shfl_sync(0xffffffffu, w, 0);
        if (!w) {
          ok = false;
          break;
        }
      }
      const int page0 = j * kPagesPerStage;
      if (page0 >= base_id + 32) {
        base_id += 32;
        cur = nxt;
        nxt = base_id + 32 + lane < n_pages ? ids[base_id + 32 + lane] : 0;
      }
      const int np = min(kPagesPerStage, n_pages - page0);
      uint8_t* dst = ring + s * C::kSlotBytes;
      if (lane == 0) mbar_arrive_expect_tx(&full[s], (uint32_t)(np * C::kHalves * kPageTokens * 128));
      __syncwarp();
      // one copy per lane (lane = D/64 q + h)
      const int q = lane / C::kHalves, h = lane % C::kHalves;
      int b = __shfl_sync(0xffffffffu, cur, (page0 - base_id + (q < kPagesPerStage ? q : 0)) & 31);
      if (lane < C::kHalves * np) {
        if ((uint64_t)b >= (uint64_t)p.n_blocks) {
          atomicCAS(p.status, 0, kDevBadIndex);
          b = 0;
        }
        tma_load_4d(dst + h * C::kKVHalfBytes + q * kPageTokens * 128, map, &full[s], 0, h, kvh * kPageTokens,
                    layer * (int)p.n_blocks + b, policy);
      }
    }
    if (!ok && lane == 0) {
      atomicCAS(p.status, 0, kDevTimeout);
      for (int t = max(0, j - n_st); t < j; ++t) mbar_wait(&full[t % n_st], (t / n_st) & 1);
    }
    return;
  }

  // ---- MMA issuer ----------------------------------------------------------------
  // One warp issues every MMA (two issuing warps interleaving on the tensor
  // pipe measured slower): all its lanes run the loop with warp-uniform
  // operands and an elected lane issues.  The issue rate bounds this kernel
  // (tens of cycles per tcgen05.mma), so the per-MMA work is a constant add:
  // a shared-memory descriptor's start field holds address / 16 (below 2^14
  // here), so the descriptor of an operand shifted by b bytes is the base
  // descriptor + b / 16.
  if (warp == kMmaWarp) {
    {
      constexpr uint32_t idesc_s = tc_idesc_bf16(kTileRows, kKeys, 0, 0);
      constexpr uint32_t idesc_o = tc_idesc_bf16(kTileRows, D, 0, 1);
      const uint64_t q_desc = tc_desc_sw128(smem_addr(base + C::kQOff), 16, 1024);
      const uint64_t k_desc0 = tc_desc_sw128(smem_addr(base + C::kKOff), 16, 1024);
      const uint64_t v_desc0 = tc_desc_sw128(smem_addr(base + C::kVOff), C::kKVHalfBytes, 1024);
      bool ok = __all_sync(0xffffffffu, mbar_wait(q_ready, 0));
      tc_fence_after_sync();
      // O_t += P_t(i) V_i, P_t(i) read from TMEM over S_t(i); each half of P
      // (64 keys) is published on its own, so the first half's MMAs run while
      // the softmax finishes the second
      auto issue_pv = [&](auto tile, int i) -> bool {
        constexpr int t = decltype(tile)::value;
        const int s = i % kVS;
        if (t == 0 && !__all_sync(0xffffffffu, mbar_wait(&v_full[s], (i / kVS) & 1))) return false;
        const uint64_t vd = v_desc0 + (uint64_t)((s * C::kSlotBytes) >> 4);
        const uint32_t acc0 = i > 0 ? 1u : 0u;
#pragma unroll
        for (int hf = 0; hf < 2; ++hf) {
          if (!__all_sync(0xffffffffu, mbar_wait(&p_full[2 * t + hf], i & 1))) return false;
          tc_fence_after_sync();
#pragma unroll
          for (int kq = 0; kq < kKeys / 32; ++kq) {
            const int ks = hf * (kKeys / 32) + kq;
            const uint64_t vk = vd + (uint64_t)((ks * 16 * 128) >> 4);
            tc_mma_bf16_tmem_a_elect(tmem + t * kTmemTile + kTmemO, tmem + t * kTmemTile + ks * 16, vk, idesc_o,
                               ks > 0 ? 1u : acc0);                                    // P_hi
            tc_mma_bf16_tmem_a_elect(tmem + t * kTmemTile + kTmemO, tmem + t * kTmemTile + ks * 16 + 8, vk, idesc_o,
                               1u);                                                     // P_lo
          }
        }
        if (t == 1) tc_commit_elect(&v_empty[s]);
        return true;
      };
      // S_t(j) = Q_t K_j^T
      auto issue_s = [&](auto tile, uint64_t kd) {
        constexpr int t = decltype(tile)::value;
#pragma unroll
        for (int h = 0; h < C::kHalves; ++h)
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16_elect(tmem + t * kTmemTile,
                        q_desc + (uint64_t)((t * C::kQTileBytes + h * C::kQHalfBytes + kk * 32) >> 4),
                        kd + (uint64_t)((h * C::kKVHalfBytes + kk * 32) >> 4), idesc_s, (h | kk) != 0);
        tc_commit_elect(&s_full[t]);
      };
      const std::integral_constant<int, 0> tile_a;
      const std::integral_constant<int, 1> tile_b;
      for (int j = 0; ok && j < n_tiles; ++j) {
        const int s = j % kKS;
        const uint64_t kd = k_desc0 + (uint64_t)((s * C::kSlotBytes) >> 4);
        if (j > 0 && !issue_pv(tile_a, j - 1)) {
          ok = false;
          break;
        }
        if (!__all_sync(0xffffffffu, mbar_wait(&k_full[s], (j / kKS) & 1))) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        issue_s(tile_a, kd);
        if (j > 0 && !issue_pv(tile_b, j - 1)) {
          ok = false;
          break;
        }
        issue_s(tile_b, kd);
        tc_commit_elect(&k_empty[s]);
      }
      if (ok && n_tiles > 0) ok = issue_pv(tile_a, n_tiles - 1) && issue_pv(tile_b, n_tiles - 1);
      tc_commit_elect(o_final);
      if (!ok && lane == 0) atomicCAS(p.status, 0, kDevTimeout);
    }
    __syncwarp();
    named_barrier_sync(1, kSoftThreads + 32);
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
    return;
  }

  // ---- softmax warps ---------------------------------------------------------------
  const int t = warp >> 2;               // tile
  const int r = (warp & 3) * 32 + lane;  // row within the tile = TMEM lane
  const int tid = threadIdx.x & (kTileRows - 1);
  const uint32_t t_lane = tmem + ((uint32_t)((warp & 3) * 32) << 16) + t * kTmemTile;
  const int tile_row0 = row_base + t * kTileRows;
  const bool valid = t * kTileRows + r < n_rows;
  int qrow = 0, head = 0;
  if (valid) {
    const int gr = tile_row0 + r;
    qrow = kDecode ? members[item.member_base + gr / G] : gr / G;
    head = kvh * G + gr % G;
  }
  // causal limit of this row (a decode row sees the whole run)
  const int limit = kDecode ? n_valid_keys : valid ? L0 + qrow + 1 : n_valid_keys;
  const int min_limit = kDecode ? n_valid_keys : L0 + tile_row0 / G + 1;  // the tile's first row sees the fewest keys
  const int64_t io_row = (int64_t)layer * p.n_rows_q + q_row0 + qrow;  // this row in Q / O / LSE
  {
    const uint4* src = reinterpret_cast<const uint4*>(p.q + (io_row * p.Hq + head) * D);
    uint8_t* q_s = base + C::kQOff + t * C::kQTileBytes;
#pragma unroll
    for (int c = 0; c < D / 8; ++c) {
      const uint4 v = valid ? src[c] : make_uint4(0u, 0u, 0u, 0u);
      *reinterpret_cast<uint4*>(q_s + (c >> 3) * C::kQHalfBytes + r * 128 + (((c & 7) ^ (r & 7)) << 4)) = v;
    }
    fence_proxy_async_smem();
  }
  mbar_arrive(q_ready);

  const float sl2 = p.scale_log2;
  float m_used = -1e30f, l = 0.f;
  bool ok = true;
  for (int j = 0; j < n_tiles; ++j) {
    if (!__all_sync(0xffffffffu, mbar_wait(&s_full[t], j & 1))) {
      ok = false;
      break;
    }
    tc_fence_after_sync();
    const int key0 = j * kKeys;
    const int loaded = min(kPagesPerStage, n_pages - j * kPagesPerStage) * kPageTokens;
    const bool edge = key0 + kKeys > min_limit || loaded < kKeys;
    // scores of keys [hf * 64, hf * 64 + 64), masked past the stage's pages and
    // past this row's causal limit
    auto load_half = [&](int hf, float* sc) {
      tmem_ld64(t_lane + hf * 64, sc);
      if (edge) {
#pragma unroll
        for (int c = 0; c < 64; ++c)
          if (hf * 64 + c >= loaded || key0 + hf * 64 + c >= limit) sc[c] = -INFINITY;
      }
    };
    // row max over both halves: independent chains of three-input max
    float mx;
    {
      float mx8[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) mx8[i] = -INFINITY;
#pragma unroll 1  // one half's scores live at a time
      for (int hf = 0; hf < 2; ++hf) {
        float sc[64];
        load_half(hf, sc);
#pragma unroll
        for (int c = 0; c < 64; c += 16)
#pragma unroll
          for (int i = 0; i < 8; ++i) mx8[i] = fmax3(mx8[i], sc[c + i], sc[c + 8 + i]);
      }
      mx = fmax3(fmax3(mx8[0], mx8[1], mx8[2]), fmax3(mx8[3], mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7]));
    }
    const float m_new = fmaxf(m_used, mx * sl2);  // sl2 > 0: max commutes with the scale
    const bool need = valid && m_new > m_used + kRescaleThreshold;
    if (__any_sync(0xffffffffu, need)) {
      const float alpha = need ? ex2(m_used - m_new) : 1.f;
      if (j > 0) {
        // O_t += P_t(j-1) V_{j-1} has completed (covered by the commit of S_t(j))
#pragma unroll 1
        for (int k = 0; k < D / 32; ++k) {
          float o[32];
          tmem_ld32(t_lane + kTmemO + k * 32, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(t_lane + kTmemO + k * 32, o);
        }
      }
      l *= alpha;
      if (need) m_used = m_new;
    }
    if (t == 0 && (key0 + kKeys > n_valid_keys || loaded < kKeys)) {
      // zero the V rows of keys that are not valid once the stage's copies
      // have landed; both tiles' P V are issued after this tile's first P half
      const int s = j % kVS;
      if (!__all_sync(0xffffffffu, mbar_wait(&v_full[s], (j / kVS) & 1))) {
        ok = false;
        break;
      }
      uint8_t* vslot = base + C::kVOff + s * C::kSlotBytes;
      for (int x = tid; x < kKeys * C::kHalves; x += kTileRows) {
        const int c = x % kKeys, h = x / kKeys;
        if (c >= loaded || key0 + c >= n_valid_keys) {
#pragma unroll
          for (int y = 0; y < 8; ++y)
            *reinterpret_cast<uint4*>(vslot + h * C::kKVHalfBytes + c * 128 + y * 16) = make_uint4(0u, 0u, 0u, 0u);
        }
      }
      fence_proxy_async_smem();
    }
    // P = 2^(s sl2 - m) (two keys per packed f32x2 FMA / add) as two bf16
    // terms, P_hi = bf16(P) and P_lo = bf16(P - P_hi), so that P V is exact to
    // about 16 bits whatever the spread of the scores.  The 16 score columns
    // of keys [16 ks, 16 ks + 16) take P_hi of those keys (8 columns of bf16
    // pairs) and then P_lo (8 columns): each store overwrites only scores
    // already read.
    {
      const float2 scale2 = make_float2(sl2, sl2), neg_m2 = make_float2(-m_used, -m_used);
      float2 rs[4] = {make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f), make_float2(0.f, 0.f)};
#pragma unroll 1
      for (int hf = 0; hf < 2; ++hf) {
        float sc[64];
        load_half(hf, sc);
#pragma unroll
        for (int kq = 0; kq < 4; ++kq) {  // 16 keys per step
          uint32_t pk[16];
#pragma unroll
          for (int c = 0; c < 16; c += 2) {
            const float2 x = __ffma2_rn(make_float2(sc[kq * 16 + c], sc[kq * 16 + c + 1]), scale2, neg_m2);
            const float a = ex2(x.x), b = ex2(x.y);
            rs[(c >> 1) & 3] = __fadd2_rn(rs[(c >> 1) & 3], make_float2(a, b));
            const uint32_t hi = pack_bf16(a, b);
            pk[c / 2] = hi;
            pk[8 + c / 2] = pack_bf16(a - __uint_as_float(hi << 16), b - __uint_as_float(hi & 0xffff0000u));
          }
          tmem_st16u_nowait(t_lane + (hf * 4 + kq) * 16, pk);
        }
        tmem_wait_st();
        tc_fence_before_sync();
        mbar_arrive(&p_full[2 * t + hf]);
      }
      const float2 s = __fadd2_rn(__fadd2_rn(rs[0], rs[1]), __fadd2_rn(rs[2], rs[3]));
      l += s.x + s.y;
    }
  }
  if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_final, 0));
  tc_fence_after_sync();
  if (ok) {
    const float inv = 1.f / l;
    // merge: the row's O and LSE; decode: its split-KV partial
    const int64_t out_idx = kDecode ? (io_row * p.Hq + head) * p.max_splits + item.split : io_row * p.Hq + head;
    float* dst = valid ? p.out_o + out_idx * D : nullptr;
#pragma unroll 1
    for (int k = 0; k < D / 32; ++k) {
      float o[32];
      tmem_ld32(t_lane + kTmemO + k * 32, o);
      if (dst) {
#pragma unroll
        for (int i = 0; i < 32; i += 4)
          *reinterpret_cast<float4*>(dst + k * 32 + i) =
              make_float4(o[i] * inv, o[i + 1] * inv, o[i + 2] * inv, o[i + 3] * inv);
      }
    }
    if (valid) p.out_lse[out_idx] = (m_used + log2f(l)) * kLn2;
  } else if (lane == 0) {
    atomicCAS(p.status, 0, kDevTimeout);
  }
  tc_fence_before_sync();
  named_barrier_sync(1, kSoftThreads + 32);
}

template <int D, bool kDecode>
cudaError_t launch_pair_t(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p,
                          const InlineDecodePlan& inl, int n_ctas, cudaStream_t s) {
  using C = PairCfg<D>;
  // the shared-memory opt-in is a per-device function attribute
  static bool configured[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  if (!configured[dev]) {
    e = cudaFuncSetAttribute(merge_pair_kernel<D, kDecode>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             C::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured[dev] = true;
  }
  dim3 grid(n_ctas, p.Hkv, p.L);
  if constexpr (kDecode)
    return launch_chained(merge_pair_kernel<D, true>, grid, dim3(kThreads), C::kSmemBytes, s, km, vm, p, inl);
  merge_pair_kernel<D, false><<<grid, kThreads, C::kSmemBytes, s>>>(km, vm, p, inl);
  return cudaGetLastError();
}

const InlineDecodePlan kNoInline{};

}  // namespace

cudaError_t launch_merge_tc(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p, int n_items,
                            int D, cudaStream_t s) {
  // one merge: ceil(T G / 256) row tiles; a batch: its work items
  const int n_ctas = p.mitems ? n_items : (p.T * p.G + 2 * kTileRows - 1) / (2 * kTileRows);
  if (n_ctas <= 0) return cudaSuccess;
  if (D == 128) return launch_pair_t<128, false>(km, vm, p, kNoInline, n_ctas, s);
  if (D == 64) return launch_pair_t<64, false>(km, vm, p, kNoInline, n_ctas, s);
  return cudaErrorInvalidValue;
}

cudaError_t launch_decode_pair(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p,
                               const InlineDecodePlan* inl, int n_items, int D, cudaStream_t s) {
  const InlineDecodePlan& ip = inl ? *inl : kNoInline;
  if (n_items <= 0) return cudaSuccess;
  if (D == 128) return launch_pair_t<128, true>(km, vm, p, ip, n_items, s);
  if (D == 64) return launch_pair_t<64, true>(km, vm, p, ip, n_items, s);
  return cudaErrorInvalidValue;
}

}  // namespace st
