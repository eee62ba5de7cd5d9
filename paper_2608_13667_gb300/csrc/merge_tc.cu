// Merge prefill on the 5th-generation tensor cores (tcgen05, accumulators in
// tensor memory).
//
// Section 3.5 of the paper: the harvested thoughts are appended after the
// main context and the next turn reads them in order, so thought row i
// attends over main's rows [0, L0 + i].  Stacked over the G query heads of a
// KV head that is a dense causal contraction: 128 (thought row, head) query
// rows per CTA against main's pages, 64 keys per stage.
//
// CTA layout (192 threads, 2 CTAs per SM):
//   warps 0..3  softmax: thread r owns query row r = TMEM lane r.  Loads its
//               Q row into shared memory, then per stage reads its 64 scores
//               from TMEM, masks (causal limit, keys past the loaded pages),
//               keeps a running max that is only raised when a score exceeds
//               it by more than 2^8 (the O accumulator in TMEM is then
//               rescaled in place), writes P = 2^(s - m) as bf16 into the
//               stage's K slot, and finally normalises O out of TMEM.
//   warp 4      loader: page ids from the block table, one 2 KiB TMA copy per
//               (page, 64-wide half of D, K|V), per-stage mbarriers.
//   warp 5      TMEM owner; lane 0 issues the MMAs:
//                 S (TMEM cols [0,64))   = Q K^T   M=128 N=64  K=D
//                 O (TMEM cols [128,..)) += P V    M=128 N=D   K=64
//               and commits them to mbarriers.  A commit tracks every MMA
//               issued before it, so the commit that announces S_j also
//               guarantees P_{j-1} V_{j-1} is complete before O is touched.
//
// Shared-memory operands use the 128-byte swizzle (8-row x 128-byte atoms):
//   Q  [D/64][128 rows][64]  K-major A       (SBO 1024)
//   K  [D/64][64 keys][64]   K-major B       (SBO 1024)
//   P  [128 rows][64 keys]   K-major A       (SBO 1024), written over K
//   V  [D/64][64 keys][64]   MN-major B      (LBO = one D-half, SBO 1024)
// V rows of keys that are not valid (past the sequence, or in pages not
// loaded for a short last stage) are zeroed before P V, so stale shared or
// pool memory cannot turn 0 * x into NaN.
#include <math.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace st {

namespace {

constexpr int kRows = 128;
constexpr int kKeys = 64;
constexpr int kPagesPerStage = kKeys / kPageTokens;
constexpr int kStages = 2;
constexpr int kLoadWarp = 4, kMmaWarp = 5;
constexpr int kThreads = 6 * 32;
constexpr int kSoftmaxThreads = 128;
constexpr uint32_t kTmemCols = 256;
constexpr uint32_t kTmemS = 0, kTmemO = 128;
constexpr float kRescaleThreshold = 8.f;  // log2 units
constexpr float kLn2 = 0.69314718055994530942f;

template <int D>
struct TcGeo {
  static constexpr int kHalves = D / 64;
  static constexpr int kQBytes = kHalves * kRows * 128;
  static constexpr int kKVHalfBytes = kKeys * 128;                   // [64 keys][64]
  static constexpr int kKSlotBytes = (kHalves * kKVHalfBytes > kRows * 128) ? kHalves * kKVHalfBytes
                                                                            : kRows * 128;  // K or P
  static constexpr int kVSlotBytes = kHalves * kKVHalfBytes;
  static constexpr int kStageBytes = kKSlotBytes + kVSlotBytes;
  static constexpr int kBarOffset = kQBytes + kStages * kStageBytes;
  static constexpr int kSmemBytes = 1024 + kBarOffset + 128;
};

template <int D>
__global__ void __launch_bounds__(kThreads, 2)
    merge_tc_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                    const AttnParams p) {
  using Geo = TcGeo<D>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* base = smem_raw + ((1024u - (raw & 1023u)) & 1023u);
  uint8_t* q_s = base;
  uint8_t* ring = base + Geo::kQBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(base + Geo::kBarOffset);
  uint64_t* full = bars;            // [kStages]
  uint64_t* empty = bars + 2;       // [kStages]
  uint64_t* s_full = bars + 4;
  uint64_t* p_full = bars + 5;
  uint64_t* o_final = bars + 6;
  uint64_t* q_ready = bars + 7;
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 8);

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int kvh = blockIdx.y;
  const int layer = blockIdx.z;
  const int G = p.G;
  const int row_base = blockIdx.x * kRows;
  const int n_rows = min(kRows, p.T * G - row_base);
  const int t_first = row_base / G;
  const int t_last = (row_base + n_rows - 1) / G;
  const int n_pages = (p.L0 + t_last + 1 + kPageTokens - 1) / kPageTokens;
  const int n_tiles = (n_pages + kPagesPerStage - 1) / kPagesPerStage;
  const int n_valid_keys = p.L0 + p.T;
  const int min_limit = p.L0 + t_first + 1;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], 1);
    }
    mbar_init(s_full, 1);
    mbar_init(p_full, kSoftmaxThreads);
    mbar_init(o_final, 1);
    mbar_init(q_ready, kSoftmaxThreads);
    fence_mbar_init();
  }
  if (warp == kMmaWarp) tmem_alloc(tmem_slot, kTmemCols);
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  // ---- loader -----------------------------------------------------------------
  if (warp == kLoadWarp) {
    if (lane == 0) {
      prefetch_tensormap(&kmap);
      prefetch_tensormap(&vmap);
    }
    const uint64_t policy = l2_policy_evict_last();  // every CTA of this (layer, head) walks these pages
    const int32_t* ids = p.table + (int64_t)p.slot * p.max_pages;
    int base_id = 0;
    int cur = lane < n_pages ? ids[lane] : 0;
    int nxt = 32 + lane < n_pages ? ids[32 + lane] : 0;
    int j = 0;
    bool ok = true;
    for (; j < n_tiles; ++j) {
      const int s = j % kStages;
      if (j >= kStages) {
        int w = 1;
        if (lane == 0) w = mbar_wait(&empty[s], ((j / kStages) - 1) & 1) ? 1 : 0;
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
      int blk[kPagesPerStage];
#pragma unroll
      for (int q = 0; q < kPagesPerStage; ++q) blk[q] = __shfl_sync(0xffffffffu, cur, (page0 - base_id + q) & 31);
      if (lane == 0) {
        uint8_t* kst = ring + s * Geo::kStageBytes;
        uint8_t* vst = kst + Geo::kKSlotBytes;
        mbar_arrive_expect_tx(&full[s], (uint32_t)(np * 2 * Geo::kHalves * kPageTokens * 128));
        for (int q = 0; q < np; ++q) {
          int b = blk[q];
          if ((uint64_t)b >= (uint64_t)p.n_blocks) {
            atomicCAS(p.status, 0, kDevBadIndex);
            b = 0;
          }
          const int c3 = layer * (int)p.n_blocks + b;
#pragma unroll
          for (int h = 0; h < Geo::kHalves; ++h) {
            tma_load_4d(kst + h * Geo::kKVHalfBytes + q * kPageTokens * 128, &kmap, &full[s], 0, h,
                        kvh * kPageTokens, c3, policy);
            tma_load_4d(vst + h * Geo::kKVHalfBytes + q * kPageTokens * 128, &vmap, &full[s], 0, h,
                        kvh * kPageTokens, c3, policy);
          }
        }
      }
    }
    if (!ok && lane == 0) {
      atomicCAS(p.status, 0, kDevTimeout);
      for (int t = max(0, j - kStages); t < j; ++t) mbar_wait(&full[t % kStages], (t / kStages) & 1);
    }
    return;
  }

  // ---- MMA issuer ---------------------------------------------------------------
  if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc_s = tc_idesc_bf16(kRows, kKeys, 0, 0);
      constexpr uint32_t idesc_o = tc_idesc_bf16(kRows, D, 0, 1);
      const uint32_t q_addr = smem_addr(q_s);
      bool ok = mbar_wait(q_ready, 0);
      tc_fence_after_sync();
      for (int j = 0; ok && j < n_tiles; ++j) {
        const int s = j % kStages;
        if (!mbar_wait(&full[s], (j / kStages) & 1)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
        const uint32_t k_addr = smem_addr(ring + s * Geo::kStageBytes);
        const uint32_t v_addr = k_addr + Geo::kKSlotBytes;
#pragma unroll
        for (int h = 0; h < Geo::kHalves; ++h)
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            tc_mma_bf16(tmem + kTmemS, tc_desc_sw128(q_addr + h * kRows * 128 + kk * 32, 16, 1024),
                        tc_desc_sw128(k_addr + h * Geo::kKVHalfBytes + kk * 32, 16, 1024), idesc_s,
                        (h | kk) != 0);
        tc_commit(s_full);
        if (!mbar_wait(p_full, j & 1)) {
          ok = false;
          break;
        }
        tc_fence_after_sync();
#pragma unroll
        for (int ks = 0; ks < kKeys / 16; ++ks)
          tc_mma_bf16(tmem + kTmemO, tc_desc_sw128(k_addr + ks * 32, 16, 1024),
                      tc_desc_sw128(v_addr + ks * 16 * 128, Geo::kKVHalfBytes, 1024), idesc_o,
                      (j > 0 || ks > 0) ? 1u : 0u);
        tc_commit(&empty[s]);
      }
      tc_commit(o_final);
      if (!ok) atomicCAS(p.status, 0, kDevTimeout);
    }
    __syncwarp();
    named_barrier_sync(1, kSoftmaxThreads + 32);
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
    return;
  }

  // ---- softmax warps ------------------------------------------------------------
  const int r = threadIdx.x;
  const uint32_t t_lane = tmem + ((uint32_t)(warp * 32) << 16);
  const int gr = row_base + r;
  const bool valid = r < n_rows;
  const int qrow = valid ? gr / G : 0;
  const int head = valid ? kvh * G + gr % G : 0;
  const int limit = valid ? p.L0 + qrow + 1 : n_valid_keys;
  {
    const uint4* src = reinterpret_cast<const uint4*>(p.q + (((int64_t)layer * p.n_rows_q + qrow) * p.Hq + head) * D);
#pragma unroll
    for (int c = 0; c < D / 8; ++c) {
      const uint4 v = valid ? src[c] : make_uint4(0u, 0u, 0u, 0u);
      *reinterpret_cast<uint4*>(q_s + (c >> 3) * kRows * 128 + r * 128 + (((c & 7) ^ (r & 7)) << 4)) = v;
    }
    fence_proxy_async_smem();
    mbar_arrive(q_ready);
  }
  const float sl2 = p.scale_log2;
  float m_used = -1e30f, l = 0.f;
  bool ok = true;
  for (int j = 0; j < n_tiles; ++j) {
    const int s = j % kStages;
    const bool got = __all_sync(0xffffffffu, mbar_wait(s_full, j & 1));
    if (!got) {
      ok = false;
      break;
    }
    tc_fence_after_sync();
    float sc[kKeys];
    tmem_ld32(t_lane + kTmemS, sc);
    tmem_ld32(t_lane + kTmemS + 32, sc + 32);
    const int key0 = j * kKeys;
    const int np = min(kPagesPerStage, n_pages - j * kPagesPerStage);
    const int loaded = np * kPageTokens;
    const bool edge = key0 + kKeys > min_limit || loaded < kKeys;
    float mx = -INFINITY;
#pragma unroll
    for (int c = 0; c < kKeys; ++c) {
      float x = sc[c] * sl2;
      if (edge && (c >= loaded || key0 + c >= limit)) x = -INFINITY;
      sc[c] = x;
      mx = fmaxf(mx, x);
    }
    const float m_new = fmaxf(m_used, mx);
    const bool need = m_new > m_used + kRescaleThreshold;
    if (__any_sync(0xffffffffu, need)) {
      const float alpha = need ? ex2(m_used - m_new) : 1.f;
      if (j > 0) {
#pragma unroll 1
        for (int c0 = 0; c0 < D; c0 += 32) {
          float o[32];
          tmem_ld32(t_lane + kTmemO + c0, o);
#pragma unroll
          for (int i = 0; i < 32; ++i) o[i] *= alpha;
          tmem_st32(t_lane + kTmemO + c0, o);
        }
      }
      l *= alpha;
      if (need) m_used = m_new;
    }
    uint32_t pk[kKeys / 2];
    float rs = 0.f;
#pragma unroll
    for (int c = 0; c < kKeys; c += 2) {
      const float a = ex2(sc[c] - m_used), b = ex2(sc[c + 1] - m_used);
      rs += a + b;
      pk[c / 2] = pack_bf16(a, b);
    }
    l += rs;
    uint8_t* kslot = ring + s * Geo::kStageBytes;  // S_j has been consumed: P_j goes over K_j
#pragma unroll
    for (int c = 0; c < 8; ++c)
      *reinterpret_cast<uint4*>(kslot + r * 128 + ((c ^ (r & 7)) << 4)) =
          make_uint4(pk[4 * c], pk[4 * c + 1], pk[4 * c + 2], pk[4 * c + 3]);
    if (key0 + kKeys > n_valid_keys || loaded < kKeys) {
      // this stage's copies have landed (S_j was computed from them); zero V
      // rows of keys that are not valid so that P V never sees stale data
      mbar_wait(&full[s], (j / kStages) & 1);
      uint8_t* vslot = kslot + Geo::kKSlotBytes;
      const int c = r & 63, h = r >> 6;
      if (h < Geo::kHalves && (c >= loaded || key0 + c >= n_valid_keys)) {
#pragma unroll
        for (int x = 0; x < 8; ++x)
          *reinterpret_cast<uint4*>(vslot + h * Geo::kKVHalfBytes + c * 128 + x * 16) = make_uint4(0u, 0u, 0u, 0u);
      }
    }
    fence_proxy_async_smem();
    tc_fence_before_sync();
    mbar_arrive(p_full);
  }
  if (ok) ok = __all_sync(0xffffffffu, mbar_wait(o_final, 0));
  tc_fence_after_sync();
  if (ok) {
    const float inv = 1.f / l;
    float* dst = valid ? p.out_o + (((int64_t)layer * p.T + qrow) * p.Hq + head) * D : nullptr;
#pragma unroll 1
    for (int c0 = 0; c0 < D; c0 += 32) {
      float o[32];
      tmem_ld32(t_lane + kTmemO + c0, o);
      if (dst) {
#pragma unroll
        for (int i = 0; i < 32; i += 4)
          *reinterpret_cast<float4*>(dst + c0 + i) = make_float4(o[i] * inv, o[i + 1] * inv, o[i + 2] * inv, o[i + 3] * inv);
      }
    }
    if (valid) p.out_lse[((int64_t)layer * p.T + qrow) * p.Hq + head] = (m_used + log2f(l)) * kLn2;
  } else if (lane == 0) {
    atomicCAS(p.status, 0, kDevTimeout);
  }
  tc_fence_before_sync();
  named_barrier_sync(1, kSoftmaxThreads + 32);
}

template <int D>
cudaError_t launch_merge_tc_t(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(merge_tc_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         TcGeo<D>::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  const int n_tiles = (p.T * p.G + kRows - 1) / kRows;
  dim3 grid(n_tiles, p.Hkv, p.L);
  merge_tc_kernel<D><<<grid, kThreads, TcGeo<D>::kSmemBytes, s>>>(km, vm, p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_merge_tc(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p, int D,
                            cudaStream_t s) {
  if (p.T <= 0) return cudaSuccess;
  if (D == 128) return launch_merge_tc_t<128>(km, vm, p, s);
  if (D == 64) return launch_merge_tc_t<64>(km, vm, p, s);
  return cudaErrorInvalidValue;
}

}  // namespace st
