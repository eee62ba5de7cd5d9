// Paged decode attention over block tables (split-KV partials + combine).
//
// Section 3.3 of the paper: all branches share the prompt prefix up to R_t, so
// the prefix KV is reused across every decoding stream; Section 4.4: branch
// load is dominated by those cached-prefix reads.  One CTA here owns one run
// of pages of one KV head of one layer and stacks every query row that reads
// that run -- for a shared prefix, all branches of the fork group x the G
// query heads of the KV head -- so each prefix page crosses HBM once per
// group instead of once per branch.
//
// CTA layout (128 threads): warps 0..2 compute, warp 3 loads; 3 CTAs per SM.
//   * Loader: reads page ids from the block table (32 at a time, one batch
//     ahead) and issues one 2 KiB TMA tensor copy per (page, 64-wide half of
//     the head, K|V) into a 4-stage ring of 2-page stages, signalling a
//     per-stage mbarrier with the byte count.
//   * Compute warp w owns query rows [16w, 16w+16).  Per stage it forms
//     S = Q K^T on the tensor cores (mma.sync m16n8k16 bf16 -> fp32; K
//     fragments by ldmatrix from the 128B-swizzled tiles), runs the online
//     softmax in the log2 domain (row max/sum via quad shuffles; the
//     accumulator is rescaled only when some row max grows), rounds P to bf16
//     and accumulates O += P V (V fragments by ldmatrix.trans).
// Each CTA writes a normalised partial (O_i, lse_i) per row into its split
// slot; combine_kernel merges a branch's partials by log-sum-exp.
//
// Key rows past the valid length of a partially filled last page may hold
// stale data; their scores are masked to -inf and their V values are zeroed
// in registers, so stale NaN/Inf bit patterns cannot leak into the output.
#include <math.h>

#include "kernels.cuh"
#include "ptx.cuh"

namespace st {

namespace {

constexpr int kPPS = 2;            // pages per pipeline stage (32 keys)
constexpr int kStages = 4;
constexpr int kComputeWarps = 3;   // up to 48 stacked query rows
constexpr int kThreads = (kComputeWarps + 1) * 32;
constexpr float kLn2 = 0.69314718055994530942f;

template <int D>
struct Geometry {
  static constexpr int kPageBytes = kPageTokens * D * 2;       // one page of one head (K or V)
  static constexpr int kHalfBytes = kPageTokens * 128;         // 16 tokens x 64 bf16
  static constexpr int kStageBytes = 2 * kPPS * kPageBytes;    // K pages, then V pages
  static constexpr int kRingBytes = kStages * kStageBytes;
  static constexpr int kSmemBytes = kRingBytes + 1024 + 2 * kStages * 8;
};

// Byte address of the 16-byte chunk holding (token, d) in a page tile laid
// out as [D/64 halves][16 tokens][64] with the TMA 128B swizzle (chunk index
// xor token % 8 inside each 128-byte line).
__device__ __forceinline__ uint32_t tile_chunk(uint32_t base, int token, int d) {
  const int half = d >> 6;
  const int chunk = (d & 63) >> 3;
  return base + half * (kPageTokens * 128) + token * 128 + ((chunk ^ (token & 7)) << 4);
}

__device__ __forceinline__ uint32_t ld_u32(const __nv_bfloat16* p) {
  return *reinterpret_cast<const uint32_t*>(p);
}

template <int D>
__global__ void __launch_bounds__(kThreads, 3)
    attend_kernel(const __grid_constant__ CUtensorMap kmap, const __grid_constant__ CUtensorMap vmap,
                  const AttnParams p) {
  using Geo = Geometry<D>;
  extern __shared__ uint8_t smem_raw[];
  const uint32_t raw = smem_addr(smem_raw);
  uint8_t* ring = smem_raw + ((1024u - (raw & 1023u)) & 1023u);
  uint64_t* full = reinterpret_cast<uint64_t*>(ring + Geo::kRingBytes);
  uint64_t* empty = full + kStages;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int kvh = blockIdx.y;
  const int layer = blockIdx.z;

  // ---- what this CTA reads and for whom -----------------------------------
  const AttnItem item = p.items[blockIdx.x];
  const int slot = item.slot;
  const int page_begin = item.page_begin;
  const int n_pages = item.n_pages;
  const int n_valid_keys = item.n_tokens;  // keys past this in the last page are stale
  const int n_rows = item.n_members * p.G;
  const int n_cw = (n_rows + 15) >> 4;
  const int n_stages = (n_pages + kPPS - 1) / kPPS;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(&full[s], 1);
      mbar_init(&empty[s], n_cw);
    }
    fence_mbar_init();
  }
  __syncthreads();

  // ---- loader warp ---------------------------------------------------------
  if (warp == kComputeWarps) {
    if (lane == 0) {
      prefetch_tensormap(&kmap);
      prefetch_tensormap(&vmap);
    }
    // each page is streamed once: keep it out of L2's way
    const uint64_t policy = l2_policy_evict_first();
    const int32_t* ids = p.table + (int64_t)slot * p.max_pages + page_begin;
    int base = 0;
    int cur = lane < n_pages ? ids[lane] : 0;
    int nxt = 32 + lane < n_pages ? ids[32 + lane] : 0;
    int st = 0;
    bool ok = true;
    for (; st < n_stages; ++st) {
      const int s = st % kStages;
      if (st >= kStages) {
        int w = 1;
        if (lane == 0) w = mbar_wait(&empty[s], ((st / kStages) - 1) & 1) ? 1 : 0;
        w = __shfl_sync(0xffffffffu, w, 0);
        if (!w) {
          ok = false;
          break;
        }
      }
      const int page0 = st * kPPS;
      if (page0 >= base + 32) {
        base += 32;
        cur = nxt;
        nxt = base + 32 + lane < n_pages ? ids[base + 32 + lane] : 0;
      }
      const int np = min(kPPS, n_pages - page0);
      int blk[kPPS];
#pragma unroll
      for (int q = 0; q < kPPS; ++q) blk[q] = __shfl_sync(0xffffffffu, cur, (page0 - base + q) & 31);
      if (lane == 0) {
        uint8_t* kst = ring + s * Geo::kStageBytes;
        uint8_t* vst = kst + kPPS * Geo::kPageBytes;
        mbar_arrive_expect_tx(&full[s], (uint32_t)(np * 2 * Geo::kPageBytes));
        for (int q = 0; q < np; ++q) {
          int b = blk[q];
          if ((uint64_t)b >= (uint64_t)p.n_blocks) {
            atomicCAS(p.status, 0, kDevBadIndex);
            b = 0;
          }
          const int c3 = layer * (int)p.n_blocks + b;
#pragma unroll
          for (int h = 0; h < D / 64; ++h) {
            tma_load_4d(kst + q * Geo::kPageBytes + h * Geo::kHalfBytes, &kmap, &full[s], 0, h,
                        kvh * kPageTokens, c3, policy);
            tma_load_4d(vst + q * Geo::kPageBytes + h * Geo::kHalfBytes, &vmap, &full[s], 0, h,
                        kvh * kPageTokens, c3, policy);
          }
        }
      }
    }
    if (!ok && lane == 0) {
      atomicCAS(p.status, 0, kDevTimeout);
      // let copies already issued land before the CTA's shared memory goes away
      for (int t = max(0, st - kStages); t < st; ++t) mbar_wait(&full[t % kStages], (t / kStages) & 1);
    }
    return;
  }
  if (warp >= n_cw) return;

  // ---- compute warps -------------------------------------------------------
  const int r0 = warp * 16 + (lane >> 2);
  const int r1 = r0 + 8;
  const int quad = lane & 3;

  // query row -> (branch of the call, head)
  const bool v0 = r0 < n_rows, v1 = r1 < n_rows;
  const int qrow0 = v0 ? p.members[item.member_base + r0 / p.G] : 0;
  const int head0 = v0 ? kvh * p.G + r0 % p.G : 0;
  const int qrow1 = v1 ? p.members[item.member_base + r1 / p.G] : 0;
  const int head1 = v1 ? kvh * p.G + r1 % p.G : 0;

  uint32_t qa[D / 16][4];
  {
    const __nv_bfloat16* q0 = p.q + (((int64_t)layer * p.n_rows_q + qrow0) * p.Hq + head0) * D;
    const __nv_bfloat16* q1 = p.q + (((int64_t)layer * p.n_rows_q + qrow1) * p.Hq + head1) * D;
#pragma unroll
    for (int kk = 0; kk < D / 16; ++kk) {
      const int c = kk * 16 + 2 * quad;
      qa[kk][0] = v0 ? ld_u32(q0 + c) : 0u;
      qa[kk][1] = v1 ? ld_u32(q1 + c) : 0u;
      qa[kk][2] = v0 ? ld_u32(q0 + c + 8) : 0u;
      qa[kk][3] = v1 ? ld_u32(q1 + c + 8) : 0u;
    }
  }

  float acc[D / 8][4];
#pragma unroll
  for (int n = 0; n < D / 8; ++n) acc[n][0] = acc[n][1] = acc[n][2] = acc[n][3] = 0.f;
  float m0 = -1e30f, m1 = -1e30f, l0 = 0.f, l1 = 0.f;
  const float sl2 = p.scale_log2;

  // per-lane ldmatrix offsets
  const int k_tok = lane & 7;                              // K: token within an 8-key n-tile
  const int k_dof = 8 * (lane >> 3);                       // K: d offset of this lane's matrix
  const int v_tok = (lane & 7) + 8 * ((lane >> 3) & 1);    // V^T: token row
  const int v_dof = 8 * (lane >> 4);                       // V^T: d offset

  bool ok = true;
  for (int st = 0; st < n_stages; ++st) {
    const int s = st % kStages;
    if (!mbar_wait(&full[s], (st / kStages) & 1)) {
      ok = false;
      break;
    }
    const int np = min(kPPS, n_pages - st * kPPS);
    const uint32_t kbase = smem_addr(ring + s * Geo::kStageBytes);
    const uint32_t vbase = kbase + kPPS * Geo::kPageBytes;
    const int key0 = st * kPPS * kPageTokens;

    float sc[kPPS][2][4];
#pragma unroll
    for (int q = 0; q < kPPS; ++q) {
#pragma unroll
      for (int j = 0; j < 2; ++j) sc[q][j][0] = sc[q][j][1] = sc[q][j][2] = sc[q][j][3] = 0.f;
      if (q < np) {
        const uint32_t kt = kbase + q * Geo::kPageBytes;
#pragma unroll
        for (int j = 0; j < 2; ++j) {
#pragma unroll
          for (int kk = 0; kk < D / 32; ++kk) {
            uint32_t b0, b1, b2, b3;
            ldsm_x4(tile_chunk(kt, 8 * j + k_tok, 32 * kk + k_dof), b0, b1, b2, b3);
            mma_bf16(sc[q][j], qa[2 * kk][0], qa[2 * kk][1], qa[2 * kk][2], qa[2 * kk][3], b0, b1);
            mma_bf16(sc[q][j], qa[2 * kk + 1][0], qa[2 * kk + 1][1], qa[2 * kk + 1][2],
                     qa[2 * kk + 1][3], b2, b3);
          }
        }
      }
    }

    // scale to the log2 domain, mask keys past the run, row maxima
    const bool edge = key0 + kPPS * kPageTokens > n_valid_keys;
    float mx0 = -INFINITY, mx1 = -INFINITY;
#pragma unroll
    for (int q = 0; q < kPPS; ++q) {
#pragma unroll
      for (int j = 0; j < 2; ++j) {
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          const int key = key0 + q * kPageTokens + j * 8 + 2 * quad + (e & 1);
          float x = sc[q][j][e] * sl2;
          if (q >= np || (edge && key >= n_valid_keys)) x = -INFINITY;
          sc[q][j][e] = x;
        }
        mx0 = fmaxf(mx0, fmaxf(sc[q][j][0], sc[q][j][1]));
        mx1 = fmaxf(mx1, fmaxf(sc[q][j][2], sc[q][j][3]));
      }
    }
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 1));
    mx0 = fmaxf(mx0, __shfl_xor_sync(0xffffffffu, mx0, 2));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 1));
    mx1 = fmaxf(mx1, __shfl_xor_sync(0xffffffffu, mx1, 2));
    const float mn0 = fmaxf(m0, mx0), mn1 = fmaxf(m1, mx1);
    if (__any_sync(0xffffffffu, (mn0 > m0) || (mn1 > m1))) {
      const float a0 = ex2(m0 - mn0), a1 = ex2(m1 - mn1);
      l0 *= a0;
      l1 *= a1;
#pragma unroll
      for (int n = 0; n < D / 8; ++n) {
        acc[n][0] *= a0;
        acc[n][1] *= a0;
        acc[n][2] *= a1;
        acc[n][3] *= a1;
      }
      m0 = mn0;
      m1 = mn1;
    }

    const bool vmask_stage = key0 + kPPS * kPageTokens > n_valid_keys;
#pragma unroll
    for (int q = 0; q < kPPS; ++q) {
      if (q < np) {
        float e[2][4];
#pragma unroll
        for (int j = 0; j < 2; ++j) {
          e[j][0] = ex2(sc[q][j][0] - m0);
          e[j][1] = ex2(sc[q][j][1] - m0);
          e[j][2] = ex2(sc[q][j][2] - m1);
          e[j][3] = ex2(sc[q][j][3] - m1);
          l0 += e[j][0] + e[j][1];
          l1 += e[j][2] + e[j][3];
        }
        const uint32_t pa0 = pack_bf16(e[0][0], e[0][1]);
        const uint32_t pa1 = pack_bf16(e[0][2], e[0][3]);
        const uint32_t pa2 = pack_bf16(e[1][0], e[1][1]);
        const uint32_t pa3 = pack_bf16(e[1][2], e[1][3]);
        const uint32_t vt = vbase + q * Geo::kPageBytes;
        const int nv = n_valid_keys - (key0 + q * kPageTokens);  // valid keys in this page
        const bool vm = vmask_stage && nv < kPageTokens;
        const int tk = 2 * quad;
        const uint32_t mk0 = (tk < nv ? 0x0000ffffu : 0u) | (tk + 1 < nv ? 0xffff0000u : 0u);
        const uint32_t mk1 = (tk + 8 < nv ? 0x0000ffffu : 0u) | (tk + 9 < nv ? 0xffff0000u : 0u);
#pragma unroll
        for (int nn = 0; nn < D / 16; ++nn) {
          uint32_t b0, b1, b2, b3;
          ldsm_x4_t(tile_chunk(vt, v_tok, 16 * nn + v_dof), b0, b1, b2, b3);
          if (vm) {
            b0 &= mk0;
            b1 &= mk1;
            b2 &= mk0;
            b3 &= mk1;
          }
          mma_bf16(acc[2 * nn], pa0, pa1, pa2, pa3, b0, b1);
          mma_bf16(acc[2 * nn + 1], pa0, pa1, pa2, pa3, b2, b3);
        }
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(&empty[s]);
  }
  if (!ok) {
    if (lane == 0) atomicCAS(p.status, 0, kDevTimeout);
    return;
  }

  // ---- epilogue -------------------------------------------------------------
  l0 += __shfl_xor_sync(0xffffffffu, l0, 1);
  l0 += __shfl_xor_sync(0xffffffffu, l0, 2);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 1);
  l1 += __shfl_xor_sync(0xffffffffu, l1, 2);
  const float inv0 = 1.f / l0, inv1 = 1.f / l1;
  float *o0 = nullptr, *o1 = nullptr, *s0 = nullptr, *s1 = nullptr;
  if (v0) {
    const int64_t i0 = (((int64_t)layer * p.n_rows_q + qrow0) * p.Hq + head0) * p.max_splits + item.split;
    o0 = p.out_o + i0 * D;
    s0 = p.out_lse + i0;
  }
  if (v1) {
    const int64_t i1 = (((int64_t)layer * p.n_rows_q + qrow1) * p.Hq + head1) * p.max_splits + item.split;
    o1 = p.out_o + i1 * D;
    s1 = p.out_lse + i1;
  }
#pragma unroll
  for (int n = 0; n < D / 8; ++n) {
    const int col = n * 8 + 2 * quad;
    if (o0) *reinterpret_cast<float2*>(o0 + col) = make_float2(acc[n][0] * inv0, acc[n][1] * inv0);
    if (o1) *reinterpret_cast<float2*>(o1 + col) = make_float2(acc[n][2] * inv1, acc[n][3] * inv1);
  }
  if (quad == 0) {
    if (s0) *s0 = (m0 + log2f(l0)) * kLn2;
    if (s1) *s1 = (m1 + log2f(l1)) * kLn2;
  }
}

// One warp per (layer, branch, query head): lse = log sum_i exp(lse_i),
// O = sum_i exp(lse_i - lse) O_i over the branch's partials.
template <int D>
__global__ void __launch_bounds__(128) combine_kernel(const CombineParams p) {
  const int lane = threadIdx.x & 31;
  const int64_t idx = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  const int64_t total = (int64_t)p.L * p.n_br * p.Hq;
  if (idx >= total) return;
  const int b = (int)((idx / p.Hq) % p.n_br);
  const int ns = p.n_splits[b];
  const float* lse_i = p.part_lse + idx * p.max_splits;
  const float li = lane < ns ? lse_i[lane] : -INFINITY;
  float mx = li;
#pragma unroll
  for (int o = 16; o; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  const float w = lane < ns ? expf(li - mx) : 0.f;
  float sum = w;
#pragma unroll
  for (int o = 16; o; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
  const float lse = mx + logf(sum);
  constexpr int kPer = D / 32;
  float out[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) out[e] = 0.f;
  const float* po = p.part_o + idx * p.max_splits * D + lane * kPer;
  for (int i = 0; i < ns; ++i) {
    const float wi = __shfl_sync(0xffffffffu, w, i) / sum;
    if (kPer == 4) {
      const float4 x = *reinterpret_cast<const float4*>(po + (int64_t)i * D);
      out[0] += wi * x.x;
      out[1] += wi * x.y;
      out[2] += wi * x.z;
      out[3] += wi * x.w;
    } else {
      const float2 x = *reinterpret_cast<const float2*>(po + (int64_t)i * D);
      out[0] += wi * x.x;
      out[1] += wi * x.y;
    }
  }
  float* dst = p.o + idx * D + lane * kPer;
  if (kPer == 4)
    *reinterpret_cast<float4*>(dst) = make_float4(out[0], out[1], out[2], out[3]);
  else
    *reinterpret_cast<float2*>(dst) = make_float2(out[0], out[1]);
  if (lane == 0) p.lse[idx] = lse;
}

template <int D>
cudaError_t launch_attend_t(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p,
                            int n_ctas, cudaStream_t s) {
  static bool configured = false;
  if (!configured) {
    cudaError_t e = cudaFuncSetAttribute(attend_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         Geometry<D>::kSmemBytes);
    if (e != cudaSuccess) return e;
    configured = true;
  }
  dim3 grid(n_ctas, p.Hkv, p.L);
  attend_kernel<D><<<grid, kThreads, Geometry<D>::kSmemBytes, s>>>(km, vm, p);
  return cudaGetLastError();
}

template <int D>
int ctas_per_sm_t() {
  cudaError_t e = cudaFuncSetAttribute(attend_kernel<D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       Geometry<D>::kSmemBytes);
  if (e != cudaSuccess) return 0;
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attend_kernel<D>, kThreads,
                                                    Geometry<D>::kSmemBytes) != cudaSuccess)
    return 0;
  return n;
}

}  // namespace

cudaError_t launch_attend(const CUtensorMap& km, const CUtensorMap& vm, const AttnParams& p,
                          int n_ctas, int D, cudaStream_t s) {
  if (n_ctas <= 0) return cudaSuccess;
  if (D == 128) return launch_attend_t<128>(km, vm, p, n_ctas, s);
  if (D == 64) return launch_attend_t<64>(km, vm, p, n_ctas, s);
  return cudaErrorInvalidValue;
}

int attend_ctas_per_sm(int D) {
  if (D == 128) return ctas_per_sm_t<128>();
  if (D == 64) return ctas_per_sm_t<64>();
  return 0;
}

cudaError_t launch_combine(const CombineParams& p, int D, cudaStream_t s) {
  const int64_t total = (int64_t)p.L * p.n_br * p.Hq;
  if (total == 0) return cudaSuccess;
  const int grid = (int)((total + 3) / 4);
  if (D == 128)
    combine_kernel<128><<<grid, 128, 0, s>>>(p);
  else if (D == 64)
    combine_kernel<64><<<grid, 128, 0, s>>>(p);
  else
    return cudaErrorInvalidValue;
  return cudaGetLastError();
}

}  // namespace st
