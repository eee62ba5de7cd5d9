// Log-sum-exp combine of split-KV decode partials.
//
// A branch's decode is split into runs of pages (shared-prefix runs read for
// the whole fork group, and the branch's own runs); each run yields a
// normalised partial O_i with its log-sum-exp lse_i.  Since softmax over the
// union of disjoint key sets is the lse-weighted mixture of the per-set
// softmaxes, lse = log sum_i exp(lse_i) and O = sum_i exp(lse_i - lse) O_i.
#include <math.h>

#include "kernels.cuh"

namespace st {

namespace {

// One row (one layer, branch and query head) for one warp: lse = log sum_i
// exp(lse_i), O = sum_i exp(lse_i - lse) O_i over the row's ns partials
// (ns <= 32).
template <int D>
__device__ __forceinline__ void combine_row(const float* lse_i, const float* part_o, int ns, float* o_out,
                                            float* lse_out, int lane) {
  constexpr int kPer = D / 32;
  constexpr int kBatch = 16;  // partials whose loads are in flight together
  const float* po = part_o + lane * kPer;
  // this lane's column slice of partial i (zero past the row's partials)
  auto load = [&](int i, float* x) {
    if (i < ns) {
      if constexpr (kPer == 4) {
        const float4 v = __ldcg(reinterpret_cast<const float4*>(po + (int64_t)i * D));
        x[0] = v.x;
        x[1] = v.y;
        x[2] = v.z;
        x[3] = v.w;
      } else {
        const float2 v = __ldcg(reinterpret_cast<const float2*>(po + (int64_t)i * D));
        x[0] = v.x;
        x[1] = v.y;
      }
    } else {
#pragma unroll
      for (int e = 0; e < kPer; ++e) x[e] = 0.f;
    }
  };
  // the first batch of partials is loaded together with the lse values: the
  // loads do not depend on the weights
  const float li = lane < ns ? __ldcg(lse_i + lane) : -INFINITY;
  float x[kBatch][kPer];
#pragma unroll
  for (int u = 0; u < kBatch; ++u) load(u, x[u]);
  float mx = li;
#pragma unroll
  for (int off = 16; off; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  const float w = lane < ns ? expf(li - mx) : 0.f;
  float sum = w;
#pragma unroll
  for (int off = 16; off; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
  const float lse = mx + logf(sum);
  const float inv_sum = 1.f / sum;
  float out[kPer];
#pragma unroll
  for (int e = 0; e < kPer; ++e) out[e] = 0.f;
  for (int i0 = 0; i0 < ns; i0 += kBatch) {
    if (i0 > 0) {
#pragma unroll
      for (int u = 0; u < kBatch; ++u) load(i0 + u, x[u]);
    }
#pragma unroll
    for (int u = 0; u < kBatch; ++u) {
      const float wv = i0 + u < ns ? __shfl_sync(0xffffffffu, w, (i0 + u) & 31) * inv_sum : 0.f;
#pragma unroll
      for (int e = 0; e < kPer; ++e) out[e] += wv * x[u][e];
    }
  }
  float* dst = o_out + lane * kPer;
  if constexpr (kPer == 4)
    *reinterpret_cast<float4*>(dst) = make_float4(out[0], out[1], out[2], out[3]);
  else
    *reinterpret_cast<float2*>(dst) = make_float2(out[0], out[1]);
  if (lane == 0) *lse_out = lse;
}


// One warp per (layer, branch, query head).
template <int D>
__global__ void __launch_bounds__(128) combine_kernel(const CombineParams p, const __grid_constant__ InlineSplits inl) {
  griddep_wait();
  griddep_launch_dependents();
  const int32_t* n_splits = p.n_splits ? p.n_splits : inl.n_splits;
  const int lane = threadIdx.x & 31;
  const int64_t idx = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  const int64_t total = (int64_t)p.L * p.n_br * p.Hq;
  if (idx >= total) return;
  const int b = (int)((idx / p.Hq) % p.n_br);
  combine_row<D>(p.part_lse + idx * p.max_splits, p.part_o + idx * p.max_splits * D, n_splits[b], p.o + idx * D,
                 p.lse + idx, lane);
}

}  // namespace

cudaError_t launch_combine(const CombineParams& p, const InlineSplits* inl, int D, cudaStream_t s) {
  static const InlineSplits kNone{};
  const InlineSplits& ip = inl ? *inl : kNone;
  const int64_t total = (int64_t)p.L * p.n_br * p.Hq;
  if (total == 0) return cudaSuccess;
  const int grid = (int)((total + 3) / 4);
  if (D == 128) return launch_chained(combine_kernel<128>, dim3(grid), dim3(128), 0, s, p, ip);
  if (D == 64) return launch_chained(combine_kernel<64>, dim3(grid), dim3(128), 0, s, p, ip);
  return cudaErrorInvalidValue;
}

}  // namespace st
