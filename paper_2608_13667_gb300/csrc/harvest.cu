// Thought harvest on the device (Section 3.5 of the paper).
//
// When the observation arrives, every branch's generated token stream is cut
// at its last closed </thought>: completed atoms (an open-tag token through
// the next close-tag token, tags included) are kept, the first `cap` per
// branch, an unfinished atom is dropped, and a branch with no completed atom
// contributes nothing.  The kept atoms are concatenated in branch order; the
// result's length T is what st_merge appends to the main sequence (T = 0:
// nothing harvested, plain ReAct).  An open tag inside an unfinished atom
// restarts the atom; a close tag outside an atom is ignored.
//
// One CTA: thread b scans branch b and records the spans of its first `cap`
// completed atoms in shared memory; thread 0 turns span lengths into output
// offsets; then the whole CTA copies the kept tokens.
#include "../../include/st.h"
#include "kernels.cuh"

namespace st {

namespace {

constexpr int kMaxHarvestBranches = 32;
constexpr int kMaxHarvestCap = 64;

__global__ void __launch_bounds__(256) harvest_kernel(const int32_t* __restrict__ streams, int stride,
                                                      const int32_t* __restrict__ lens, int n_br, int32_t open_id,
                                                      int32_t close_id, int cap, int32_t* __restrict__ out_ids,
                                                      int32_t* __restrict__ out_src, int32_t* __restrict__ out_atoms,
                                                      int32_t* __restrict__ out_count) {
  __shared__ int32_t span_start[kMaxHarvestBranches][kMaxHarvestCap];
  __shared__ int32_t span_off[kMaxHarvestBranches][kMaxHarvestCap + 1];
  __shared__ int32_t n_atoms[kMaxHarvestBranches];
  __shared__ int32_t branch_off[kMaxHarvestBranches + 1];

  const int b = threadIdx.x;
  if (b < n_br) {
    const int32_t* s = streams + (int64_t)b * stride;
    int len = lens[b];
    len = len < 0 ? 0 : (len > stride ? stride : len);
    int open = -1, k = 0, tok = 0;
    span_off[b][0] = 0;
    for (int i = 0; i < len && k < cap; ++i) {
      const int32_t t = s[i];
      if (t == open_id) {
        open = i;
      } else if (t == close_id && open >= 0) {
        span_start[b][k] = open;
        tok += i - open + 1;
        span_off[b][k + 1] = tok;
        ++k;
        open = -1;
      }
    }
    n_atoms[b] = k;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    int total = 0;
    for (int i = 0; i < n_br; ++i) {
      branch_off[i] = total;
      total += span_off[i][n_atoms[i]];
      if (out_atoms) out_atoms[i] = n_atoms[i];
    }
    branch_off[n_br] = total;
    *out_count = total;
  }
  __syncthreads();
  for (int i = 0; i < n_br; ++i) {
    const int32_t* s = streams + (int64_t)i * stride;
    const int n = span_off[i][n_atoms[i]];
    for (int x = threadIdx.x; x < n; x += blockDim.x) {
      // atom containing output slot x of branch i (few atoms: linear search)
      int a = 0;
      while (span_off[i][a + 1] <= x) ++a;
      const int pos = span_start[i][a] + (x - span_off[i][a]);
      out_ids[branch_off[i] + x] = s[pos];
      if (out_src) out_src[branch_off[i] + x] = i * stride + pos;
    }
  }
}

}  // namespace

}  // namespace st

extern "C" ST_API st_status st_harvest(const int32_t* streams, int stride, const int32_t* lens, int n_br,
                                       int32_t open_id, int32_t close_id, int cap, int32_t* out_ids,
                                       int32_t* out_src, int32_t* out_atoms, int32_t* out_count, void* stream) {
  if (!streams || !lens || !out_ids || !out_count || stride < 1 || n_br < 1 ||
      n_br > st::kMaxHarvestBranches || cap < 0 || cap > st::kMaxHarvestCap || open_id == close_id)
    return ST_ERR_INVALID;
  st::harvest_kernel<<<1, 256, 0, static_cast<cudaStream_t>(stream)>>>(streams, stride, lens, n_br, open_id,
                                                                        close_id, cap, out_ids, out_src, out_atoms,
                                                                        out_count);
  return cudaGetLastError() == cudaSuccess ? ST_OK : ST_ERR_CUDA;
}
