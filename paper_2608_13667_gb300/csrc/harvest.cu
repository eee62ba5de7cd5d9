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
// One CTA, a warp per branch.  A warp scans its branch 32 tokens at a time (the
// next chunk's load in flight while one is classified): a close
// tag ends an atom iff an open tag follows the previous close tag (in the
// chunk, or carried from the chunks before), and the atom starts at the last
// such open tag; ballots over the chunk find both.  The spans of the first
// `cap` atoms go to shared memory; thread 0 turns their lengths into output
// offsets; then the whole CTA copies the kept tokens.
#include "../../include/st.h"
#include "kernels.cuh"

namespace st {

namespace {

constexpr int kMaxHarvestBranches = 32;
constexpr int kMaxHarvestCap = 64;
constexpr int kHarvestWarps = 32;  // one warp per branch

// highest set bit of a non-zero mask
__device__ __forceinline__ int top_bit(uint32_t m) { return 31 - __clz(m); }

__global__ void __launch_bounds__(kHarvestWarps * 32) harvest_kernel(
    const int32_t* __restrict__ streams, int stride, const int32_t* __restrict__ lens, int n_br, int32_t open_id,
    int32_t close_id, int cap, int32_t* __restrict__ out_ids, int32_t* __restrict__ out_src,
    int32_t* __restrict__ out_atoms, int32_t* __restrict__ out_count) {
  __shared__ int32_t span_start[kMaxHarvestBranches][kMaxHarvestCap];
  __shared__ int32_t span_end[kMaxHarvestBranches][kMaxHarvestCap];
  __shared__ int32_t span_off[kMaxHarvestBranches][kMaxHarvestCap + 1];
  __shared__ int32_t n_atoms[kMaxHarvestBranches];
  __shared__ int32_t branch_off[kMaxHarvestBranches + 1];

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t below = (1u << lane) - 1u;
  for (int b = warp; b < n_br; b += kHarvestWarps) {
    const int32_t* s = streams + (int64_t)b * stride;
    int len = lens[b];
    len = len < 0 ? 0 : (len > stride ? stride : len);
    int open = -1;  // last open tag since the last close tag, or -1
    int k = 0;      // atoms found so far
    int32_t nxt = lane < len ? s[lane] : 0;
    for (int base = 0; base < len && k < cap; base += 32) {
      const int i = base + lane;
      const int32_t t = nxt;  // lanes past the stream match no tag (ballots test i < len)
      nxt = i + 32 < len ? s[i + 32] : 0;
      const uint32_t opens = __ballot_sync(0xffffffffu, i < len && t == open_id);
      const uint32_t closes = __ballot_sync(0xffffffffu, i < len && t == close_id);
      // the atom a close tag at this lane would end: the last open tag after
      // the previous close tag
      int start = -1;
      if (closes & (1u << lane)) {
        const uint32_t pc = closes & below;
        uint32_t om = opens & below;
        if (pc) om &= ~((2u << top_bit(pc)) - 1u);
        if (om) start = base + top_bit(om);
        else if (!pc) start = open;
      }
      const uint32_t ends = __ballot_sync(0xffffffffu, start >= 0);
      const int idx = k + __popc(ends & below);
      if (start >= 0 && idx < cap) {
        span_start[b][idx] = start;
        span_end[b][idx] = i;
      }
      k += __popc(ends);
      // carry: the last open tag after the chunk's last close tag
      if (closes) {
        const uint32_t om = opens & ~((2u << top_bit(closes)) - 1u);
        open = om ? base + top_bit(om) : -1;
      } else if (opens) {
        open = base + top_bit(opens);
      }
    }
    k = k < cap ? k : cap;
    if (lane == 0) {
      n_atoms[b] = k;
      int tok = 0;
      span_off[b][0] = 0;
      for (int a = 0; a < k; ++a) {
        tok += span_end[b][a] - span_start[b][a] + 1;
        span_off[b][a + 1] = tok;
      }
    }
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
  st::harvest_kernel<<<1, st::kHarvestWarps * 32, 0, static_cast<cudaStream_t>(stream)>>>(
      streams, stride, lens, n_br, open_id, close_id, cap, out_ids, out_src, out_atoms, out_count);
  return cudaGetLastError() == cudaSuccess ? ST_OK : ST_ERR_CUDA;
}
