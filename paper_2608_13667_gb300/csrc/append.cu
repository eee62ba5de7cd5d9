// Block-table refresh and the KV append (scatter + copy-on-write).
//
// The host owns the allocator; the device keeps a copy of every live block
// table.  An append call first refreshes the table entries the host changed
// (table_update), then one launch of append_kv performs the call's
// copy-on-write page copies and writes its new rows.  The two parts of
// append_kv never touch the same row: a copy fills rows [0, off) of a fresh
// page and the appended rows start at row off, so they need no ordering.
#include "kernels.cuh"

namespace st {

namespace {

__global__ void table_update_kernel(int32_t* __restrict__ table, const TableRun* __restrict__ runs,
                                    const int32_t* __restrict__ values, int n_runs) {
  griddep_wait();
  griddep_launch_dependents();
  for (int r = blockIdx.x; r < n_runs; r += gridDim.x) {
    const TableRun run = runs[r];
    for (int i = threadIdx.x; i < run.count; i += blockDim.x) table[run.dst + i] = values[run.src + i];
  }
}

// One thread moves 16 bytes (8 bf16).  Index space: copy-on-write chunks
// first (n_cow x L x Hkv x 16 rows x D/8, rows past the copy length idle),
// then the appended rows in the input's own order [L][n_rows][Hkv][D/8];
// row r belongs to the branch whose [row0, row0 + n) holds it.
template <int D>
__global__ void __launch_bounds__(256) append_kernel(const AppendParams p,
                                                     const __grid_constant__ InlineAppendPlan inl) {
  griddep_wait();
  griddep_launch_dependents();
  const AppendBranch* branches = p.branches ? p.branches : inl.branches;
  const CowCopy* cows = p.cows ? p.cows : inl.cows;
  constexpr int kChunks = D / 8;
  const int64_t cow_total = (int64_t)p.n_cow * p.L * p.Hkv * kPageTokens * kChunks;
  const int64_t app_total = (int64_t)p.L * p.n_rows * p.Hkv * kChunks;
  const int64_t total = cow_total + app_total;
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total; i += stride) {
    if (i < cow_total) {
      int64_t x = i;
      const int c = (int)(x % kChunks); x /= kChunks;
      const int row = (int)(x % kPageTokens); x /= kPageTokens;
      const int g = (int)(x % p.Hkv); x /= p.Hkv;
      const int l = (int)(x % p.L); x /= p.L;
      const CowCopy cw = cows[x];
      if (row >= cw.rows) continue;
      if ((uint64_t)cw.src_block >= (uint64_t)p.n_blocks ||
          (uint64_t)cw.dst_block >= (uint64_t)p.n_blocks) {
        atomicCAS(p.status, 0, kDevBadIndex);
        continue;
      }
      const int64_t src = ((((int64_t)l * p.n_blocks + cw.src_block) * p.Hkv + g) * kPageTokens + row) * D + c * 8;
      const int64_t dst = ((((int64_t)l * p.n_blocks + cw.dst_block) * p.Hkv + g) * kPageTokens + row) * D + c * 8;
      *reinterpret_cast<uint4*>(p.k_pool + dst) = *reinterpret_cast<const uint4*>(p.k_pool + src);
      *reinterpret_cast<uint4*>(p.v_pool + dst) = *reinterpret_cast<const uint4*>(p.v_pool + src);
    } else {
      const int64_t j = i - cow_total;
      int64_t x = j;
      const int c = (int)(x % kChunks); x /= kChunks;
      const int g = (int)(x % p.Hkv); x /= p.Hkv;
      const int row = (int)(x % p.n_rows); x /= p.n_rows;
      const int l = (int)x;
      int b;
      if (p.ragged) {  // the last branch whose first row is <= row
        int lo = 0, hi = p.n_br - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (branches[mid].row0 <= row) lo = mid;
          else hi = mid - 1;
        }
        b = lo;
      } else {
        b = row / p.n_tok;
      }
      const AppendBranch br = branches[b];
      const int pos = br.start + (row - br.row0);
      const int32_t blk = p.table[(int64_t)br.slot * p.max_pages + pos / kPageTokens];
      if ((uint64_t)blk >= (uint64_t)p.n_blocks) {
        atomicCAS(p.status, 0, kDevBadIndex);
        continue;
      }
      const int64_t dst = ((((int64_t)l * p.n_blocks + blk) * p.Hkv + g) * kPageTokens + (pos % kPageTokens)) * D + c * 8;
      *reinterpret_cast<uint4*>(p.k_pool + dst) = *reinterpret_cast<const uint4*>(p.k + j * 8);
      *reinterpret_cast<uint4*>(p.v_pool + dst) = *reinterpret_cast<const uint4*>(p.v + j * 8);
    }
  }
}

int grid_for(int64_t total, int threads) {
  static int sms_of[64] = {};
  int dev = 0, sms = 148;
  cudaGetDevice(&dev);
  if (dev >= 0 && dev < 64) {
    if (!sms_of[dev]) cudaDeviceGetAttribute(&sms_of[dev], cudaDevAttrMultiProcessorCount, dev);
    if (sms_of[dev] > 0) sms = sms_of[dev];
  }
  const int64_t want = (total + threads - 1) / threads;
  const int64_t cap = (int64_t)sms * 16;
  return (int)(want < 1 ? 1 : (want > cap ? cap : want));
}

}  // namespace

cudaError_t launch_table_update(int32_t* table, const TableRun* runs, const int32_t* values,
                                int n_runs, cudaStream_t s) {
  if (n_runs <= 0) return cudaSuccess;
  const int grid = n_runs < 1024 ? n_runs : 1024;
  return launch_chained(table_update_kernel, dim3(grid), dim3(256), 0, s, table, runs, values, n_runs);
}

cudaError_t launch_append(const AppendParams& p, const InlineAppendPlan* inl, int D, cudaStream_t s) {
  static const InlineAppendPlan kNone{};
  const InlineAppendPlan& ip = inl ? *inl : kNone;
  const int64_t total = (int64_t)p.n_cow * p.L * p.Hkv * kPageTokens * (D / 8) +
                        (int64_t)p.L * p.n_rows * p.Hkv * (D / 8);
  if (total == 0) return cudaSuccess;
  const int grid = grid_for(total, 256);
  if (D == 128) return launch_chained(append_kernel<128>, dim3(grid), dim3(256), 0, s, p, ip);
  if (D == 64) return launch_chained(append_kernel<64>, dim3(grid), dim3(256), 0, s, p, ip);
  return cudaErrorInvalidValue;
}

}  // namespace st
