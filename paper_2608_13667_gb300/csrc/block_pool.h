// Host-side paged KV block pool: free FIFO, per-page refcounts, per-sequence
// block tables, fork / append (copy-on-write) / release.  Pure C++, no CUDA.
//
// Section 3.3 of the paper: every branch receives the snapshot H_t + R_t, so
// the prefix KV is shared by all decoding streams.  Here that sharing is a
// block table copied at fork time with one reference taken per page; a
// shared page is never written -- the first appender to a shared partial
// page copies it.  The allocation order is fixed so that any two
// implementations of these rules produce identical tables:
//   * free FIFO starts as Fisher-Yates(splitmix64(seed)) over [0, n_blocks):
//     for i = n-1 .. 1: j = next() % (i + 1); swap(i, j).  Pop from the head.
//   * append: new page when len % page == 0; else copy-on-write when the last
//     page's refcount > 1 (the copy is allocated before any new page).
//   * release: drop references in logical order; zeros go to the FIFO tail.
#pragma once

#include <cstdint>
#include <vector>

namespace st {

struct CowEvent {
  int32_t src_block;
  int32_t dst_block;
  int32_t rows;  // rows [0, rows) are copied, for every layer and KV head
};

struct SeqSlot {
  uint32_t gen = 0;   // generation; bumped on release
  bool live = false;
  int32_t family = -1;  // id of the root sequence this one descends from (by fork)
  int64_t len = 0;
  std::vector<int32_t> table;
  // table entries [dirty_lo, dirty_hi) changed since the device copy was refreshed
  int32_t dirty_lo = 0, dirty_hi = 0;
  void mark_dirty(int32_t lo, int32_t hi) {
    if (lo >= hi) return;
    if (dirty_lo >= dirty_hi) { dirty_lo = lo; dirty_hi = hi; return; }
    if (lo < dirty_lo) dirty_lo = lo;
    if (hi > dirty_hi) dirty_hi = hi;
  }
};

class BlockPool {
 public:
  BlockPool(int64_t n_blocks, uint64_t seed, int page_size, int max_seqs, int max_pages);

  int64_t n_blocks() const { return n_blocks_; }
  int page_size() const { return page_; }
  int max_seqs() const { return (int)slots_.size(); }
  int max_pages() const { return max_pages_; }
  int64_t free_count() const { return free_count_; }

  // -1 when no slot is free.
  int create_seq();
  // Fills out[n_aux] with new slots; false (no change) when slots run out.
  bool fork(int parent, int n_aux, int* out);
  // Fork from the parent's first `length` rows (0 <= length <= parent length):
  // the children take the first ceil(length / page) table entries.
  bool fork_at(int parent, int64_t length, int n_aux, int* out);
  // Pages an append of n_tok rows to `slot` takes from the free list.
  int64_t pages_needed(int slot, int64_t n_tok) const;
  // Would the table outgrow max_pages?
  bool fits(int slot, int64_t n_tok) const;
  // Appends n_tok rows to each slot in order.  Precondition: the caller has
  // checked the total pages_needed against free_count() and fits().
  // Copy-on-write events are appended to `cows`.
  void append(const int* slots, int n, int64_t n_tok, std::vector<CowEvent>* cows);
  void release(int slot);

  const SeqSlot& slot(int i) const { return slots_[i]; }
  SeqSlot& slot_mut(int i) { return slots_[i]; }
  const std::vector<int32_t>& refcounts() const { return ref_; }
  // Free list in FIFO order.
  void free_list(std::vector<int32_t>* out) const;

 private:
  int32_t pop_free();
  void push_free(int32_t b);

  int64_t n_blocks_;
  int page_;
  int max_pages_;
  std::vector<int32_t> ref_;
  std::vector<int32_t> ring_;  // FIFO ring buffer of capacity n_blocks
  int64_t head_ = 0, free_count_ = 0;
  std::vector<SeqSlot> slots_;
  int32_t next_family_ = 0;
};

}  // namespace st
