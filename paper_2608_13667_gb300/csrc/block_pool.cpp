#include "block_pool.h"

#include <utility>

namespace st {

namespace {

// splitmix64 (Steele, Lea & Flood, OOPSLA 2014): add the golden-ratio
// increment, then two xor-shift-multiply rounds and a final xor-shift.
struct SplitMix64 {
  uint64_t state;
  uint64_t next() {
    state += 0x9E3779B97F4A7C15ull;
    uint64_t z = state;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
  }
};

}  // namespace

BlockPool::BlockPool(int64_t n_blocks, uint64_t seed, int page_size, int max_seqs, int max_pages)
    : n_blocks_(n_blocks), page_(page_size), max_pages_(max_pages), ref_(n_blocks, 0),
      ring_(n_blocks), slots_(max_seqs) {
  for (int64_t i = 0; i < n_blocks; ++i) ring_[i] = (int32_t)i;
  SplitMix64 g{seed};
  for (int64_t i = n_blocks - 1; i >= 1; --i) {
    const int64_t j = (int64_t)(g.next() % (uint64_t)(i + 1));
    std::swap(ring_[i], ring_[j]);
  }
  head_ = 0;
  free_count_ = n_blocks;
  for (auto& s : slots_) s.gen = 1;
}

int32_t BlockPool::pop_free() {
  const int32_t b = ring_[head_];
  head_ = (head_ + 1) % n_blocks_;
  --free_count_;
  ref_[b] = 1;
  return b;
}

void BlockPool::push_free(int32_t b) {
  ring_[(head_ + free_count_) % n_blocks_] = b;
  ++free_count_;
}

void BlockPool::free_list(std::vector<int32_t>* out) const {
  out->resize(free_count_);
  for (int64_t i = 0; i < free_count_; ++i) (*out)[i] = ring_[(head_ + i) % n_blocks_];
}

int BlockPool::create_seq() {
  for (int i = 0; i < (int)slots_.size(); ++i) {
    SeqSlot& s = slots_[i];
    if (!s.live) {
      s.live = true;
      s.family = next_family_++;
      s.len = 0;
      s.table.clear();
      s.dirty_lo = s.dirty_hi = 0;
      return i;
    }
  }
  return -1;
}

bool BlockPool::fork(int parent, int n_aux, int* out) {
  return fork_at(parent, slots_[parent].len, n_aux, out);
}

bool BlockPool::fork_at(int parent, int64_t length, int n_aux, int* out) {
  int found = 0;
  for (int i = 0; i < (int)slots_.size() && found < n_aux; ++i)
    if (!slots_[i].live) out[found++] = i;
  if (found < n_aux) return false;
  const SeqSlot& src = slots_[parent];
  const size_t n_pages = (size_t)((length + page_ - 1) / page_);
  for (int a = 0; a < n_aux; ++a) {
    SeqSlot& s = slots_[out[a]];
    s.live = true;
    s.family = src.family;
    s.len = length;
    s.table.assign(src.table.begin(), src.table.begin() + n_pages);
    s.dirty_lo = s.dirty_hi = 0;
    s.mark_dirty(0, (int32_t)s.table.size());
    for (int32_t b : s.table) ++ref_[b];
  }
  return true;
}

int64_t BlockPool::pages_needed(int slot, int64_t n_tok) const {
  if (n_tok <= 0) return 0;
  const SeqSlot& s = slots_[slot];
  const int64_t p = page_;
  int64_t need = (s.len + n_tok + p - 1) / p - (s.len + p - 1) / p;
  if (s.len % p != 0 && ref_[s.table.back()] > 1) need += 1;  // copy-on-write
  return need;
}

bool BlockPool::fits(int slot, int64_t n_tok) const {
  const SeqSlot& s = slots_[slot];
  return (s.len + n_tok + page_ - 1) / page_ <= max_pages_;
}

void BlockPool::append(const int* slots, int n, int64_t n_tok, std::vector<CowEvent>* cows) {
  if (n_tok <= 0) return;
  for (int i = 0; i < n; ++i) {
    SeqSlot& s = slots_[slots[i]];
    const int64_t off = s.len % page_;
    if (off != 0 && ref_[s.table.back()] > 1) {
      const int32_t old = s.table.back();
      const int32_t fresh = pop_free();
      --ref_[old];
      s.table.back() = fresh;
      cows->push_back(CowEvent{old, fresh, (int32_t)off});
      s.mark_dirty((int32_t)s.table.size() - 1, (int32_t)s.table.size());
    }
    const int64_t new_len = s.len + n_tok;
    const int64_t have = (int64_t)s.table.size();
    const int64_t want = (new_len + page_ - 1) / page_;
    for (int64_t pg = have; pg < want; ++pg) s.table.push_back(pop_free());
    s.len = new_len;
    s.mark_dirty((int32_t)have, (int32_t)s.table.size());  // only entries that changed
  }
}

void BlockPool::release(int slot) {
  SeqSlot& s = slots_[slot];
  for (int32_t b : s.table) {
    if (--ref_[b] == 0) push_free(b);
  }
  s.table.clear();
  s.len = 0;
  s.live = false;
  s.family = -1;
  s.dirty_lo = s.dirty_hi = 0;
  ++s.gen;
  if (s.gen == 0) s.gen = 1;
}

}  // namespace st
