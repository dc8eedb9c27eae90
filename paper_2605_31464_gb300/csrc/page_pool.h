// Host bookkeeping of the paged KV cache: one block table per sequence slot
// (entry j is the pool page that holds the slot's tokens [64j, 64j + 64), or
// -1) and a reference-counted pool of pages.  A page of a shared prefix, or of
// a sampled row forked from its prompt, is pointed at by several block tables;
// it returns to the free list when the last entry pointing at it is dropped.
// Plain C++ (no CUDA), so that its invariants can be tested without a GPU.
#pragma once

#include <cstdint>
#include <utility>
#include <vector>

namespace gf {

class KvPagePool {
 public:
  // (slot, entry) pairs that alloc() and share() set, in order; rollback() drops them.
  using Undo = std::vector<std::pair<int, int>>;

  // `slots` block tables of `pages_per_slot` entries, all empty; pages 0 .. pages-1 free
  // (handed out from page 0 up).
  void init(int slots, int pages_per_slot, int64_t pages) {
    per_slot_ = pages_per_slot;
    table_.assign((size_t)slots * pages_per_slot, -1);
    ref_.assign((size_t)pages, 0);
    free_.clear();
    free_.reserve((size_t)pages);
    for (int64_t p = pages - 1; p >= 0; --p) free_.push_back((int32_t)p);
  }

  int32_t entry(int slot, int j) const { return table_[(size_t)slot * per_slot_ + j]; }
  // All block tables, [slot][pages_per_slot] (what the kernels read).
  const std::vector<int32_t>& table() const { return table_; }
  int pages_per_slot() const { return per_slot_; }
  int64_t num_pages() const { return (int64_t)ref_.size(); }
  int64_t free_pages() const { return (int64_t)free_.size(); }
  // Block-table entries that point at `page`.
  int32_t refs(int32_t page) const { return ref_[page]; }
  // The free pages, the next one handed out last.
  const std::vector<int32_t>& free_list() const { return free_; }

  // Entries [first, first + count) of `slot` that hold no page get a fresh page (one reference).
  // Returns false when the pool runs dry; the entries set before that are in *undo either way.
  bool alloc(int slot, int first, int count, Undo* undo) {
    for (int j = first; j < first + count; ++j) {
      int32_t& e = at(slot, j);
      if (e >= 0) continue;
      if (free_.empty()) return false;
      e = free_.back();
      free_.pop_back();
      ref_[e] = 1;
      undo->push_back({slot, j});
    }
    return true;
  }

  // Entries [0, count) of `slot` (empty) point at the pages of the same entries of `from`
  // (copy-free sharing of a cached prefix); empty entries of `from` are skipped.
  void share(int slot, int from, int count, Undo* undo) {
    for (int j = 0; j < count; ++j) {
      const int32_t p = at(from, j);
      if (p < 0) continue;
      drop(at(slot, j));
      at(slot, j) = p;
      ref_[p] += 1;
      undo->push_back({slot, j});
    }
  }

  // Drop the entries in `undo`, last first: a failed or abandoned call leaves no trace.
  void rollback(const Undo& undo) {
    for (auto it = undo.rbegin(); it != undo.rend(); ++it) drop(at(it->first, it->second));
  }

  // Drop every entry of `slot`.
  void clear(int slot) {
    for (int j = 0; j < per_slot_; ++j) drop(at(slot, j));
  }

 private:
  int32_t& at(int slot, int j) { return table_[(size_t)slot * per_slot_ + j]; }
  void drop(int32_t& e) {
    if (e >= 0 && --ref_[e] == 0) free_.push_back(e);
    e = -1;
  }

  int per_slot_ = 0;
  std::vector<int32_t> table_, ref_, free_;
};

}  // namespace gf
