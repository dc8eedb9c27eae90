// Checks of gf::KvPagePool, the host allocator behind the paged KV cache
// (block tables + reference-counted pages), compiled and run on the CPU by
// tests/test_page_pool.py.  Hand-written scenarios (prefix sharing, forks,
// exhaustion, rollback), then a seeded random walk compared after every step
// against the invariants that define the pool:
//   - refs(p) equals the number of block-table entries that hold p;
//   - the free list holds exactly the pages with no reference, once each;
//   - a rolled-back call leaves the pool exactly as it found it.
#include <cstdio>
#include <random>
#include <vector>

#include "page_pool.h"

static int failures = 0;
#define CHECK(c)                                                           \
  do {                                                                     \
    if (!(c)) {                                                            \
      std::fprintf(stderr, "FAILED %s:%d: %s\n", __FILE__, __LINE__, #c); \
      ++failures;                                                          \
    }                                                                      \
  } while (0)

using gf::KvPagePool;

struct Snapshot {
  std::vector<int32_t> table, refs, free_list;
  bool operator==(const Snapshot& o) const {
    return table == o.table && refs == o.refs && free_list == o.free_list;
  }
};

static Snapshot snap(const KvPagePool& p) {
  Snapshot s;
  s.table = p.table();
  for (int64_t q = 0; q < p.num_pages(); ++q) s.refs.push_back(p.refs((int32_t)q));
  s.free_list = p.free_list();
  return s;
}

static void check_invariants(const KvPagePool& p) {
  const int64_t n = p.num_pages();
  std::vector<int32_t> held(n, 0), listed(n, 0);
  for (int32_t e : p.table()) {
    CHECK(e >= -1 && e < n);
    if (e >= 0) held[e] += 1;
  }
  for (int32_t f : p.free_list()) {
    CHECK(f >= 0 && f < n);
    if (f >= 0 && f < n) listed[f] += 1;
  }
  for (int64_t q = 0; q < n; ++q) {
    CHECK(p.refs((int32_t)q) == held[q]);
    CHECK(listed[q] == (held[q] == 0 ? 1 : 0));
  }
  CHECK(p.free_pages() == (int64_t)p.free_list().size());
}

static void scenario_prefix_sharing() {
  KvPagePool p;
  p.init(4, 8, 20);
  KvPagePool::Undo u;
  // a prompt of 3 pages in slot 0: pages are handed out from page 0 up
  CHECK(p.alloc(0, 0, 3, &u));
  CHECK(p.entry(0, 0) == 0 && p.entry(0, 1) == 1 && p.entry(0, 2) == 2 && p.entry(0, 3) == -1);
  CHECK(p.free_pages() == 17);
  // two candidates continue its first two (full) pages and add pages of their own
  u.clear();
  p.share(1, 0, 2, &u);
  p.share(2, 0, 2, &u);
  CHECK(p.alloc(1, 2, 2, &u) && p.alloc(2, 2, 1, &u));
  CHECK(p.entry(1, 0) == 0 && p.entry(2, 1) == 1 && p.refs(0) == 3 && p.refs(1) == 3);
  CHECK(p.entry(1, 2) != p.entry(0, 2) && p.entry(2, 2) != p.entry(1, 2));
  check_invariants(p);
  // releasing the prefix owner keeps the shared pages alive; only its own page returns
  p.clear(0);
  CHECK(p.refs(0) == 2 && p.refs(2) == 0 && p.free_pages() == 20 - 2 - 3);
  check_invariants(p);
  p.clear(1);
  p.clear(2);
  CHECK(p.free_pages() == 20);
  check_invariants(p);
}

static void scenario_fork_with_partial_page() {
  // a sampled row forked from a prompt of 150 tokens: shares pages 0-1, copies page 2 into a
  // page of its own, and takes pages for 20 decode tokens (170 tokens: 3 pages)
  KvPagePool p;
  p.init(3, 4, 10);
  KvPagePool::Undo u;
  CHECK(p.alloc(0, 0, 3, &u));
  u.clear();
  const int len = 150, full = len / 64;
  p.share(1, 0, full, &u);
  CHECK(p.alloc(1, full, (len + 20 + 63) / 64 - full, &u));
  CHECK(p.entry(1, 0) == p.entry(0, 0) && p.entry(1, 1) == p.entry(0, 1));
  CHECK(p.entry(1, 2) >= 0 && p.entry(1, 2) != p.entry(0, 2));
  CHECK(u.size() == 3);
  check_invariants(p);
  // the whole fork rolls back
  p.rollback(u);
  CHECK(p.entry(1, 0) == -1 && p.entry(1, 2) == -1 && p.refs(p.entry(0, 0)) == 1 && p.free_pages() == 7);
  check_invariants(p);
}

static void scenario_exhaustion() {
  KvPagePool p;
  p.init(2, 8, 5);
  const Snapshot before = snap(p);
  KvPagePool::Undo u;
  CHECK(!p.alloc(0, 0, 8, &u));  // 8 pages asked, 5 exist
  CHECK(u.size() == 5 && p.free_pages() == 0);
  check_invariants(p);
  p.rollback(u);
  CHECK(snap(p) == before);
  // entries that already hold a page are kept, not replaced
  u.clear();
  CHECK(p.alloc(0, 0, 2, &u));
  u.clear();
  CHECK(p.alloc(0, 0, 4, &u));
  CHECK(u.size() == 2 && p.free_pages() == 1);
  check_invariants(p);
  // sharing skips entries the source does not hold
  u.clear();
  p.share(1, 0, 8, &u);
  CHECK(u.size() == 4 && p.entry(1, 4) == -1);
  check_invariants(p);
}

static void random_walk(uint32_t seed) {
  const int slots = 6, per = 16;
  const int64_t pages = 40;
  KvPagePool p;
  p.init(slots, per, pages);
  std::mt19937 rng(seed);
  auto pick = [&](int n) { return (int)(rng() % (uint32_t)n); };
  for (int step = 0; step < 4000; ++step) {
    const Snapshot before = snap(p);
    KvPagePool::Undo u;
    const int op = pick(10);
    const int s = pick(slots);
    bool undo_it = pick(4) == 0;
    if (op < 5) {
      const int first = pick(per), count = pick(per - first + 1);
      if (!p.alloc(s, first, count, &u)) undo_it = true;  // a failed call is always rolled back
    } else if (op < 8) {
      const int from = pick(slots);
      if (from == s) continue;
      p.clear(s);
      const Snapshot cleared = snap(p);
      p.share(s, from, pick(per + 1), &u);
      check_invariants(p);
      if (undo_it) {
        p.rollback(u);
        CHECK(snap(p) == cleared);
      }
      check_invariants(p);
      continue;
    } else {
      p.clear(s);
      for (int j = 0; j < per; ++j) CHECK(p.entry(s, j) == -1);
      check_invariants(p);
      continue;
    }
    check_invariants(p);
    if (undo_it) {
      p.rollback(u);
      CHECK(snap(p) == before);
    }
    check_invariants(p);
  }
  for (int s = 0; s < slots; ++s) p.clear(s);
  CHECK(p.free_pages() == pages);
  check_invariants(p);
}

int main() {
  scenario_prefix_sharing();
  scenario_fork_with_partial_page();
  scenario_exhaustion();
  for (uint32_t seed = 1; seed <= 5; ++seed) random_walk(seed);
  if (failures) {
    std::fprintf(stderr, "%d check(s) failed\n", failures);
    return 1;
  }
  std::printf("ok\n");
  return 0;
}
