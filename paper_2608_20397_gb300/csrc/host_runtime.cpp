// Host runtime of the splice path: the depth-adaptive policy (Eq. 2,
// Sec. III-C), the fail-closed splice gate (Sec. III-B), the page pool
// (Sec. V-C analogue) and the splice planner (Sec. III-B / Sec. V-A).
#include <algorithm>
#include <cstdint>
#include <cstring>
#include <mutex>
#include <new>
#include <numeric>
#include <vector>

#include "nexus.h"

namespace {

constexpr int kPage = 16;

bool policy_ok(const nexus_policy* p) {
  if (!p) return false;
  if (p->splice_threshold < 1 || p->splice_threshold > (1 << 24)) return false;
  if (p->full_mult < 2 || p->full_mult > (1 << 16)) return false;
  if (p->r_base_pct < 0 || p->r_base_pct > 100) return false;
  return true;
}

int64_t gcd64(int64_t a, int64_t b) {
  while (b) { const int64_t t = a % b; a = b; b = t; }
  return a < 0 ? -a : a;
}

// R(n_past) = num / den percent (Eq. 2), clamped to 100.
void recompute_fraction(int32_t n_past, const nexus_policy* p, int64_t* num, int64_t* den) {
  const int64_t M = p->splice_threshold, K = p->full_mult, Rb = p->r_base_pct;
  if (n_past <= M) { *num = Rb; *den = 1; return; }
  const int64_t D = M * (K - 1);
  const int64_t N = Rb * D + (static_cast<int64_t>(n_past) - M) * (100 - Rb);
  if (N >= 100 * D) { *num = 100; *den = 1; return; }
  const int64_t g = gcd64(N, D);
  *num = N / g;
  *den = D / g;
}

// ceil(S * num / (100 * den)), at most S.
int32_t ceil_fraction(int32_t S, int64_t num, int64_t den) {
  const unsigned __int128 a = static_cast<unsigned __int128>(S) * static_cast<unsigned __int128>(num);
  const unsigned __int128 b = static_cast<unsigned __int128>(100) * static_cast<unsigned __int128>(den);
  const unsigned __int128 q = (a + b - 1) / b;
  return q > static_cast<unsigned __int128>(S) ? S : static_cast<int32_t>(q);
}

}  // namespace

// ------------------------------------------------------------------ pool
// Page ids are handed out in the order of `order`; a page whose last reference
// is dropped goes to the back. Pages may be shared by several page tables (a
// warm prefix, Sec. V-D), so each carries a reference count. All storage is
// reserved at creation: alloc, retain and free never allocate. The mutex sits
// on its own 128-byte line, away from the data the allocating threads read, so
// contended locking does not false-share.
struct alignas(128) nexus_page_pool {
  alignas(128) std::mutex mu;
  alignas(128) int64_t n_pages = 0;
  std::vector<int32_t> ring;    // free pages in hand-out order: ring[head .. head + n_free)
  int64_t head = 0;
  int64_t n_free = 0;
  std::vector<uint32_t> refs;   // references per page; 0 = free
  std::vector<uint32_t> mark;   // duplicate check of one request (epoch stamps)
  uint32_t epoch = 0;
};
static_assert(alignof(nexus_page_pool) % 128 == 0, "page pool must be cache-line aligned");

namespace {

void ring_push(nexus_page_pool* p, int32_t pg) {
  p->ring[static_cast<size_t>((p->head + p->n_free) % p->n_pages)] = pg;
  ++p->n_free;
}

int32_t ring_pop(nexus_page_pool* p) {
  const int32_t pg = p->ring[static_cast<size_t>(p->head)];
  p->head = (p->head + 1) % p->n_pages;
  --p->n_free;
  return pg;
}

// Stamps pages[0, n) for one request; false if a page repeats. Caller holds mu.
bool distinct(nexus_page_pool* p, int32_t n, const int32_t* pages) {
  if (++p->epoch == 0) {
    std::fill(p->mark.begin(), p->mark.end(), 0u);
    p->epoch = 1;
  }
  for (int32_t i = 0; i < n; ++i) {
    if (p->mark[pages[i]] == p->epoch) return false;
    p->mark[pages[i]] = p->epoch;
  }
  return true;
}

}  // namespace

extern "C" {

const char* nexus_status_string(nexus_status s) {
  switch (s) {
    case NEXUS_OK: return "ok";
    case NEXUS_EINVAL: return "invalid argument";
    case NEXUS_ERANGE: return "position, page, row or layer out of range";
    case NEXUS_EROPE_MISMATCH: return "block RoPE parameters differ from the cache's";
    case NEXUS_ELAYOUT: return "buffer layout or alignment check failed";
    case NEXUS_ENOMEM: return "page pool, workspace or capacity too small";
    case NEXUS_EDECLINED: return "splice past the threshold without enough redecode";
    case NEXUS_ECUDA: return "CUDA call failed";
    case NEXUS_ETIMEOUT: return "a bounded device wait gave up";
    case NEXUS_EOVERLAP: return "destination rows overlap";
  }
  return "unknown status";
}

int32_t nexus_version(void) { return NEXUS_VERSION; }

nexus_status nexus_recompute_pct(int32_t n_past, const nexus_policy* policy, int64_t* num,
                                 int64_t* den) {
  if (!policy_ok(policy) || !num || !den) return NEXUS_EINVAL;
  recompute_fraction(n_past, policy, num, den);
  return NEXUS_OK;
}

int32_t nexus_redecode_len(int32_t S, int32_t n_past, const nexus_policy* policy) {
  if (!policy_ok(policy) || S < 0) return -1;
  int64_t num, den;
  recompute_fraction(n_past, policy, &num, &den);
  return ceil_fraction(S, num, den);
}

int32_t nexus_suffix_len(int32_t S, int32_t pct) {
  if (S < 0 || pct < 0 || pct > 100) return -1;
  return ceil_fraction(S, pct, 1);
}

nexus_status nexus_check_splice(int32_t n_past, int32_t S, int32_t n_redecode,
                                const nexus_policy* policy) {
  if (!policy_ok(policy) || S < 0 || n_redecode < 0 || n_past < 0) return NEXUS_EINVAL;
  if (n_past <= policy->splice_threshold) return NEXUS_OK;
  return n_redecode >= nexus_redecode_len(S, n_past, policy) ? NEXUS_OK : NEXUS_EDECLINED;
}

nexus_status nexus_page_pool_create(int64_t n_pages, const int32_t* order, nexus_page_pool** out) {
  if (!out || n_pages <= 0 || n_pages > 0x7FFFFFFF) return NEXUS_EINVAL;
  *out = nullptr;
  nexus_page_pool* pool = new (std::nothrow) nexus_page_pool();
  if (!pool) return NEXUS_ENOMEM;
  pool->n_pages = n_pages;
  pool->refs.assign(static_cast<size_t>(n_pages), 0u);
  pool->mark.assign(static_cast<size_t>(n_pages), 0u);
  pool->ring.assign(static_cast<size_t>(n_pages), 0);
  if (order) {
    for (int64_t i = 0; i < n_pages; ++i) {
      const int32_t pg = order[i];
      if (pg < 0 || pg >= n_pages || pool->mark[pg]) { delete pool; return NEXUS_EINVAL; }
      pool->mark[pg] = 1;
      pool->ring[i] = pg;
    }
    std::fill(pool->mark.begin(), pool->mark.end(), 0u);
  } else {
    for (int64_t i = 0; i < n_pages; ++i) pool->ring[i] = static_cast<int32_t>(i);
  }
  pool->n_free = n_pages;
  *out = pool;
  return NEXUS_OK;
}

void nexus_page_pool_destroy(nexus_page_pool* pool) { delete pool; }

nexus_status nexus_page_pool_alloc(nexus_page_pool* pool, int32_t n, int32_t* pages) {
  if (!pool || n < 0 || (n > 0 && !pages)) return NEXUS_EINVAL;
  std::lock_guard<std::mutex> lock(pool->mu);
  if (pool->n_free < n) return NEXUS_ENOMEM;
  for (int32_t i = 0; i < n; ++i) {
    const int32_t pg = ring_pop(pool);
    pool->refs[pg] = 1;
    pages[i] = pg;
  }
  return NEXUS_OK;
}

nexus_status nexus_page_pool_free(nexus_page_pool* pool, int32_t n, const int32_t* pages) {
  if (!pool || n < 0 || (n > 0 && !pages)) return NEXUS_EINVAL;
  std::lock_guard<std::mutex> lock(pool->mu);
  for (int32_t i = 0; i < n; ++i) {
    if (pages[i] < 0 || pages[i] >= pool->n_pages) return NEXUS_ERANGE;
    if (pool->refs[pages[i]] == 0) return NEXUS_EINVAL;
  }
  if (!distinct(pool, n, pages)) return NEXUS_EINVAL;   // a page listed twice
  for (int32_t i = 0; i < n; ++i)
    if (--pool->refs[pages[i]] == 0) ring_push(pool, pages[i]);
  return NEXUS_OK;
}

nexus_status nexus_page_pool_retain(nexus_page_pool* pool, int32_t n, const int32_t* pages) {
  if (!pool || n < 0 || (n > 0 && !pages)) return NEXUS_EINVAL;
  std::lock_guard<std::mutex> lock(pool->mu);
  for (int32_t i = 0; i < n; ++i) {
    if (pages[i] < 0 || pages[i] >= pool->n_pages) return NEXUS_ERANGE;
    if (pool->refs[pages[i]] == 0 || pool->refs[pages[i]] == UINT32_MAX) return NEXUS_EINVAL;
  }
  if (!distinct(pool, n, pages)) return NEXUS_EINVAL;
  for (int32_t i = 0; i < n; ++i) ++pool->refs[pages[i]];
  return NEXUS_OK;
}

int64_t nexus_page_pool_refs(const nexus_page_pool* pool, int32_t page) {
  if (!pool || page < 0 || page >= pool->n_pages) return -1;
  std::lock_guard<std::mutex> lock(const_cast<nexus_page_pool*>(pool)->mu);
  return pool->refs[page];
}

int64_t nexus_page_pool_available(const nexus_page_pool* pool) {
  if (!pool) return -1;
  std::lock_guard<std::mutex> lock(const_cast<nexus_page_pool*>(pool)->mu);
  return pool->n_free;
}

nexus_status nexus_page_pool_make_private(nexus_page_pool* pool, int32_t* h_pt, int32_t first_page,
                                          int32_t n, int32_t* src_pages, int32_t* dst_pages,
                                          int32_t capacity, int32_t* n_copies) {
  if (!pool || !h_pt || first_page < 0 || n < 0 || !n_copies || capacity < 0) return NEXUS_EINVAL;
  *n_copies = 0;
  std::lock_guard<std::mutex> lock(pool->mu);
  int32_t shared = 0;
  for (int32_t i = first_page; i < first_page + n; ++i) {
    const int32_t pg = h_pt[i];
    if (pg < 0 || pg >= pool->n_pages) return NEXUS_ERANGE;
    if (pool->refs[pg] == 0) return NEXUS_EINVAL;
    if (pool->refs[pg] > 1) ++shared;
  }
  if (shared > capacity || (shared > 0 && (!src_pages || !dst_pages))) return NEXUS_ENOMEM;
  if (shared > pool->n_free) return NEXUS_ENOMEM;
  if (!distinct(pool, n, h_pt + first_page)) return NEXUS_EINVAL;   // one page twice in a table
  int32_t k = 0;
  for (int32_t i = first_page; i < first_page + n; ++i) {
    const int32_t pg = h_pt[i];
    if (pool->refs[pg] <= 1) continue;
    const int32_t fresh = ring_pop(pool);
    pool->refs[fresh] = 1;
    --pool->refs[pg];   // still referenced elsewhere: stays in use
    src_pages[k] = pg;
    dst_pages[k] = fresh;
    h_pt[i] = fresh;
    ++k;
  }
  *n_copies = k;
  return NEXUS_OK;
}

nexus_status nexus_plan_splice(nexus_page_pool* pool, const int32_t* h_old_pt, int32_t n_past,
                               int32_t max_pages, const nexus_block* blocks, int32_t n_blocks,
                               const nexus_insert* inserts, int32_t n_inserts, int32_t old_row,
                               int32_t new_row, int32_t* h_new_pt, nexus_splice_segment* segs,
                               int32_t seg_capacity, int32_t* n_segs, int32_t* freed,
                               int32_t* n_freed) {
  if (!pool || !h_new_pt || !n_segs || n_past < 0 || max_pages <= 0 || n_inserts < 0 ||
      seg_capacity < 0 || (n_inserts > 0 && (!inserts || !blocks)) || (n_past > 0 && !h_old_pt) ||
      old_row < 0 || new_row < 0)
    return NEXUS_EINVAL;
  *n_segs = 0;
  if (n_freed) *n_freed = 0;
  int64_t total = n_past;
  for (int32_t k = 0; k < n_inserts; ++k) {
    const nexus_insert& in = inserts[k];
    if (in.block_index < 0 || in.block_index >= n_blocks) return NEXUS_EINVAL;
    if (in.depth < 0 || in.depth > n_past) return NEXUS_ERANGE;
    if (k > 0 && in.depth < inserts[k - 1].depth) return NEXUS_EINVAL;
    if (blocks[in.block_index].n_tokens < 0) return NEXUS_EINVAL;
    total += blocks[in.block_index].n_tokens;
  }
  if (total > static_cast<int64_t>(max_pages) * kPage) return NEXUS_ERANGE;
  const int32_t old_pages = (n_past + kPage - 1) / kPage;
  const int32_t new_pages = static_cast<int32_t>((total + kPage - 1) / kPage);
  for (int32_t i = 0; i < old_pages; ++i)
    if (h_old_pt[i] < 0 || h_old_pt[i] >= pool->n_pages) return NEXUS_ERANGE;

  if (n_inserts == 0) {
    for (int32_t i = 0; i < max_pages; ++i) h_new_pt[i] = i < old_pages ? h_old_pt[i] : -1;
    return NEXUS_OK;
  }
  const int32_t d1 = inserts[0].depth;
  const bool append = d1 == n_past;   // every depth is the cursor
  if (!append && old_row == new_row) return NEXUS_EINVAL;
  // Pages [0, keep) hold no changed row and are shared with the old table.
  const int32_t keep = append ? old_pages : d1 / kPage;

  // Count segments before touching the pool.
  int32_t need = (!append && d1 % kPage != 0) ? 1 : 0;
  {
    int32_t cursor = d1;
    for (int32_t k = 0; k < n_inserts; ++k) {
      if (inserts[k].depth > cursor) ++need;
      if (blocks[inserts[k].block_index].n_tokens > 0) ++need;
      cursor = inserts[k].depth;
    }
    if (n_past > cursor) ++need;
  }
  if (need > seg_capacity || (need > 0 && !segs)) return NEXUS_ENOMEM;

  const int32_t fresh = std::max(0, new_pages - keep);
  std::vector<int32_t> got(static_cast<size_t>(fresh));
  if (fresh > 0) {
    const nexus_status st = nexus_page_pool_alloc(pool, fresh, got.data());
    if (st != NEXUS_OK) return st;
  }
  for (int32_t i = 0; i < max_pages; ++i) {
    if (i < keep) h_new_pt[i] = h_old_pt[i];
    else if (i < new_pages) h_new_pt[i] = got[i - keep];
    else h_new_pt[i] = -1;
  }

  int32_t ns = 0;
  auto add = [&](int32_t kind, int32_t idx, int32_t src_start, int32_t dst_start, int32_t n,
                 int32_t delta) {
    nexus_splice_segment& s = segs[ns++];
    s.src_kind = kind;
    s.src_index = idx;
    s.src_start = src_start;
    s.dst_row = new_row;
    s.dst_start = dst_start;
    s.n_tokens = n;
    s.delta = delta;
    s.flags = 0;
  };
  if (!append && d1 % kPage != 0) {
    // copy-on-write of the boundary page: its rows before d1 keep their bits
    const int32_t b0 = (d1 / kPage) * kPage;
    add(NEXUS_SRC_CACHE, old_row, b0, b0, d1 - b0, 0);
  }
  int32_t cursor = d1;
  int32_t shift = 0;
  for (int32_t k = 0; k < n_inserts; ++k) {
    const nexus_insert& in = inserts[k];
    if (in.depth > cursor)   // displaced live rows between two inserts move by `shift`
      add(NEXUS_SRC_CACHE, old_row, cursor, cursor + shift, in.depth - cursor, shift);
    const nexus_block& b = blocks[in.block_index];
    const int32_t pos = in.depth + shift;
    if (b.n_tokens > 0) add(NEXUS_SRC_BLOCK, in.block_index, 0, pos, b.n_tokens, pos - b.base_pos);
    shift += b.n_tokens;
    cursor = in.depth;
  }
  if (n_past > cursor) add(NEXUS_SRC_CACHE, old_row, cursor, cursor + shift, n_past - cursor, shift);
  *n_segs = ns;

  if (!append && freed && n_freed) {
    int32_t nf = 0;
    for (int32_t i = keep; i < old_pages; ++i) freed[nf++] = h_old_pt[i];
    *n_freed = nf;
  }
  return NEXUS_OK;
}

}  // extern "C"
