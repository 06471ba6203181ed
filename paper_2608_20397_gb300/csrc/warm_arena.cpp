// L0 exact-token radix arena (Sec. V-D): a fixed set of sequence slots whose
// warm prefixes new requests reuse by exact-token longest-common-prefix match.
//
// A slot holds a sequence's tokens and references to the cache pages of its
// rows; it never copies them. A new sequence forked from a slot shares the
// pages that hold only prefix rows and gets a private copy of the one page it
// will keep writing (copy-on-write), so reusing a warm prefix of m tokens costs
// at most one page copy on the GPU whatever m is.
//
// Matching keeps, for every pair of slots, the length of their common prefix.
// While the query is compared slot after slot, the slot with the longest match
// so far (length r) decides most others without touching their tokens: a slot
// sharing fewer than r tokens with it shares exactly that many with the query,
// one sharing more than r shares exactly r; only a slot sharing exactly r is
// compared, from token r on. Each token comparison past the first mismatch
// extends the best match, so one query costs O(n + slots) however many slots
// hold the same long prompt. Every buffer is reserved at creation.
#include <algorithm>
#include <cstdint>
#include <new>
#include <vector>

#include "nexus.h"

namespace {
constexpr int kPage = 16;
constexpr int kMaxSlots = 32;
}  // namespace

struct nexus_warm_arena {
  int32_t n_slots = 0;
  int32_t max_tokens = 0;
  int32_t max_pages = 0;
  std::vector<int32_t> tokens;     // [n_slots][max_tokens]
  std::vector<int32_t> len;        // tokens held; 0 = empty
  std::vector<int32_t> pages;      // [n_slots][max_pages]
  std::vector<int32_t> pair_lcp;   // [n_slots][n_slots]
  std::vector<uint64_t> last_use;
  std::vector<int32_t> scratch;    // [n_slots] prefix lengths of one query
  uint64_t clock = 0;

  const int32_t* toks(int s) const { return tokens.data() + static_cast<size_t>(s) * max_tokens; }
  int32_t* toks(int s) { return tokens.data() + static_cast<size_t>(s) * max_tokens; }
  int32_t* pgs(int s) { return pages.data() + static_cast<size_t>(s) * max_pages; }
  const int32_t* pgs(int s) const { return pages.data() + static_cast<size_t>(s) * max_pages; }
  int32_t& lcp(int a, int b) { return pair_lcp[static_cast<size_t>(a) * n_slots + b]; }
  int32_t lcp(int a, int b) const { return pair_lcp[static_cast<size_t>(a) * n_slots + b]; }
};

namespace {

// out[s] = common prefix length of q[0, n) and slot s (0 for an empty slot).
void prefixes(const nexus_warm_arena& a, const int32_t* q, int32_t n, int32_t* out) {
  int ref = -1;
  int32_t ref_len = 0;
  for (int s = 0; s < a.n_slots; ++s) {
    if (a.len[s] == 0) { out[s] = 0; continue; }
    const int32_t lim = std::min(a.len[s], n);
    int32_t k = 0;
    if (ref >= 0) {
      const int32_t l = a.lcp(ref, s);
      if (l < ref_len) { out[s] = l; continue; }
      if (l > ref_len) { out[s] = ref_len; continue; }
      k = ref_len;
    }
    const int32_t* t = a.toks(s);
    while (k < lim && t[k] == q[k]) ++k;
    out[s] = k;
    if (ref < 0 || k > ref_len) { ref = s; ref_len = k; }
  }
}

int best_slot(const nexus_warm_arena& a, const int32_t* pre, int32_t* best_len) {
  int best = -1;
  int32_t bl = 0;
  for (int s = 0; s < a.n_slots; ++s) {
    if (pre[s] == 0) continue;
    if (pre[s] > bl || (pre[s] == bl && a.last_use[s] > a.last_use[best])) { best = s; bl = pre[s]; }
  }
  *best_len = bl;
  return best;
}

int32_t pages_of(int32_t n) { return (n + kPage - 1) / kPage; }

}  // namespace

extern "C" {

nexus_status nexus_warm_arena_create(int32_t n_slots, int32_t max_tokens, nexus_warm_arena** out) {
  if (!out) return NEXUS_EINVAL;
  *out = nullptr;
  if (n_slots < 1 || n_slots > kMaxSlots || max_tokens < 1 || max_tokens > (1 << 24))
    return NEXUS_EINVAL;
  nexus_warm_arena* a = new (std::nothrow) nexus_warm_arena();
  if (!a) return NEXUS_ENOMEM;
  try {
    a->n_slots = n_slots;
    a->max_tokens = max_tokens;
    a->max_pages = pages_of(max_tokens);
    a->tokens.assign(static_cast<size_t>(n_slots) * max_tokens, 0);
    a->len.assign(n_slots, 0);
    a->pages.assign(static_cast<size_t>(n_slots) * a->max_pages, -1);
    a->pair_lcp.assign(static_cast<size_t>(n_slots) * n_slots, 0);
    a->last_use.assign(n_slots, 0);
    a->scratch.assign(n_slots, 0);
  } catch (...) {
    delete a;
    return NEXUS_ENOMEM;
  }
  *out = a;
  return NEXUS_OK;
}

void nexus_warm_arena_destroy(nexus_warm_arena* a, nexus_page_pool* pool) {
  if (!a) return;
  if (pool)
    for (int s = 0; s < a->n_slots; ++s)
      if (a->len[s] > 0) nexus_page_pool_free(pool, pages_of(a->len[s]), a->pgs(s));
  delete a;
}

nexus_status nexus_warm_arena_match(nexus_warm_arena* a, const int32_t* tokens, int32_t n,
                                    int32_t* slot, int32_t* prefix) {
  if (!a || !slot || !prefix || n < 0 || (n > 0 && !tokens)) return NEXUS_EINVAL;
  int32_t* pre = a->scratch.data();   // the only buffer a match writes
  prefixes(*a, tokens, n, pre);
  *slot = best_slot(*a, pre, prefix);
  return NEXUS_OK;
}

nexus_status nexus_warm_arena_fork(nexus_warm_arena* a, nexus_page_pool* pool, int32_t slot,
                                   int32_t m, int32_t* h_new_pt, int32_t max_pages,
                                   int32_t* copy_src, int32_t* copy_dst, int32_t* n_copies) {
  if (!a || !pool || !h_new_pt || !n_copies || max_pages < 0) return NEXUS_EINVAL;
  *n_copies = 0;
  if (slot < 0 || slot >= a->n_slots || a->len[slot] == 0) return NEXUS_ERANGE;
  if (m < 0 || m > a->len[slot]) return NEXUS_ERANGE;
  const int32_t full = m / kPage;
  const bool partial = m % kPage != 0;
  if (full + (partial ? 1 : 0) > max_pages) return NEXUS_ERANGE;
  if (partial && (!copy_src || !copy_dst)) return NEXUS_EINVAL;
  int32_t fresh = -1;
  if (partial) {
    const nexus_status st = nexus_page_pool_alloc(pool, 1, &fresh);
    if (st != NEXUS_OK) return st;
  }
  if (full > 0) {
    const nexus_status st = nexus_page_pool_retain(pool, full, a->pgs(slot));
    if (st != NEXUS_OK) {
      if (partial) nexus_page_pool_free(pool, 1, &fresh);
      return st;
    }
  }
  std::copy(a->pgs(slot), a->pgs(slot) + full, h_new_pt);
  if (partial) {
    h_new_pt[full] = fresh;
    copy_src[0] = a->pgs(slot)[full];
    copy_dst[0] = fresh;
    *n_copies = 1;
  }
  a->last_use[slot] = ++a->clock;
  return NEXUS_OK;
}

nexus_status nexus_warm_arena_store(nexus_warm_arena* a, nexus_page_pool* pool,
                                    const int32_t* tokens, int32_t n, const int32_t* h_pt,
                                    int32_t* slot_out) {
  if (!a || !pool || !tokens || !h_pt || n < 1) return NEXUS_EINVAL;
  const int32_t nk = std::min(n, a->max_tokens);
  int32_t* pre = a->scratch.data();
  prefixes(*a, tokens, nk, pre);
  // Already held: a slot whose sequence starts with these tokens.
  for (int s = 0; s < a->n_slots; ++s) {
    if (a->len[s] >= nk && pre[s] == nk) {
      a->last_use[s] = ++a->clock;
      if (slot_out) *slot_out = s;
      return NEXUS_OK;
    }
  }
  int target = -1;
  for (int s = 0; s < a->n_slots; ++s)   // a slot holding a prefix of them: extended
    if (a->len[s] > 0 && pre[s] == a->len[s] && (target < 0 || a->len[s] > a->len[target]))
      target = s;
  if (target < 0)
    for (int s = 0; s < a->n_slots && target < 0; ++s)
      if (a->len[s] == 0) target = s;
  if (target < 0) {
    target = 0;
    for (int s = 1; s < a->n_slots; ++s)
      if (a->last_use[s] < a->last_use[target]) target = s;
  }
  const int32_t np = pages_of(nk);
  nexus_status st = nexus_page_pool_retain(pool, np, h_pt);   // before dropping the old ones
  if (st != NEXUS_OK) return st;
  if (a->len[target] > 0) {
    st = nexus_page_pool_free(pool, pages_of(a->len[target]), a->pgs(target));
    if (st != NEXUS_OK) {
      nexus_page_pool_free(pool, np, h_pt);
      return st;
    }
  }
  std::copy(tokens, tokens + nk, a->toks(target));
  std::copy(h_pt, h_pt + np, a->pgs(target));
  std::fill(a->pgs(target) + np, a->pgs(target) + a->max_pages, -1);
  a->len[target] = nk;
  for (int s = 0; s < a->n_slots; ++s) {
    const int32_t l = s == target ? nk : (a->len[s] > 0 ? pre[s] : 0);
    a->lcp(target, s) = l;
    a->lcp(s, target) = l;
  }
  a->last_use[target] = ++a->clock;
  if (slot_out) *slot_out = target;
  return NEXUS_OK;
}

nexus_status nexus_warm_arena_slot(const nexus_warm_arena* a, int32_t slot, int32_t* n_tokens,
                                   int32_t* h_pages, int32_t capacity) {
  if (!a || !n_tokens) return NEXUS_EINVAL;
  if (slot < 0 || slot >= a->n_slots) return NEXUS_ERANGE;
  *n_tokens = a->len[slot];
  if (h_pages) {
    const int32_t np = pages_of(a->len[slot]);
    if (capacity < np) return NEXUS_ENOMEM;
    std::copy(a->pgs(slot), a->pgs(slot) + np, h_pages);
  }
  return NEXUS_OK;
}

}  // extern "C"
