/*
 * nexus.h - C ABI of the GB300 (sm_103a) KV-cache splicing hot path.
 *
 * The operations follow "Nexus: Depth-Adaptive KV-Cache Splicing and
 * Retrieval-Decoupled Tool Routing for Agentic LLMs on Unified Memory":
 *
 *   nexus_splice_kv          write compiled schema K/V rows into a live paged
 *                            cache at the runtime cursor, reanchoring K by
 *                            delta = position - base_pos (Sec. III-B, Sec. V-A),
 *                            row-major or token-innermost V (Sec. V-B)
 *   nexus_rope_rerotate      rotate cached keys by a position offset
 *                            (Sec. III-B, Eq. 1)
 *   nexus_copy_pages         bit-exact page copies (the in-arena KV copy of
 *                            Sec. V-D)
 *   nexus_suffix_attention   causal GQA attention of the last R positions over
 *                            the spliced cache: the redecoded suffix of
 *                            Sec. III-C / Sec. V-A, softmax(QK^T/sqrt(d))V of
 *                            Sec. III-A
 *   nexus_reprefill          the same with R = T: the full re-prefill that
 *                            R(n_past) = 100 % amounts to (Sec. III-C)
 *   nexus_suffix_qkv         fresh Q, K, V of the re-decoded suffix tokens:
 *                            QKV projection, RoPE at the new positions, K/V
 *                            written into the paged cache (Sec. V-A, Sec. III-B)
 *   nexus_recompute_pct, nexus_redecode_len, nexus_check_splice
 *                            the depth-adaptive policy of Eq. 2 and the
 *                            splice threshold P (Sec. III-B, Sec. III-C)
 *   nexus_page_pool_*, nexus_plan_splice
 *                            host page allocator (reference-counted pages,
 *                            copy-on-write) and splice planner
 *   nexus_warm_arena_*       the L0 exact-token radix arena of warm prefixes
 *                            (Sec. V-D)
 *   nexus_slb_*              INT8 tool scan with the top-2 margin gate of the
 *                            semantic lookaside buffer (Sec. IV-A)
 *   nexus_host_alloc, nexus_host_free
 *                            page-locked host staging memory for the copies
 *                            around the path
 *
 * Conventions
 *   - Device buffers are owned by the caller. The library never allocates or
 *     frees device memory and keeps no per-call state; it caches per-device
 *     properties and one error word per device.
 *   - Every call validates its arguments on the host before any launch and
 *     reports problems as a nexus_status; no exception crosses the ABI.
 *   - Device calls are asynchronous on the given stream (a cudaStream_t passed
 *     as void*; NULL is the legacy default stream). A failed launch returns
 *     NEXUS_ECUDA. nexus_device_status() synchronises a stream and reports
 *     whether any bounded device wait gave up.
 *   - Only head_dim = 128, page_size = 16 and bf16 data are accepted.
 *   - Layouts (all bf16, innermost last):
 *       K pool        [n_layers][n_pages][n_kv_heads][page_size][head_dim]
 *       V pool        same, or, when v_transposed,
 *                     [n_layers][n_pages][n_kv_heads][head_dim][page_size]
 *       block K / V   [n_layers][n_tokens][n_kv_heads][head_dim]
 *       page tables   int32 [n_rows][max_pages]; position t of row r lives in
 *                     page table[r][t / 16], slot t % 16
 *       Q, O          [n_layers_call][sum of q_len][n_q_heads][head_dim]
 *       LSE           float [n_layers_call][sum of q_len][n_q_heads]
 *     Pointers passed for device data must be 16-byte aligned.
 */
#ifndef NEXUS_H
#define NEXUS_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define NEXUS_VERSION 1

typedef void* nexus_stream; /* cudaStream_t */

typedef enum nexus_status {
  NEXUS_OK = 0,
  NEXUS_EINVAL = 1,          /* malformed argument (null pointer, bad count, unsupported shape) */
  NEXUS_ERANGE = 2,          /* a position, page id, row or layer lies outside its table */
  NEXUS_EROPE_MISMATCH = 3,  /* block RoPE parameters differ from the cache's; the block is
                                rejected rather than spliced (Sec. V-A) */
  NEXUS_ELAYOUT = 4,         /* shape or alignment check of a buffer failed (Sec. V-B) */
  NEXUS_ENOMEM = 5,          /* page pool exhausted, workspace or output capacity too small */
  NEXUS_EDECLINED = 6,       /* splice past the threshold P without the redecode Eq. 2 asks
                                for (Sec. III-B) */
  NEXUS_ECUDA = 7,           /* a CUDA runtime or driver call failed */
  NEXUS_ETIMEOUT = 8,        /* a bounded device-side wait gave up; results are invalid */
  NEXUS_EOVERLAP = 9         /* destination rows overlap each other or the source rows */
} nexus_status;

enum { NEXUS_ROPE_NEOX = 0, NEXUS_ROPE_GPTJ = 1 };

/* Live paged KV cache. RoPE parameters are those of the runtime model; a
 * block is spliced only if its header carries the same ones (Sec. V-A). */
typedef struct nexus_kv_cache {
  void* k_pool;             /* device */
  void* v_pool;             /* device */
  int64_t n_pages;          /* pages per layer */
  int32_t n_layers;
  int32_t n_kv_heads;
  int32_t head_dim;         /* 128 */
  int32_t page_size;        /* 16 */
  int32_t v_transposed;     /* 0: row-major V; 1: token-innermost V (Sec. V-B) */
  int32_t rope_type;        /* NEXUS_ROPE_NEOX (half-split pairs) or NEXUS_ROPE_GPTJ */
  double rope_theta;        /* base b of theta_i = b^(-2i/d); 1e6 (Sec. III-B) */
  double rope_freq_scale;   /* linear position scale; 1.0 */
} nexus_kv_cache;

/* Device-resident analogue of a compiled tool block (Sec. V-A): its header
 * fields and its K/V tensors. Token j of the block was rotated at base_pos + j. */
typedef struct nexus_block {
  const void* k;            /* device [n_layers][n_tokens][n_kv_heads][head_dim] */
  const void* v;            /* device, same shape */
  int32_t n_tokens;
  int32_t base_pos;         /* RoPE anchor m0 */
  int32_t n_layers;
  int32_t n_kv_heads;
  int32_t head_dim;
  int32_t rope_type;
  double rope_theta;
  double rope_freq_scale;
} nexus_block;

enum { NEXUS_SRC_BLOCK = 0, NEXUS_SRC_CACHE = 1 };
enum { NEXUS_SEG_K_ONLY = 1 };

/* One run of destination rows written by nexus_splice_kv. */
typedef struct nexus_splice_segment {
  int32_t src_kind;         /* NEXUS_SRC_BLOCK or NEXUS_SRC_CACHE */
  int32_t src_index;        /* block index, or page-table row of the source sequence */
  int32_t src_start;        /* first block token, or first source position */
  int32_t dst_row;          /* page-table row of the destination sequence */
  int32_t dst_start;        /* first destination position */
  int32_t n_tokens;
  int32_t delta;            /* RoPE offset applied to K; 0 copies the bits (Sec. IV-A) */
  int32_t flags;            /* NEXUS_SEG_K_ONLY leaves V untouched */
} nexus_splice_segment;

/* Splice policy: threshold P = M, base fraction R_base and full-recompute
 * multiple K of Eq. 2 (paper defaults 256, 5, 4; tuned K = 16). */
typedef struct nexus_policy {
  int32_t splice_threshold; /* M = P */
  int32_t r_base_pct;       /* R_base in percent */
  int32_t full_mult;        /* K >= 2 */
} nexus_policy;

typedef struct nexus_insert {
  int32_t depth;            /* position in the pre-splice sequence, non-decreasing */
  int32_t block_index;      /* index into the blocks array */
} nexus_insert;

typedef struct nexus_page_pool nexus_page_pool;

/* ---------------------------------------------------------------- status */
const char* nexus_status_string(nexus_status s);
int32_t nexus_version(void);

/* Synchronises `stream`, then reports NEXUS_ETIMEOUT if any kernel of this
 * library on the current device gave up a bounded wait since the last call
 * (and clears that record), NEXUS_ERANGE if nexus_suffix_qkv or the splice
 * kernel (nexus_splice_kv, nexus_rope_rerotate, nexus_rope_rerotate_f32) met a
 * page id outside the pool in a device page table (and skipped the writes that
 * needed it), NEXUS_ECUDA if the stream reports an error, else NEXUS_OK. */
nexus_status nexus_device_status(nexus_stream stream);

/* Self-test of the failure path above, for callers that want to see it work on
 * their GPU: launches one CTA whose thread waits, with the same bounded
 * mbarrier wait the kernels use, on a barrier that nothing arrives on. The wait
 * gives up after budget_us microseconds and records a timeout, so the next
 * nexus_device_status returns NEXUS_ETIMEOUT (and clears the record) while the
 * context stays usable. budget_us must lie in [1, 1000000]; NEXUS_EINVAL
 * otherwise, NEXUS_ECUDA if the launch fails. */
nexus_status nexus_selftest_wait(uint32_t budget_us, nexus_stream stream);

/* ---------------------------------------------------------------- policy */
/* R(n_past) of Eq. 2 (Sec. III-C) as an exact fraction *num / *den in percent,
 * clamped to 100. Returns NEXUS_EINVAL for K < 2, M < 1 or R_base outside [0, 100]. */
nexus_status nexus_recompute_pct(int32_t n_past, const nexus_policy* policy,
                                 int64_t* num, int64_t* den);

/* ceil(S * R(n_past) / 100), at most S: the suffix that is invalidated and
 * re-decoded after a splice (Sec. V-A). Negative on invalid input. */
int32_t nexus_redecode_len(int32_t S, int32_t n_past, const nexus_policy* policy);

/* ceil(S * pct / 100) for a fixed percentage in [0, 100]; negative on invalid input. */
int32_t nexus_suffix_len(int32_t S, int32_t pct);

/* Fail-closed gate of Sec. III-B / III-C: NEXUS_EDECLINED if n_past exceeds the
 * threshold P and fewer than nexus_redecode_len(S, n_past) rows will be
 * re-decoded, else NEXUS_OK. */
nexus_status nexus_check_splice(int32_t n_past, int32_t S, int32_t n_redecode,
                                const nexus_policy* policy);

/* ------------------------------------------------------------- page pool */
/* Host allocator of cache pages (the analogue of the paper's cache-line
 * hardened bitmap allocator, Sec. V-C). `order` (nullable) gives the order in
 * which pages are handed out; NULL means 0, 1, 2, ... Thread-safe. */
nexus_status nexus_page_pool_create(int64_t n_pages, const int32_t* order,
                                    nexus_page_pool** out);
void nexus_page_pool_destroy(nexus_page_pool* pool);
/* Takes n pages in pool order; NEXUS_ENOMEM (and no change) if fewer are free. */
nexus_status nexus_page_pool_alloc(nexus_page_pool* pool, int32_t n, int32_t* pages);
/* Drops one reference from each page; a page whose last reference goes returns
 * to the back of the order. NEXUS_ERANGE for an id outside the pool,
 * NEXUS_EINVAL for a page that is already free or listed twice (nothing
 * changes then). */
nexus_status nexus_page_pool_free(nexus_page_pool* pool, int32_t n, const int32_t* pages);
int64_t nexus_page_pool_available(const nexus_page_pool* pool);
/* Adds one reference to each page, for a page shared by several page tables
 * (a warm prefix, Sec. V-D). Each page must be in use and listed once;
 * NEXUS_EINVAL / NEXUS_ERANGE otherwise (nothing changes). A page goes back to
 * the pool when nexus_page_pool_free has dropped every reference. */
nexus_status nexus_page_pool_retain(nexus_page_pool* pool, int32_t n, const int32_t* pages);
/* References held on a page: 0 when free, -1 for an id outside the pool. */
int64_t nexus_page_pool_refs(const nexus_page_pool* pool, int32_t page);
/* Copy-on-write before rows are written in place: every page of
 * h_pt[first_page, first_page + n) with more than one reference is replaced in
 * h_pt by a fresh page, the table's reference on the old page is dropped, and
 * the (old, fresh) pairs are written to src_pages / dst_pages (capacity pairs)
 * for nexus_copy_pages, which must run before the rows are written.
 * NEXUS_ENOMEM (nothing changes) if the pool or the capacity is too small. */
nexus_status nexus_page_pool_make_private(nexus_page_pool* pool, int32_t* h_pt,
                                          int32_t first_page, int32_t n, int32_t* src_pages,
                                          int32_t* dst_pages, int32_t capacity,
                                          int32_t* n_copies);

/* ---------------------------------------------------------- L0 warm arena */
/* The L0 exact-token radix arena (Sec. V-D): n_slots (1..32) sequence slots of
 * up to max_tokens tokens. A new request looks up the slot sharing the longest
 * exact-token prefix with it and starts from that prefix's KV instead of
 * recomputing it. A slot holds its sequence's tokens and one reference on each
 * cache page of its rows (no copy); a sequence forked from a slot shares the
 * pages that hold only prefix rows and gets a private copy of the page it will
 * go on writing, so reusing m warm tokens costs at most one page copy.
 * Rule for callers: rows [0, n) of a stored sequence must keep their bits while
 * a slot holds them; before writing any of them in place (re-rotation, Q/K/V
 * recompute of a suffix), make their pages private
 * (nexus_page_pool_make_private). Writing rows past n is free: slots never read
 * them. All memory is reserved by create; match, fork and store allocate
 * nothing. An arena is not thread-safe: serialise calls on one arena. */
typedef struct nexus_warm_arena nexus_warm_arena;
nexus_status nexus_warm_arena_create(int32_t n_slots, int32_t max_tokens,
                                     nexus_warm_arena** out);
/* Drops the slots' page references into `pool` (nullable) and frees the arena. */
void nexus_warm_arena_destroy(nexus_warm_arena* arena, nexus_page_pool* pool);
/* The slot sharing the longest exact-token prefix with tokens[0, n): *slot and
 * *prefix (its length); equal prefixes go to the most recently used slot;
 * *slot = -1, *prefix = 0 when no slot shares the first token. Changes no slot. */
nexus_status nexus_warm_arena_match(nexus_warm_arena* arena, const int32_t* tokens, int32_t n,
                                    int32_t* slot, int32_t* prefix);
/* Starts a sequence from the first m tokens of `slot` (m <= its length):
 * writes h_new_pt[0, ceil(m / 16)). Pages holding only rows < m are shared
 * (one more reference each); when m is not a multiple of 16 the page holding
 * row m - 1 is copied to a fresh page from `pool`, returned as one pair in
 * copy_src[0] -> copy_dst[0] (*n_copies = 1) for nexus_copy_pages. The new
 * sequence then writes its rows m.. itself. Counts as a use of the slot. */
nexus_status nexus_warm_arena_fork(nexus_warm_arena* arena, nexus_page_pool* pool, int32_t slot,
                                   int32_t m, int32_t* h_new_pt, int32_t max_pages,
                                   int32_t* copy_src, int32_t* copy_dst, int32_t* n_copies);
/* Enters a sequence of n tokens whose rows live in the pages h_pt[0, ceil(n' /
 * 16)), n' = min(n, max_tokens). If a slot already holds a sequence starting
 * with these n' tokens, only its use is refreshed. Otherwise the sequence
 * replaces the longest slot that holds a prefix of it, else the lowest empty
 * slot, else the least recently used one; that slot takes a reference on each
 * of the pages and drops those of the sequence it held. *slot_out (nullable)
 * receives the slot. */
nexus_status nexus_warm_arena_store(nexus_warm_arena* arena, nexus_page_pool* pool,
                                    const int32_t* tokens, int32_t n, const int32_t* h_pt,
                                    int32_t* slot_out);
/* A slot's token count (0 = empty) and, when h_pages is given, its pages
 * (capacity >= ceil(count / 16), else NEXUS_ENOMEM). */
nexus_status nexus_warm_arena_slot(const nexus_warm_arena* arena, int32_t slot, int32_t* n_tokens,
                                   int32_t* h_pages, int32_t capacity);

/* --------------------------------------------------------------- planner */
/* Plans the insertion of blocks into one sequence of length n_past whose page
 * table is h_old_pt (host, [max_pages]). The post-splice sequence is
 * live[0:d1] ++ block1 ++ live[d1:d2] ++ ... ++ live[dk:n_past]; block rows are
 * reanchored by delta = final position - base_pos (Sec. III-B) and displaced
 * live rows are re-rotated by the number of block rows inserted before them.
 * Pages that hold no changed row are shared with the old table; every other
 * page of the new table is taken from `pool`, so no destination row overlaps a
 * source row. Appending at the cursor (all depths == n_past) keeps the
 * partially filled last page in place.
 *   h_new_pt    out [max_pages]: the new page table (entries past the
 *               sequence end are set to -1)
 *   segs        out: the segments for nexus_splice_kv, reading live rows from
 *               page-table row old_row and writing row new_row
 *   freed       out (nullable, capacity max_pages): old pages the new table
 *               no longer uses; the caller frees them once the splice is done
 * Returns NEXUS_ENOMEM if the pool or seg_capacity is too small (the pool is
 * then unchanged), NEXUS_ERANGE if the result exceeds max_pages * 16 rows. */
nexus_status nexus_plan_splice(nexus_page_pool* pool, const int32_t* h_old_pt,
                               int32_t n_past, int32_t max_pages,
                               const nexus_block* blocks, int32_t n_blocks,
                               const nexus_insert* inserts, int32_t n_inserts,
                               int32_t old_row, int32_t new_row, int32_t* h_new_pt,
                               nexus_splice_segment* segs, int32_t seg_capacity,
                               int32_t* n_segs, int32_t* freed, int32_t* n_freed);

/* ----------------------------------------------------------------- splice */
/* Writes every segment for layers [layer_begin, layer_end) in one launch
 * (Sec. V-A splice; Sec. III-B reanchoring; Sec. V-B transposed V). K rows are
 * rotated by the segment's delta in float32 from float64-reduced angles and
 * stored round-to-nearest-even; delta = 0 copies K bits unchanged; V bits are
 * always copied unchanged.
 *   d_page_tables  device int32 [n_rows][max_pages]
 *   h_page_tables  host copy of the same (nullable). When given, every page
 *                  id is range-checked and destination rows are checked not
 *                  to overlap each other or any source row (NEXUS_EOVERLAP);
 *                  a segment may read and write the same rows only if it is
 *                  K-only (an in-place rotation). Either way the kernel checks
 *                  each page id it reads from the device table against the
 *                  pool before using it: the rows of one destination page
 *                  whose ids (destination, or a source page) fall outside
 *                  [0, n_pages) are skipped whole, never dereferenced, and
 *                  nexus_device_status then reports NEXUS_ERANGE. Overlap is
 *                  only checked with the host tables.
 *   blocks         host array of n_blocks descriptors; each block's RoPE
 *                  parameters and shape must match the cache
 *                  (NEXUS_EROPE_MISMATCH / NEXUS_ELAYOUT)
 *   segments       host array of n_segments (at most 4096)
 * Block layer l feeds cache layer l. */
nexus_status nexus_splice_kv(const nexus_kv_cache* cache,
                             const int32_t* d_page_tables, const int32_t* h_page_tables,
                             int32_t n_rows, int32_t max_pages,
                             const nexus_block* blocks, int32_t n_blocks,
                             const nexus_splice_segment* segments, int32_t n_segments,
                             int32_t layer_begin, int32_t layer_end, nexus_stream stream);

/* In-place rotation of the keys of positions [pos_begin, pos_begin + n_tokens)
 * of page-table row `row` by `delta` positions (Sec. III-B, Eq. 1), for layers
 * [layer_begin, layer_end). V is untouched. */
nexus_status nexus_rope_rerotate(const nexus_kv_cache* cache,
                                 const int32_t* d_page_tables, const int32_t* h_page_tables,
                                 int32_t n_rows, int32_t max_pages, int32_t row,
                                 int32_t pos_begin, int32_t n_tokens, int32_t delta,
                                 int32_t layer_begin, int32_t layer_end, nexus_stream stream);

/* The rotation of nexus_rope_rerotate written, unrounded, as float32 into
 * out_f32 (device [layer_end - layer_begin][n_tokens][n_kv_heads][head_dim]);
 * the cache is only read. It exposes the float32 arithmetic ahead of the bf16
 * store for verification. */
nexus_status nexus_rope_rerotate_f32(const nexus_kv_cache* cache,
                                     const int32_t* d_page_tables, const int32_t* h_page_tables,
                                     int32_t n_rows, int32_t max_pages, int32_t row,
                                     int32_t pos_begin, int32_t n_tokens, int32_t delta,
                                     int32_t layer_begin, int32_t layer_end,
                                     float* out_f32, nexus_stream stream);

/* Bit-exact copy of whole pages src_pages[i] -> dst_pages[i] (K and V, all
 * heads) for layers [layer_begin, layer_end): the in-arena KV copy of the
 * paper's L0 radix arena (Sec. V-D), also used for copy-on-write. Host arrays,
 * at most 2048 pairs per call; NEXUS_EOVERLAP if a page is both a source and a
 * destination or is written twice. */
nexus_status nexus_copy_pages(const nexus_kv_cache* cache, const int32_t* h_src_pages,
                              const int32_t* h_dst_pages, int32_t n, int32_t layer_begin,
                              int32_t layer_end, nexus_stream stream);

/* -------------------------------------------------------------- attention */
/* Causal GQA attention of the last q_len[s] positions of each sequence s over
 * its kv_len[s] cached positions (Sec. III-A; the redecoded suffix of
 * Sec. III-C / Sec. V-A). Query t of sequence s sits at position
 * kv_len[s] - q_len[s] + t and sees keys at positions <= its own; query head h
 * reads KV head h / (n_q_heads / n_kv_heads). Scores are scaled by
 * 1/sqrt(head_dim). bf16 operands, float32 accumulation; O is bf16 and LSE
 * (natural log of the softmax denominator of the scaled scores) float32.
 *   d_page_tables  device int32 [n_rows][max_pages]
 *   h_rows         host [n_seqs]: page-table row of each sequence (nullable:
 *                  sequence s uses row s)
 *   h_kv_len, h_q_len  host [n_seqs]; 0 <= q_len <= kv_len <= max_pages * 16
 *   q, out         device bf16, see the layout above; sequences are packed
 *                  back to back along the token axis in order
 *   lse            device float (nullable)
 *   n_seqs         1 .. 512
 *   split_kv       number of key-range partitions: 1 = none, 2 .. 32 as
 *                  given (larger values are taken as 32), 0 = chosen by the
 *                  library from the work size and SM count (at most 32)
 *   workspace      device scratch for split partials (nullable when no split
 *                  is used); its size comes from nexus_attention_workspace_size
 *                  with the same arguments; NEXUS_ENOMEM if too small
 * Cache slots past kv_len may hold any bits: they never reach the output. */
nexus_status nexus_suffix_attention(const nexus_kv_cache* cache,
                                    const int32_t* d_page_tables, int32_t n_rows,
                                    int32_t max_pages, int32_t n_seqs, const int32_t* h_rows,
                                    const int32_t* h_kv_len, const int32_t* h_q_len,
                                    const void* q, void* out, float* lse, int32_t n_q_heads,
                                    int32_t layer_begin, int32_t layer_end, int32_t split_kv,
                                    void* workspace, size_t workspace_bytes,
                                    nexus_stream stream);

/* nexus_suffix_attention with attention-logit soft-capping, the attention of the
 * models whose V cache is token-innermost (Sec. V-B): each scaled score s is
 * replaced by softcap * tanh(s / softcap) before the softmax (LSE is over the
 * capped scores). softcap > 0 (e.g. 50); NEXUS_EINVAL otherwise. Both V
 * layouts are accepted. */
nexus_status nexus_suffix_attention_softcap(const nexus_kv_cache* cache,
                                            const int32_t* d_page_tables, int32_t n_rows,
                                            int32_t max_pages, int32_t n_seqs,
                                            const int32_t* h_rows, const int32_t* h_kv_len,
                                            const int32_t* h_q_len, const void* q, void* out,
                                            float* lse, int32_t n_q_heads, int32_t layer_begin,
                                            int32_t layer_end, int32_t split_kv, void* workspace,
                                            size_t workspace_bytes, float softcap,
                                            nexus_stream stream);

/* Full causal re-prefill: nexus_suffix_attention with q_len = kv_len (the
 * R = 100 % end point of Eq. 2, Sec. III-C). */
nexus_status nexus_reprefill(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                             int32_t n_rows, int32_t max_pages, int32_t n_seqs,
                             const int32_t* h_rows, const int32_t* h_kv_len, const void* q,
                             void* out, float* lse, int32_t n_q_heads, int32_t layer_begin,
                             int32_t layer_end, int32_t split_kv, void* workspace,
                             size_t workspace_bytes, nexus_stream stream);

/* ------------------------------------------------- suffix Q/K/V recompute */
/* The re-decode half of stitching the seam (Sec. V-A): after the splice, the
 * last q_len[s] positions of each sequence are invalidated and re-decoded, which
 * gives each of those tokens a fresh query, key and value. For one layer this
 * computes, per token, y = x W^T + b, splits y into n_q_heads query heads, then
 * n_kv_heads key heads, then n_kv_heads value heads (128 features each), rotates
 * the query and key heads at the token's position (RoPE of Sec. III-B with the
 * cache's parameters), writes the queries to q_out and the keys and values into
 * the token's slot of the paged cache at `layer` (either V layout, Sec. V-B).
 *   sequences   token t of sequence s (t < q_len[s]) sits at position
 *               kv_len[s] - q_len[s] + t of page-table row h_rows[s] (h_rows
 *               NULL: row s); its input is row q_off[s] + t of x, where
 *               q_off[s] = sum of the earlier q_len
 *   x           device bf16 [sum of q_len][hidden] (the layer's normalised
 *               hidden states of the re-decoded tokens); hidden a multiple of 8
 *   w_qkv       device bf16 [(n_q_heads + 2 n_kv_heads) * 128][hidden]
 *   b_qkv       device float [(n_q_heads + 2 n_kv_heads) * 128], or NULL
 *   q_out       device bf16 [sum of q_len][n_q_heads][128], the layout the
 *               attention calls read their queries in
 *   h_page_tables  host copy of the page tables (nullable): when given, every
 *               written page is checked to lie in the pool (NEXUS_ERANGE) and
 *               no two tokens may write one slot (NEXUS_EOVERLAP); without it
 *               the kernel skips writes to a page id outside the pool and
 *               nexus_device_status reports NEXUS_ERANGE
 * Products accumulate in float32 on the tensor cores; the bias, the rotation
 * (angles reduced to one float ulp) and the bf16 rounding of the stores follow.
 * kv_len <= 2^24 (NEXUS_ERANGE). Writes nothing outside q_out and those slots. */
nexus_status nexus_suffix_qkv(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                              const int32_t* h_page_tables, int32_t n_rows, int32_t max_pages,
                              int32_t n_seqs, const int32_t* h_rows, const int32_t* h_kv_len,
                              const int32_t* h_q_len, const void* x, int32_t hidden,
                              const void* w_qkv, const float* b_qkv, int32_t n_q_heads,
                              int32_t layer, void* q_out, nexus_stream stream);

/* ------------------------------------------------- INT8 tool scan + gate */
/* INT8 quantisation of embeddings for the tool scan (Sec. IV-A), on the host:
 * per row of h_x [n][dim] (finite floats), scale = max|x| / 127 and code =
 * round-half-even(x / scale) in [-127, 127], in float32; an all-zero row gets
 * scale 0 and zero codes. NEXUS_EINVAL for a non-finite input. */
nexus_status nexus_slb_quantize(const float* h_x, int32_t n, int32_t dim, int8_t* h_codes,
                                float* h_scales);
/* Bytes of workspace nexus_slb_route needs for a registry of n_tools. */
size_t nexus_slb_workspace_size(int32_t n_tools);
/* The semantic lookaside buffer's scan and margin gate (Sec. IV-A): for every
 * query q, score(q, t) = float(dot(codes_q, codes_t)) * (scale_q * scale_t)
 * over all tools t (float32; the integer dot is exact), the two best tools
 * (higher score first, then lower index) and their scores, and the decision:
 * route[q] = the best tool when top1 - top2 > tau, else -1 (escalate to the
 * cross-encoder, which is not part of this library). With one tool the
 * runner-up is index -1 with score -inf and the query always routes.
 *   d_tools     device int8 [n_tools][dim], dim a multiple of 4 (<= 4096),
 *               16-byte aligned; d_tool_scales float [n_tools]
 *   d_queries   device int8 [n_queries][dim], d_query_scales float [n_queries]
 *   d_top_idx   device int32 [n_queries][2]; d_top_score float [n_queries][2];
 *               d_route int32 [n_queries]
 *   workspace   device, nexus_slb_workspace_size(n_tools) bytes, 16-byte
 *               aligned, all zero before its first use; every call leaves it
 *               ready for the next (calls sharing one workspace must be ordered
 *               on the GPU, e.g. by one stream)
 * Queries are scanned 32 per launch. tau (e.g. 0.0136) must be finite. */
nexus_status nexus_slb_route(const int8_t* d_tools, const float* d_tool_scales, int32_t n_tools,
                             int32_t dim, const int8_t* d_queries, const float* d_query_scales,
                             int32_t n_queries, float tau, int32_t* d_top_idx, float* d_top_score,
                             int32_t* d_route, void* workspace, size_t workspace_bytes,
                             nexus_stream stream);

/* Bytes of workspace nexus_suffix_attention needs for these arguments
 * (0 when no split is used). *splits_out (nullable) receives the partition
 * count the call will use. Uses the current device's SM count, or 152 when no
 * device is visible. Arguments the attention call would reject (n_seqs outside
 * 1 .. 512, q_len > kv_len, bad head counts) give 0 and *splits_out = 0. */
size_t nexus_attention_workspace_size(int32_t n_seqs, const int32_t* h_kv_len,
                                      const int32_t* h_q_len, int32_t n_q_heads,
                                      int32_t n_kv_heads, int32_t n_layers_call,
                                      int32_t split_kv, int32_t* splits_out);

/* ------------------------------------------------ attention, no allocation */
/* nexus_suffix_attention for callers that cannot allocate device memory: code
 * running while a stream is captured (no cudaMalloc there), plug-ins handed only
 * their input and output buffers, or processes with a fixed memory pool. The
 * paper has no counterpart; this is a deployment convenience of this library.
 *
 * Arguments, results and errors are those of nexus_suffix_attention, without
 * the workspace: the split-KV partials live in a 32 MiB array inside the
 * library, which every GPU that loads the library holds until the process
 * exits. Arguments are checked first, exactly as nexus_suffix_attention checks
 * them; then requests whose partials need more than 32 MiB (see
 * nexus_attention_workspace_size) return NEXUS_ENOMEM before any launch; pass
 * split_kv = 1 to need none. The first call in each CUDA context (the current
 * device's primary context, unless the caller made another one current) looks
 * up the array's device address in that context and remembers it; make that
 * first call before any stream capture. Every call shares the one array and overwrites what the
 * previous call left (nothing in it needs to start at zero), so calls that may
 * run at the same time on the GPU (different streams, no ordering between
 * them) race; order them on one stream or with events. Allocates nothing. */
nexus_status nexus_suffix_attention_noalloc(const nexus_kv_cache* cache,
                                            const int32_t* d_page_tables, int32_t n_rows,
                                            int32_t max_pages, int32_t n_seqs,
                                            const int32_t* h_rows, const int32_t* h_kv_len,
                                            const int32_t* h_q_len, const void* q, void* out,
                                            float* lse, int32_t n_q_heads, int32_t layer_begin,
                                            int32_t layer_end, int32_t split_kv,
                                            nexus_stream stream);

/* ------------------------------------------------------ host staging memory */
/* Page-locked host memory for the host<->device copies around the path (the
 * per-layer Q/O transfers of a re-prefill, a compiled block read from host
 * memory). The paper has no counterpart; this is a deployment convenience of
 * this library. The library maps `bytes` of fresh anonymous memory, faults it
 * in and registers it with the CUDA driver, so cudaMemcpyAsync from or to it is
 * asynchronous. Requests of at least a quarter of the kernel's transparent huge
 * page size are rounded up to whole huge pages, aligned to them, advised to use
 * them and, once faulted in, offered for collapse into huge pages (where the
 * kernel supports it; both are best effort); smaller ones are rounded up to the
 * base page size. On Grace hosts
 * (64 KiB base pages, 512 MiB huge pages) copies from page-locked memory on
 * scattered base pages, whether from cudaHostAlloc or registered, ran at 4 to
 * 200 GB/s depending on the buffer; from huge pages at a steady 200 GB/s.
 *
 * *out receives the page-aligned address (zero-filled memory) or NULL.
 * NEXUS_EINVAL for bytes == 0 or out == NULL, NEXUS_ENOMEM if the mapping
 * fails, NEXUS_ECUDA if the driver refuses the registration (no GPU, or the
 * page-locked limit is reached); nothing is left mapped on failure. The caller
 * owns the memory and returns it with nexus_host_free, giving the same size. */
nexus_status nexus_host_alloc(size_t bytes, void** out);
/* Unregisters and unmaps memory from nexus_host_alloc. No copy may still be
 * reading or writing it. NULL is a no-op. NEXUS_EINVAL, with nothing changed,
 * for bytes == 0, an address nexus_host_alloc did not return (or already
 * freed), or a size that maps to a different length than that allocation's;
 * NEXUS_ECUDA if the driver refuses to unregister it (the memory then stays
 * mapped and may be freed again later). */
nexus_status nexus_host_free(void* p, size_t bytes);

#ifdef __cplusplus
}
#endif

#endif /* NEXUS_H */
