// Launch-side structures shared by the C-ABI layer and the CUDA kernels.
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>
#include <cstdint>

#include "nexus.h"

namespace nexus {

constexpr int kHeadDim = 128;
constexpr int kPageSize = 16;
constexpr int kMaxKvHeads = 16;

// ------------------------------------------------------------------ splice
// One destination run, resolved for the device. A CTA handles the rows of one
// segment that fall into one destination page ("piece"), for one layer.
struct DevSegment {
  const uint16_t* src_k;     // block K at layer 0 (nullptr: source is the cache)
  const uint16_t* src_v;     // block V at layer 0
  int64_t src_layer_stride;  // elements between consecutive layers of the block
  int32_t src_row;           // page-table row of a cache source (-1 for a block)
  int32_t src_start;
  int32_t dst_row;
  int32_t dst_start;
  int32_t n_tokens;
  int32_t delta;
  int32_t flags;
  int32_t piece_begin;       // prefix sum of pieces over earlier segments
};

constexpr int kMaxSegmentsPerLaunch = 224;

enum SpliceOut : int32_t { kOutPool = 0, kOutF32 = 1 };

struct SpliceLaunch {
  uint16_t* k_pool;
  uint16_t* v_pool;
  const int32_t* page_tables;
  float* out_f32;            // kOutF32: [n_layers_call][n_tokens][Hkv][128]
  int64_t n_pages;
  int32_t n_kv_heads;
  int32_t max_pages;
  int32_t layer_begin;
  int32_t n_layers_call;
  int32_t n_segments;
  int32_t n_pieces;
  int32_t v_transposed;
  int32_t rope_gptj;
  int32_t out_mode;
  int32_t out_pos_begin;     // kOutF32: source position of output token 0
  double inv_freq_over_pi[kHeadDim / 2];   // theta_i / pi
  DevSegment seg[kMaxSegmentsPerLaunch];
};

cudaError_t launch_splice(const SpliceLaunch& p, cudaStream_t stream);
// Reads and clears the splice kernel's record of a page id outside the pool.
cudaError_t splice_take_status(unsigned int* bad_page, cudaStream_t stream);

// -------------------------------------------------------------- page copy
constexpr int kMaxPageCopies = 2048;
struct PageCopyLaunch {
  uint16_t* k_pool;
  uint16_t* v_pool;
  int64_t n_pages;
  int32_t n_kv_heads;
  int32_t layer_begin;
  int32_t n_layers_call;
  int32_t n;
  int32_t src[kMaxPageCopies];
  int32_t dst[kMaxPageCopies];
};
cudaError_t launch_page_copy(const PageCopyLaunch& p, cudaStream_t stream);

// --------------------------------------------------------------- attention
constexpr int kMaxSeqs = 512;
constexpr int kMaxSplits = 32;

struct AttnSeq {
  int32_t kv_len;
  int32_t q_len;
  int32_t q_off;        // first packed token of this sequence in Q / O
  int32_t pt_row;
};

struct AttnLaunch {
  const int32_t* page_tables;
  uint16_t* out;            // bf16 O (no split) [n_layers_call][n_tok][Hq][128]
  float* lse;               // nullable
  float* part_o;            // split partials [splits][n_layers_call][n_tok][Hq][128]
  float* part_lse;          // [splits][n_layers_call][n_tok][Hq]
  int32_t max_pages;
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t group;            // n_q_heads / n_kv_heads
  int32_t tile_tokens;      // query tokens per 128-row tile = 128 / group
  int32_t n_tok;            // packed tokens (sum of q_len)
  int32_t n_pages;          // pages per layer (as int: the pool index range)
  int32_t layer_begin;
  int32_t n_layers_call;
  int32_t n_seqs;
  int32_t splits;
  int32_t v_transposed;
  int32_t total_tiles;      // CTAs per (KV head, layer, split): pairs of 128-row query tiles
  float scale_log2;         // log2(e) / sqrt(head_dim)
  float softcap_in;         // soft-capping: 2 log2(e) / (sqrt(head_dim) cap)
  float softcap_out;        // soft-capping: cap log2(e); 0 = no soft-capping
  int32_t tile_prefix[kMaxSeqs + 1];   // first CTA (tile pair) of each sequence
  AttnSeq seq[kMaxSeqs];
  int32_t pair0[kMaxSeqs];  // first tile pair of each sequence in this launch
  int32_t short_rows;       // this launch's tile pairs hold rows that see fewer than 128 keys
  // Key splits of a pair holding two query tiles / one query tile (both at
  // most `splits`, which sizes the grid and the partials).
  int32_t splits_pair;
  int32_t splits_single;
  // Split plans with per-kind counts: the grid's x runs over exactly the
  // (tile pair, split) CTAs of every sequence; cta_prefix[s] is the first of
  // sequence s (kinds launches only).
  int32_t cta_prefix[kMaxSeqs + 1];
};

struct AttnMaps {
  CUtensorMap q;
  CUtensorMap k;
  CUtensorMap v;
  // The same K / V with boxes of eight pages: one copy per 64-column half of a
  // key tile whose eight page ids are consecutive.
  CUtensorMap k8;
  CUtensorMap v8;
};

cudaError_t launch_attention(const AttnLaunch& p, const AttnMaps& maps, cudaStream_t stream);
cudaError_t launch_attn_combine(const AttnLaunch& p, cudaStream_t stream);
// Reads and clears the timeout record of the current device.
cudaError_t attention_take_timeout(unsigned int* flag, cudaStream_t stream);
// One CTA waits, bounded by budget_ns, on a barrier nothing arrives on.
cudaError_t launch_wait_selftest(uint64_t budget_ns, cudaStream_t stream);

// ------------------------------------------------- suffix Q/K/V recompute
struct QkvLaunch {
  const int32_t* page_tables;
  const float* bias;        // nullable, [n_heads * 128]
  uint16_t* q_out;          // [n_tok][n_q_heads][128]
  uint16_t* k_pool;
  uint16_t* v_pool;
  int64_t n_pages;
  int32_t max_pages;
  int32_t n_q_heads;
  int32_t n_kv_heads;
  int32_t n_heads;          // n_q_heads + 2 n_kv_heads
  int32_t layer;
  int32_t v_transposed;
  int32_t rope_gptj;
  int32_t n_tok;            // packed tokens (sum of q_len)
  int32_t k_blocks;         // ceil(hidden / 64)
  int32_t n_tiles;          // feature tiles: ceil(n_heads / 2), or n_heads with short tiles
  int32_t m_tiles;          // 128-token tiles: ceil(n_tok / 128)
  int32_t group_m;          // token tiles per raster band
  int32_t total_tiles;      // m_tiles * n_tiles
  int32_t n_seqs;
  int32_t short_tiles;      // n_tok <= 64: one-head tiles, 64 token rows per stage
  int32_t pair_split;       // short tiles: two CTAs (a cluster) per tile split the hidden dim
  float inv_freq_hi[kHeadDim / 2];   // theta_i / pi = hi + lo
  float inv_freq_lo[kHeadDim / 2];
  AttnSeq seq[kMaxSeqs];
};

struct QkvMaps {
  CUtensorMap x;            // [n_tok][hidden], box 128 x 64 (64 x 64 for short tiles)
  CUtensorMap w;            // [n_heads * 128][hidden], box 256 x 64 (128 x 64 for short tiles)
};

cudaError_t launch_qkv(const QkvLaunch& p, const QkvMaps& maps, int grid, cudaStream_t stream);
// Reads and clears the device records of the Q/K/V kernel: a wait that gave up,
// a page id outside the pool.
cudaError_t qkv_take_status(unsigned int* timeout, unsigned int* bad_page, cudaStream_t stream);

// ----------------------------------------------------- INT8 tool scan + gate
struct SlbLaunch {
  const int8_t* tools;          // [n_tools][dim]
  const float* tool_scales;     // [n_tools]
  const int8_t* queries;        // [n_queries][dim] (this launch's queries)
  const float* query_scales;    // [n_queries]
  int32_t* top_idx;             // [n_queries][2]
  float* top_score;             // [n_queries][2]
  int32_t* route;               // [n_queries]
  float* part_score;            // workspace [grid][32][2]
  int32_t* part_idx;            // workspace [grid][32][2]
  unsigned int* counter;        // workspace ticket, 0 between calls
  int32_t n_tools;
  int32_t dim;                  // multiple of 4
  int32_t n_queries;            // 1..32
  int32_t tools_per_cta;
  float tau;
  int32_t chunk_tools;          // streamed scan: tools per shared-memory stage (0: not streamed)
  int32_t stages;               // streamed scan: stages in the ring
};
constexpr int kSlbMaxQueries = 32;
constexpr int kSlbSmallQueries = 4;   // up to this many queries: the latency path
// Few queries over at least this many tools: the registry streams through
// shared memory by bulk copies (two CTAs per SM).
constexpr int kSlbStreamMinTools = 16384;
constexpr int kSlbStreamSmemPerCta = 110 * 1024;  // stage ring + queries, two CTAs per SM
cudaError_t launch_slb(const SlbLaunch& p, int grid, cudaStream_t stream);
// 5..32 queries over at least kSlbStreamMinTools tools, dim a multiple of 64 up
// to kSlbTcMaxDim: tensor-core scan; `tools` maps the int8 codes [n_tools][dim]
// with 64 x 128 boxes.
constexpr int kSlbTcMaxDim = 1024;
cudaError_t launch_slb_tc(const SlbLaunch& p, const CUtensorMap& tools, int grid,
                          cudaStream_t stream);
cudaError_t slb_take_timeout(unsigned int* flag, cudaStream_t stream);

}  // namespace nexus
