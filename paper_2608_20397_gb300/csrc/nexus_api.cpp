// C-ABI entry points of the device path: argument validation on the host,
// TMA tensor-map encoding, and the launches of the splice, page-copy and
// attention kernels.
#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>
#include <sys/mman.h>
#include <unistd.h>

#include <algorithm>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <map>
#include <memory>
#include <mutex>
#include <vector>

#include "internal.h"

using namespace nexus;

namespace {

constexpr int kNumSmsFallback = 152;

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

nexus_status check_cache(const nexus_kv_cache* c) {
  if (!c || !c->k_pool || !c->v_pool) return NEXUS_EINVAL;
  if (c->head_dim != kHeadDim || c->page_size != kPageSize) return NEXUS_ELAYOUT;
  if (c->n_kv_heads < 1 || c->n_kv_heads > kMaxKvHeads || c->n_layers < 1 || c->n_pages < 1)
    return NEXUS_EINVAL;
  if (c->n_pages * static_cast<int64_t>(c->n_layers) > 0x7FFFFFFFLL) return NEXUS_ERANGE;
  if (!aligned16(c->k_pool) || !aligned16(c->v_pool)) return NEXUS_ELAYOUT;
  if (c->rope_type != NEXUS_ROPE_NEOX && c->rope_type != NEXUS_ROPE_GPTJ) return NEXUS_EINVAL;
  if (!(c->rope_theta > 1.0) || !(c->rope_freq_scale > 0.0) || !std::isfinite(c->rope_theta) ||
      !std::isfinite(c->rope_freq_scale))
    return NEXUS_EINVAL;
  if (c->v_transposed != 0 && c->v_transposed != 1) return NEXUS_EINVAL;
  return NEXUS_OK;
}

nexus_status check_layers(const nexus_kv_cache* c, int32_t lb, int32_t le) {
  if (lb < 0 || le > c->n_layers || lb > le) return NEXUS_ERANGE;
  return NEXUS_OK;
}

// A block is spliced only if its header matches the runtime model (Sec. V-A).
nexus_status check_block(const nexus_kv_cache* c, const nexus_block& b) {
  if (!b.k || !b.v || b.n_tokens < 0) return NEXUS_EINVAL;
  if (!aligned16(b.k) || !aligned16(b.v)) return NEXUS_ELAYOUT;
  if (b.n_layers != c->n_layers || b.n_kv_heads != c->n_kv_heads || b.head_dim != c->head_dim)
    return NEXUS_ELAYOUT;
  if (b.rope_type != c->rope_type || b.rope_theta != c->rope_theta ||
      b.rope_freq_scale != c->rope_freq_scale)
    return NEXUS_EROPE_MISMATCH;
  return NEXUS_OK;
}

void fill_inv_freq_over_pi(const nexus_kv_cache* c, double* out) {
  for (int i = 0; i < kHeadDim / 2; ++i)
    out[i] = c->rope_freq_scale * std::pow(c->rope_theta, -2.0 * i / kHeadDim) / M_PI;
}

int num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) { cudaGetLastError(); return kNumSmsFallback; }
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) {
    cudaGetLastError();
    return kNumSmsFallback;
  }
  return n;
}

int32_t pieces_of(int32_t dst_start, int32_t n) {
  if (n <= 0) return 0;
  return (dst_start + n - 1) / kPageSize - dst_start / kPageSize + 1;
}

// Destination / source slot bookkeeping for the overlap check, kept per thread
// so repeated calls do not reallocate.
struct SlotMarks {
  std::vector<int32_t> owner;
  std::vector<int64_t> touched;
  void ensure(int64_t n) {
    if (static_cast<int64_t>(owner.size()) < n) owner.assign(static_cast<size_t>(n), -1);
  }
  void reset() {
    for (int64_t s : touched) owner[s] = -1;
    touched.clear();
  }
};

nexus_status validate_segments(const nexus_kv_cache* c, const int32_t* h_pt, int32_t n_rows,
                               int32_t max_pages, const nexus_block* blocks, int32_t n_blocks,
                               const nexus_splice_segment* segs, int32_t n_segs) {
  const int64_t cap = static_cast<int64_t>(max_pages) * kPageSize;
  for (int32_t i = 0; i < n_segs; ++i) {
    const nexus_splice_segment& s = segs[i];
    if (s.n_tokens < 0 || s.dst_start < 0 || s.src_start < 0) return NEXUS_EINVAL;
    if (s.dst_row < 0 || s.dst_row >= n_rows) return NEXUS_ERANGE;
    if (s.dst_start + static_cast<int64_t>(s.n_tokens) > cap) return NEXUS_ERANGE;
    if (s.flags & ~NEXUS_SEG_K_ONLY) return NEXUS_EINVAL;
    if (s.src_kind == NEXUS_SRC_BLOCK) {
      if (s.src_index < 0 || s.src_index >= n_blocks) return NEXUS_ERANGE;
      const nexus_status st = check_block(c, blocks[s.src_index]);
      if (st != NEXUS_OK) return st;
      if (s.src_start + static_cast<int64_t>(s.n_tokens) > blocks[s.src_index].n_tokens)
        return NEXUS_ERANGE;
    } else if (s.src_kind == NEXUS_SRC_CACHE) {
      if (s.src_index < 0 || s.src_index >= n_rows) return NEXUS_ERANGE;
      if (s.src_start + static_cast<int64_t>(s.n_tokens) > cap) return NEXUS_ERANGE;
    } else {
      return NEXUS_EINVAL;
    }
  }
  if (!h_pt) return NEXUS_OK;

  thread_local SlotMarks marks;
  marks.ensure(c->n_pages * kPageSize);
  nexus_status result = NEXUS_OK;
  auto slot_of = [&](int32_t row, int32_t pos, int64_t* slot) -> bool {
    const int32_t pg = h_pt[static_cast<int64_t>(row) * max_pages + pos / kPageSize];
    if (pg < 0 || pg >= c->n_pages) return false;
    *slot = static_cast<int64_t>(pg) * kPageSize + pos % kPageSize;
    return true;
  };
  for (int32_t i = 0; i < n_segs && result == NEXUS_OK; ++i) {
    const nexus_splice_segment& s = segs[i];
    for (int32_t r = 0; r < s.n_tokens; ++r) {
      int64_t slot;
      if (!slot_of(s.dst_row, s.dst_start + r, &slot)) { result = NEXUS_ERANGE; break; }
      if (marks.owner[slot] != -1) { result = NEXUS_EOVERLAP; break; }
      marks.owner[slot] = i;
      marks.touched.push_back(slot);
    }
  }
  for (int32_t i = 0; i < n_segs && result == NEXUS_OK; ++i) {
    const nexus_splice_segment& s = segs[i];
    if (s.src_kind != NEXUS_SRC_CACHE) continue;
    const bool in_place = (s.flags & NEXUS_SEG_K_ONLY) && s.src_index == s.dst_row &&
                          s.src_start == s.dst_start;
    for (int32_t r = 0; r < s.n_tokens; ++r) {
      int64_t slot;
      if (!slot_of(s.src_index, s.src_start + r, &slot)) { result = NEXUS_ERANGE; break; }
      const int32_t o = marks.owner[slot];
      if (o != -1 && !(o == i && in_place)) { result = NEXUS_EOVERLAP; break; }
    }
  }
  marks.reset();
  return result;
}

nexus_status launch_segments(const nexus_kv_cache* c, const int32_t* d_pt, int32_t max_pages,
                             const nexus_block* blocks, const nexus_splice_segment* segs,
                             int32_t n_segs, int32_t lb, int32_t le, int32_t out_mode,
                             float* out_f32, int32_t out_pos_begin, cudaStream_t stream) {
  std::unique_ptr<SpliceLaunch> p(new SpliceLaunch());
  std::memset(p.get(), 0, sizeof(SpliceLaunch));
  p->k_pool = static_cast<uint16_t*>(c->k_pool);
  p->v_pool = static_cast<uint16_t*>(c->v_pool);
  p->page_tables = d_pt;
  p->out_f32 = out_f32;
  p->n_pages = c->n_pages;
  p->n_kv_heads = c->n_kv_heads;
  p->max_pages = max_pages;
  p->layer_begin = lb;
  p->n_layers_call = le - lb;
  p->v_transposed = c->v_transposed;
  p->rope_gptj = c->rope_type == NEXUS_ROPE_GPTJ;
  p->out_mode = out_mode;
  p->out_pos_begin = out_pos_begin;
  fill_inv_freq_over_pi(c, p->inv_freq_over_pi);
  int32_t i = 0;
  while (i < n_segs) {
    int32_t ns = 0, pieces = 0;
    for (; i < n_segs && ns < kMaxSegmentsPerLaunch; ++i) {
      const nexus_splice_segment& s = segs[i];
      const int32_t np = pieces_of(s.dst_start, s.n_tokens);
      if (np == 0) continue;
      DevSegment& d = p->seg[ns++];
      if (s.src_kind == NEXUS_SRC_BLOCK) {
        const nexus_block& b = blocks[s.src_index];
        d.src_k = static_cast<const uint16_t*>(b.k);
        d.src_v = static_cast<const uint16_t*>(b.v);
        d.src_layer_stride = static_cast<int64_t>(b.n_tokens) * c->n_kv_heads * kHeadDim;
        d.src_row = -1;
      } else {
        d.src_k = nullptr;
        d.src_v = nullptr;
        d.src_layer_stride = 0;
        d.src_row = s.src_index;
      }
      d.src_start = s.src_start;
      d.dst_row = s.dst_row;
      d.dst_start = s.dst_start;
      d.n_tokens = s.n_tokens;
      d.delta = s.delta;
      d.flags = s.flags;
      d.piece_begin = pieces;
      pieces += np;
    }
    if (ns == 0) continue;
    p->n_segments = ns;
    p->n_pieces = pieces;
    if (launch_splice(*p, stream) != cudaSuccess) return NEXUS_ECUDA;
  }
  return NEXUS_OK;
}

// ------------------------------------------------------------- attention
PFN_cuTensorMapEncodeTiled_v12000 tensor_map_encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* f = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &f, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(f);
    else
      cudaGetLastError();
  });
  return fn;
}

bool encode_4d(CUtensorMap* m, const void* base, const uint64_t dims[4], const uint64_t strides[3],
               const uint32_t box[4], CUtensorMapSwizzle swz) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint32_t elem[4] = {1, 1, 1, 1};
  const CUresult r =
      enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 4, const_cast<void*>(base),
          reinterpret_cast<const cuuint64_t*>(dims), reinterpret_cast<const cuuint64_t*>(strides),
          reinterpret_cast<const cuuint32_t*>(box), elem, CU_TENSOR_MAP_INTERLEAVE_NONE, swz,
          CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

bool encode_2d_sw128(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                     uint32_t box_outer) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {inner * 2};
  const cuuint32_t box[2] = {64, box_outer};
  const cuuint32_t elem[2] = {1, 1};
  const CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims,
                         strides, box, elem, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// int8 [outer][inner] with boxes of 64 bytes x box_outer rows, no swizzle.
bool encode_2d_u8(CUtensorMap* m, const void* base, uint64_t inner, uint64_t outer,
                  uint32_t box_outer) {
  auto enc = tensor_map_encoder();
  if (!enc) return false;
  const cuuint64_t dims[2] = {inner, outer};
  const cuuint64_t strides[1] = {inner};
  const cuuint32_t box[2] = {64, box_outer};
  const cuuint32_t elem[2] = {1, 1};
  const CUresult r = enc(m, CU_TENSOR_MAP_DATA_TYPE_UINT8, 2, const_cast<void*>(base), dims,
                         strides, box, elem, CU_TENSOR_MAP_INTERLEAVE_NONE,
                         CU_TENSOR_MAP_SWIZZLE_NONE, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                         CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// Tool scan: CTAs of 8 warps. Few queries (the latency path, 64 registers, 4
// CTAs per SM): 8 tools per CTA, one per warp, up to four CTAs per SM, so a
// large registry keeps 32 warps of loads in flight on every SM. Batches (one
// CTA per SM by registers): about 64 tools per CTA, at most two waves.
constexpr size_t kSlbPartOffset = 256;
int slb_grid(int32_t n_tools, int32_t n_queries, int32_t* per_out) {
  const bool small = n_queries <= kSlbSmallQueries;
  const int64_t target = small ? 8 : 64;
  int grid = static_cast<int>(std::min<int64_t>((n_tools + target - 1) / target,
                                                (small ? 4 : 2) * num_sms()));
  grid = std::max(grid, 1);
  const int32_t per = (n_tools + grid - 1) / grid;
  if (per_out) *per_out = per;
  return (n_tools + per - 1) / per;
}

struct AttnPlan {
  int32_t total_tiles = 0;
  int32_t n_tok = 0;
  int32_t splits = 1;          // grid and partials: the larger of the two below
  int32_t splits_pair = 1;     // key splits of a pair holding two query tiles
  int32_t splits_single = 1;   // ... holding one query tile
  int32_t kt_max = 0;
};

nexus_status plan_attention(int32_t n_seqs, const int32_t* kv_len, const int32_t* q_len,
                            int32_t n_q_heads, int32_t n_kv_heads, int32_t n_layers_call,
                            int32_t split_kv, AttnPlan* out) {
  if (n_seqs < 1 || n_seqs > kMaxSeqs || !kv_len || !q_len) return NEXUS_EINVAL;
  if (n_kv_heads < 1 || n_q_heads < n_kv_heads || n_q_heads % n_kv_heads != 0) return NEXUS_EINVAL;
  const int32_t group = n_q_heads / n_kv_heads;
  if (group > 128) return NEXUS_EINVAL;
  const int32_t tile_tokens = 128 / group;
  AttnPlan pl;
  int64_t tok = 0, tiles = 0;
  double key_tiles = 0.0;   // key tiles over all CTAs of one KV head (no split)
  int64_t n_pair = 0, n_single = 0;   // pairs holding two / one query tile
  int32_t kt_pair = 0, kt_single = 0; // their largest key-tile counts
  for (int32_t s = 0; s < n_seqs; ++s) {
    if (q_len[s] < 0 || kv_len[s] < q_len[s]) return NEXUS_EINVAL;
    tok += q_len[s];
    const int32_t q_tiles = (q_len[s] + tile_tokens - 1) / tile_tokens;
    const int32_t pairs = (q_tiles + 1) / 2;   // CTAs: pairs of query tiles
    tiles += pairs;
    if (q_len[s] > 0) pl.kt_max = std::max(pl.kt_max, (kv_len[s] + 127) / 128);
    for (int32_t k = 0; k < pairs; ++k) {
      const int64_t last_tok = std::min<int64_t>(q_len[s], (2 * k + 2) * int64_t{tile_tokens}) - 1;
      const int32_t kt = static_cast<int32_t>((kv_len[s] - q_len[s] + last_tok) / 128 + 1);
      key_tiles += static_cast<double>(kt);
      if (2 * k + 1 < q_tiles) { ++n_pair; kt_pair = std::max(kt_pair, kt); }
      else { ++n_single; kt_single = std::max(kt_single, kt); }
    }
  }
  if (tok > 0x7FFFFFFF || tiles > 0x7FFFFFFF) return NEXUS_ERANGE;
  pl.n_tok = static_cast<int32_t>(tok);
  pl.total_tiles = static_cast<int32_t>(tiles);
  if (split_kv < 0) return NEXUS_EINVAL;
  if (split_kv == 0) {
    // Waves of one-CTA-per-SM work against the merge of the partials, in units
    // of one key-tile step of a CTA (~1.66 us). A CTA runs its share of the mean
    // key tiles per CTA plus a fixed start (Q and the first K/V tiles, filling
    // the pipeline) and end (its partial rows) worth about four steps; the merge
    // reads every split's partial rows (~3 us plus 4 MB/us). Calibrated on the
    // c5 suffix (9 splits in one wave, 72 us a layer) and on sweeps of c2 and
    // c3, whose best counts this model picks; a split is taken only where it is
    // predicted to save at least 10 %.
    constexpr double kCtaFixedSteps = 4.0, kStepUs = 1.66, kMergeBytesPerUs = 4.0e6;
    const int64_t ctas = tiles * n_kv_heads * std::max(1, n_layers_call);
    const int sms = num_sms();
    const double rows = static_cast<double>(tok) * n_q_heads * std::max(1, n_layers_call);
    const double mean_tiles = tiles > 0 ? key_tiles / static_cast<double>(tiles) : 0.0;
    auto cost = [&](int s) {
      const double waves = std::ceil(static_cast<double>(ctas) * s / sms);
      double c = waves * (mean_tiles / s + kCtaFixedSteps);
      if (s > 1) c += (3.0 + s * rows * (kHeadDim * 4 + 4) / kMergeBytesPerUs) / kStepUs;
      return c;
    };
    int best = 1;
    if (ctas > 0 && pl.kt_max > 1) {
      const double c1 = cost(1);
      double best_cost = c1;
      for (int s = 2; s <= std::min<int>(kMaxSplits, pl.kt_max); ++s) {
        const double c = cost(s);
        if (c < best_cost - 1e-9) { best_cost = c; best = s; }
      }
      if (best_cost > 0.9 * c1) best = 1;
    }
    pl.splits = pl.splits_pair = pl.splits_single = best;
    // Split, all CTAs in one wave, pairs of both kinds present: a pair holding
    // one query tile runs a key-tile step in about a two-tile pair's time (whose
    // two issuing warps take turns; a one-tile pair has one) and ends ~3 steps
    // sooner (one tile to write back), so the two kinds take their own split
    // counts and end together. Calibrated on the c5 suffix, swept over the
    // counts (two-tile / one-tile pairs, one layer): 10 / 9 57.4 us, 9 / 9 58.6,
    // 11 / 8 60.8, 10 / 8 60.5, 9 / 10 62.1, 8 / 8 63.2.
    const int64_t units = static_cast<int64_t>(n_kv_heads) * std::max(1, n_layers_call);
    bool short_rows = false;   // tile pairs whose rows see fewer than 128 keys: uniform splits
    for (int32_t s = 0; s < n_seqs; ++s)
      short_rows = short_rows || (q_len[s] > 0 && kv_len[s] - q_len[s] < 127);
    if (best > 1 && n_pair > 0 && n_single > 0 && ctas * best <= sms && !short_rows) {
      constexpr double kSingleStep = 1.0, kPairFixed = 6.1, kSingleFixed = 3.2;
      auto span = [&](int sp, int ss) {
        const double tp = std::ceil(static_cast<double>(kt_pair) / sp) + kPairFixed;
        const double ts = kSingleStep * std::ceil(static_cast<double>(kt_single) / ss) + kSingleFixed;
        const int sm = std::max(sp, ss);
        return std::max(tp, ts) + (3.0 + sm * rows * (kHeadDim * 4 + 4) / kMergeBytesPerUs) / kStepUs;
      };
      double best_span = span(best, best);
      for (int sp = 1; sp <= std::min<int>(kMaxSplits, kt_pair); ++sp)
        for (int ss = 1; ss <= std::min<int>(kMaxSplits, kt_single); ++ss) {
          if (units * (n_pair * sp + n_single * ss) > sms) continue;
          const double c = span(sp, ss);
          if (c < best_span - 1e-9) {
            best_span = c;
            pl.splits_pair = sp;
            pl.splits_single = ss;
          }
        }
      pl.splits = std::max(pl.splits_pair, pl.splits_single);
    }
  } else {
    pl.splits = pl.splits_pair = pl.splits_single = std::min(split_kv, kMaxSplits);
  }
  *out = pl;
  return NEXUS_OK;
}

size_t workspace_bytes_for(const AttnPlan& pl, int32_t n_q_heads, int32_t n_layers_call) {
  if (pl.splits <= 1) return 0;
  const size_t rows = static_cast<size_t>(pl.n_tok) * n_q_heads * n_layers_call;
  return static_cast<size_t>(pl.splits) * rows * (kHeadDim * sizeof(float) + sizeof(float));
}

nexus_status attention_impl(const nexus_kv_cache* c, const int32_t* d_pt, int32_t n_rows,
                            int32_t max_pages, int32_t n_seqs, const int32_t* h_rows,
                            const int32_t* kv_len, const int32_t* q_len, const void* q, void* out,
                            float* lse, int32_t n_q_heads, int32_t lb, int32_t le,
                            int32_t split_kv, void* ws, size_t ws_bytes, cudaStream_t stream,
                            float softcap = 0.f) {
  nexus_status st = check_cache(c);
  if (!(softcap >= 0.f) || !std::isfinite(softcap)) return NEXUS_EINVAL;
  if (st != NEXUS_OK) return st;
  if ((st = check_layers(c, lb, le)) != NEXUS_OK) return st;
  if (!d_pt || n_rows < 1 || max_pages < 1 || !q || !out) return NEXUS_EINVAL;
  if (!aligned16(q) || !aligned16(out) || (lse && (reinterpret_cast<uintptr_t>(lse) & 3u)))
    return NEXUS_ELAYOUT;
  AttnPlan pl;
  if ((st = plan_attention(n_seqs, kv_len, q_len, n_q_heads, c->n_kv_heads, le - lb, split_kv,
                           &pl)) != NEXUS_OK)
    return st;
  const int64_t cap = static_cast<int64_t>(max_pages) * kPageSize;
  for (int32_t s = 0; s < n_seqs; ++s) {
    const int32_t row = h_rows ? h_rows[s] : s;
    if (row < 0 || row >= n_rows) return NEXUS_ERANGE;
    if (kv_len[s] > cap) return NEXUS_ERANGE;
  }
  if (pl.n_tok == 0 || le == lb) return NEXUS_OK;
  const size_t need = workspace_bytes_for(pl, n_q_heads, le - lb);
  if (need > 0 && (!ws || ws_bytes < need || !aligned16(ws))) return NEXUS_ENOMEM;

  std::unique_ptr<AttnLaunch> p(new AttnLaunch());
  std::memset(p.get(), 0, sizeof(AttnLaunch));
  const int32_t group = n_q_heads / c->n_kv_heads;
  p->page_tables = d_pt;
  p->out = static_cast<uint16_t*>(out);
  p->lse = lse;
  p->max_pages = max_pages;
  p->n_q_heads = n_q_heads;
  p->n_kv_heads = c->n_kv_heads;
  p->group = group;
  p->tile_tokens = 128 / group;
  p->n_tok = pl.n_tok;
  p->n_pages = static_cast<int32_t>(c->n_pages);
  p->layer_begin = lb;
  p->n_layers_call = le - lb;
  p->n_seqs = n_seqs;
  p->splits = pl.splits;
  p->splits_pair = pl.splits_pair;
  p->splits_single = pl.splits_single;
  p->v_transposed = c->v_transposed;
  p->total_tiles = pl.total_tiles;
  p->scale_log2 = static_cast<float>(1.4426950408889634 / std::sqrt(static_cast<double>(kHeadDim)));
  if (softcap > 0.f) {
    p->softcap_in = static_cast<float>(2.0 * 1.4426950408889634 /
                                       (std::sqrt(static_cast<double>(kHeadDim)) * softcap));
    p->softcap_out = static_cast<float>(1.4426950408889634 * softcap);
  }
  if (pl.splits > 1) {
    const size_t rows = static_cast<size_t>(pl.n_tok) * n_q_heads * (le - lb);
    p->part_o = static_cast<float*>(ws);
    p->part_lse = static_cast<float*>(ws) + static_cast<size_t>(pl.splits) * rows * kHeadDim;
  }
  // Tile pairs whose first query row sees fewer than 128 keys (position below
  // 127) go to a launch of their own (the kernel's short-row instantiation);
  // the rest, usually all but a few pairs, to the plain kernel.
  const int32_t tt = p->tile_tokens;
  std::vector<int32_t> short_pairs(static_cast<size_t>(n_seqs), 0);
  int32_t n_short = 0;
  int32_t off = 0;
  for (int32_t s = 0; s < n_seqs; ++s) {
    p->seq[s].kv_len = kv_len[s];
    p->seq[s].q_len = q_len[s];
    p->seq[s].q_off = off;
    p->seq[s].pt_row = h_rows ? h_rows[s] : s;
    off += q_len[s];
    const int32_t pairs = ((q_len[s] + tt - 1) / tt + 1) / 2;
    const int32_t c = kv_len[s] - q_len[s];   // position of the sequence's first query
    if (pairs > 0 && c < 127)
      short_pairs[s] = std::min(pairs, (127 - c + 2 * tt - 1) / (2 * tt));
    n_short += short_pairs[s];
  }
  std::unique_ptr<AttnLaunch> ps;
  if (n_short > 0) {
    ps.reset(new AttnLaunch(*p));
    ps->short_rows = 1;
    int32_t t = 0;
    for (int32_t s = 0; s < n_seqs; ++s) {
      ps->tile_prefix[s] = t;
      ps->pair0[s] = 0;
      t += short_pairs[s];
    }
    ps->tile_prefix[n_seqs] = t;
    ps->total_tiles = t;
  }
  int32_t tiles = 0;
  for (int32_t s = 0; s < n_seqs; ++s) {
    p->tile_prefix[s] = tiles;
    p->pair0[s] = short_pairs[s];
    tiles += ((q_len[s] + tt - 1) / tt + 1) / 2 - short_pairs[s];
  }
  p->tile_prefix[n_seqs] = tiles;
  p->total_tiles = tiles;
  if (pl.splits > 1 && n_short == 0) {
    // split plans without short-row pairs (per-kind split counts occur only
    // there): the grid enumerates each pair's own (pair, split) CTAs
    int32_t ctas = 0;
    for (int32_t s = 0; s < n_seqs; ++s) {
      p->cta_prefix[s] = ctas;
      const int32_t q_tiles = (q_len[s] + tt - 1) / tt;
      ctas += (q_tiles / 2) * pl.splits_pair + (q_tiles % 2) * pl.splits_single;
    }
    p->cta_prefix[n_seqs] = ctas;
  }

  AttnMaps maps;
  const uint64_t tok_stride = static_cast<uint64_t>(n_q_heads) * kHeadDim * 2;
  {
    const uint64_t dims[4] = {kHeadDim, static_cast<uint64_t>(n_q_heads),
                              static_cast<uint64_t>(pl.n_tok), static_cast<uint64_t>(le - lb)};
    const uint64_t strides[3] = {kHeadDim * 2, tok_stride, tok_stride * pl.n_tok};
    const uint32_t box[4] = {64, static_cast<uint32_t>(group), static_cast<uint32_t>(p->tile_tokens), 1};
    if (!encode_4d(&maps.q, q, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B)) return NEXUS_ECUDA;
  }
  const uint64_t head_bytes = kPageSize * kHeadDim * 2;   // 4 KiB per (page, head)
  const uint64_t gpages = static_cast<uint64_t>(c->n_pages) * c->n_layers;
  {
    const uint64_t dims[4] = {kHeadDim, kPageSize, static_cast<uint64_t>(c->n_kv_heads), gpages};
    const uint64_t strides[3] = {kHeadDim * 2, head_bytes, head_bytes * c->n_kv_heads};
    const uint32_t box[4] = {64, kPageSize, 1, 1};
    const uint32_t box8[4] = {64, kPageSize, 1, 8};   // eight consecutive pages
    if (!encode_4d(&maps.k, c->k_pool, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B) ||
        !encode_4d(&maps.k8, c->k_pool, dims, strides, box8, CU_TENSOR_MAP_SWIZZLE_128B))
      return NEXUS_ECUDA;
    if (!c->v_transposed) {
      if (!encode_4d(&maps.v, c->v_pool, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_128B) ||
          !encode_4d(&maps.v8, c->v_pool, dims, strides, box8, CU_TENSOR_MAP_SWIZZLE_128B))
        return NEXUS_ECUDA;
    }
  }
  if (c->v_transposed) {
    const uint64_t dims[4] = {kPageSize, kHeadDim, static_cast<uint64_t>(c->n_kv_heads), gpages};
    const uint64_t strides[3] = {kPageSize * 2, head_bytes, head_bytes * c->n_kv_heads};
    const uint32_t box[4] = {kPageSize, kHeadDim, 1, 1};
    const uint32_t box8[4] = {kPageSize, kHeadDim, 1, 8};
    if (!encode_4d(&maps.v, c->v_pool, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_32B) ||
        !encode_4d(&maps.v8, c->v_pool, dims, strides, box8, CU_TENSOR_MAP_SWIZZLE_32B))
      return NEXUS_ECUDA;
  }
  if (launch_attention(*p, maps, stream) != cudaSuccess) return NEXUS_ECUDA;
  if (ps && launch_attention(*ps, maps, stream) != cudaSuccess) return NEXUS_ECUDA;
  if (pl.splits > 1 && launch_attn_combine(*p, stream) != cudaSuccess) return NEXUS_ECUDA;
  return NEXUS_OK;
}

}  // namespace

extern "C" {

nexus_status nexus_device_status(nexus_stream stream) {
  unsigned int flag = 0, qkv_timeout = 0, bad_page = 0, slb_timeout = 0, splice_bad = 0;
  if (attention_take_timeout(&flag, static_cast<cudaStream_t>(stream)) != cudaSuccess ||
      qkv_take_status(&qkv_timeout, &bad_page, static_cast<cudaStream_t>(stream)) != cudaSuccess ||
      slb_take_timeout(&slb_timeout, static_cast<cudaStream_t>(stream)) != cudaSuccess ||
      splice_take_status(&splice_bad, static_cast<cudaStream_t>(stream)) != cudaSuccess) {
    cudaGetLastError();
    return NEXUS_ECUDA;
  }
  if (flag || qkv_timeout || slb_timeout) return NEXUS_ETIMEOUT;
  return (bad_page || splice_bad) ? NEXUS_ERANGE : NEXUS_OK;
}

nexus_status nexus_selftest_wait(uint32_t budget_us, nexus_stream stream) {
  if (budget_us < 1 || budget_us > 1000000) return NEXUS_EINVAL;
  return launch_wait_selftest(static_cast<uint64_t>(budget_us) * 1000u,
                              static_cast<cudaStream_t>(stream)) == cudaSuccess
             ? NEXUS_OK
             : NEXUS_ECUDA;
}

nexus_status nexus_splice_kv(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                             const int32_t* h_page_tables, int32_t n_rows, int32_t max_pages,
                             const nexus_block* blocks, int32_t n_blocks,
                             const nexus_splice_segment* segments, int32_t n_segments,
                             int32_t layer_begin, int32_t layer_end, nexus_stream stream) {
  nexus_status st = check_cache(cache);
  if (st != NEXUS_OK) return st;
  if ((st = check_layers(cache, layer_begin, layer_end)) != NEXUS_OK) return st;
  if (n_segments < 0 || n_segments > 4096 || n_blocks < 0 || (n_segments > 0 && !segments) ||
      (n_blocks > 0 && !blocks) || !d_page_tables || n_rows < 1 || max_pages < 1)
    return NEXUS_EINVAL;
  if ((st = validate_segments(cache, h_page_tables, n_rows, max_pages, blocks, n_blocks, segments,
                              n_segments)) != NEXUS_OK)
    return st;
  if (layer_end == layer_begin || n_segments == 0) return NEXUS_OK;
  return launch_segments(cache, d_page_tables, max_pages, blocks, segments, n_segments,
                         layer_begin, layer_end, kOutPool, nullptr, 0,
                         static_cast<cudaStream_t>(stream));
}

nexus_status nexus_rope_rerotate(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                                 const int32_t* h_page_tables, int32_t n_rows, int32_t max_pages,
                                 int32_t row, int32_t pos_begin, int32_t n_tokens, int32_t delta,
                                 int32_t layer_begin, int32_t layer_end, nexus_stream stream) {
  nexus_status st = check_cache(cache);
  if (st != NEXUS_OK) return st;
  if ((st = check_layers(cache, layer_begin, layer_end)) != NEXUS_OK) return st;
  if (!d_page_tables || n_rows < 1 || max_pages < 1) return NEXUS_EINVAL;
  nexus_splice_segment s{NEXUS_SRC_CACHE, row, pos_begin, row, pos_begin, n_tokens, delta,
                         NEXUS_SEG_K_ONLY};
  if ((st = validate_segments(cache, h_page_tables, n_rows, max_pages, nullptr, 0, &s, 1)) !=
      NEXUS_OK)
    return st;
  if (layer_end == layer_begin || n_tokens == 0 || delta == 0) return NEXUS_OK;
  return launch_segments(cache, d_page_tables, max_pages, nullptr, &s, 1, layer_begin, layer_end,
                         kOutPool, nullptr, 0, static_cast<cudaStream_t>(stream));
}

nexus_status nexus_rope_rerotate_f32(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                                     const int32_t* h_page_tables, int32_t n_rows,
                                     int32_t max_pages, int32_t row, int32_t pos_begin,
                                     int32_t n_tokens, int32_t delta, int32_t layer_begin,
                                     int32_t layer_end, float* out_f32, nexus_stream stream) {
  nexus_status st = check_cache(cache);
  if (st != NEXUS_OK) return st;
  if ((st = check_layers(cache, layer_begin, layer_end)) != NEXUS_OK) return st;
  if (!d_page_tables || n_rows < 1 || max_pages < 1 || !out_f32) return NEXUS_EINVAL;
  if (!aligned16(out_f32)) return NEXUS_ELAYOUT;
  nexus_splice_segment s{NEXUS_SRC_CACHE, row, pos_begin, row, pos_begin, n_tokens, delta,
                         NEXUS_SEG_K_ONLY};
  if ((st = validate_segments(cache, h_page_tables, n_rows, max_pages, nullptr, 0, &s, 1)) !=
      NEXUS_OK)
    return st;
  if (layer_end == layer_begin || n_tokens == 0) return NEXUS_OK;
  return launch_segments(cache, d_page_tables, max_pages, nullptr, &s, 1, layer_begin, layer_end,
                         kOutF32, out_f32, pos_begin, static_cast<cudaStream_t>(stream));
}

nexus_status nexus_copy_pages(const nexus_kv_cache* cache, const int32_t* h_src_pages,
                              const int32_t* h_dst_pages, int32_t n, int32_t layer_begin,
                              int32_t layer_end, nexus_stream stream) {
  nexus_status st = check_cache(cache);
  if (st != NEXUS_OK) return st;
  if ((st = check_layers(cache, layer_begin, layer_end)) != NEXUS_OK) return st;
  if (n < 0 || n > kMaxPageCopies || (n > 0 && (!h_src_pages || !h_dst_pages))) return NEXUS_EINVAL;
  std::vector<int32_t> dst(h_dst_pages, h_dst_pages + n);
  for (int32_t i = 0; i < n; ++i)
    if (h_src_pages[i] < 0 || h_src_pages[i] >= cache->n_pages || h_dst_pages[i] < 0 ||
        h_dst_pages[i] >= cache->n_pages)
      return NEXUS_ERANGE;
  std::sort(dst.begin(), dst.end());
  if (std::adjacent_find(dst.begin(), dst.end()) != dst.end()) return NEXUS_EOVERLAP;
  for (int32_t i = 0; i < n; ++i)
    if (std::binary_search(dst.begin(), dst.end(), h_src_pages[i])) return NEXUS_EOVERLAP;
  if (n == 0 || layer_end == layer_begin) return NEXUS_OK;
  std::unique_ptr<PageCopyLaunch> p(new PageCopyLaunch());
  p->k_pool = static_cast<uint16_t*>(cache->k_pool);
  p->v_pool = static_cast<uint16_t*>(cache->v_pool);
  p->n_pages = cache->n_pages;
  p->n_kv_heads = cache->n_kv_heads;
  p->layer_begin = layer_begin;
  p->n_layers_call = layer_end - layer_begin;
  p->n = n;
  std::memcpy(p->src, h_src_pages, sizeof(int32_t) * n);
  std::memcpy(p->dst, h_dst_pages, sizeof(int32_t) * n);
  return launch_page_copy(*p, static_cast<cudaStream_t>(stream)) == cudaSuccess ? NEXUS_OK
                                                                                 : NEXUS_ECUDA;
}

nexus_status nexus_suffix_attention(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                                    int32_t n_rows, int32_t max_pages, int32_t n_seqs,
                                    const int32_t* h_rows, const int32_t* h_kv_len,
                                    const int32_t* h_q_len, const void* q, void* out, float* lse,
                                    int32_t n_q_heads, int32_t layer_begin, int32_t layer_end,
                                    int32_t split_kv, void* workspace, size_t workspace_bytes,
                                    nexus_stream stream) {
  return attention_impl(cache, d_page_tables, n_rows, max_pages, n_seqs, h_rows, h_kv_len, h_q_len,
                        q, out, lse, n_q_heads, layer_begin, layer_end, split_kv, workspace,
                        workspace_bytes, static_cast<cudaStream_t>(stream));
}

nexus_status nexus_suffix_attention_softcap(
    const nexus_kv_cache* cache, const int32_t* d_page_tables, int32_t n_rows, int32_t max_pages,
    int32_t n_seqs, const int32_t* h_rows, const int32_t* h_kv_len, const int32_t* h_q_len,
    const void* q, void* out, float* lse, int32_t n_q_heads, int32_t layer_begin,
    int32_t layer_end, int32_t split_kv, void* workspace, size_t workspace_bytes, float softcap,
    nexus_stream stream) {
  if (!(softcap > 0.f)) return NEXUS_EINVAL;
  return attention_impl(cache, d_page_tables, n_rows, max_pages, n_seqs, h_rows, h_kv_len, h_q_len,
                        q, out, lse, n_q_heads, layer_begin, layer_end, split_kv, workspace,
                        workspace_bytes, static_cast<cudaStream_t>(stream), softcap);
}

nexus_status nexus_reprefill(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                             int32_t n_rows, int32_t max_pages, int32_t n_seqs,
                             const int32_t* h_rows, const int32_t* h_kv_len, const void* q,
                             void* out, float* lse, int32_t n_q_heads, int32_t layer_begin,
                             int32_t layer_end, int32_t split_kv, void* workspace,
                             size_t workspace_bytes, nexus_stream stream) {
  return attention_impl(cache, d_page_tables, n_rows, max_pages, n_seqs, h_rows, h_kv_len, h_kv_len,
                        q, out, lse, n_q_heads, layer_begin, layer_end, split_kv, workspace,
                        workspace_bytes, static_cast<cudaStream_t>(stream));
}

nexus_status nexus_suffix_qkv(const nexus_kv_cache* cache, const int32_t* d_page_tables,
                              const int32_t* h_page_tables, int32_t n_rows, int32_t max_pages,
                              int32_t n_seqs, const int32_t* h_rows, const int32_t* h_kv_len,
                              const int32_t* h_q_len, const void* x, int32_t hidden,
                              const void* w_qkv, const float* b_qkv, int32_t n_q_heads,
                              int32_t layer, void* q_out, nexus_stream stream) {
  nexus_status st = check_cache(cache);
  if (st != NEXUS_OK) return st;
  if (layer < 0 || layer >= cache->n_layers) return NEXUS_ERANGE;
  if (!d_page_tables || n_rows < 1 || max_pages < 1 || !x || !w_qkv || !q_out) return NEXUS_EINVAL;
  if (n_seqs < 1 || n_seqs > kMaxSeqs || !h_kv_len || !h_q_len) return NEXUS_EINVAL;
  if (n_q_heads < 1 || n_q_heads > 256 || hidden < 1) return NEXUS_EINVAL;
  if (hidden % 8 != 0 || !aligned16(x) || !aligned16(w_qkv) || !aligned16(q_out) ||
      (b_qkv && !aligned16(b_qkv)))
    return NEXUS_ELAYOUT;
  const int64_t cap = static_cast<int64_t>(max_pages) * kPageSize;
  int64_t n_tok = 0;
  for (int32_t s = 0; s < n_seqs; ++s) {
    const int32_t row = h_rows ? h_rows[s] : s;
    if (h_q_len[s] < 0 || h_kv_len[s] < h_q_len[s]) return NEXUS_EINVAL;
    if (row < 0 || row >= n_rows || h_kv_len[s] > cap || h_kv_len[s] > (1 << 24))
      return NEXUS_ERANGE;
    n_tok += h_q_len[s];
  }
  const int32_t n_heads = n_q_heads + 2 * cache->n_kv_heads;
  // Up to 64 tokens the launch is bound by the weight read: one-head tiles.
  const bool short_tiles = n_tok <= 64;
  const int64_t n_tiles = short_tiles ? n_heads : (n_heads + 1) / 2;
  const int64_t total = (n_tok + 127) / 128 * n_tiles;
  if (n_tok > 0x7FFFFFFF || total > 0x7FFFFFFF) return NEXUS_ERANGE;
  if (h_page_tables) {
    // Every written slot lies in the pool and no two tokens share one.
    std::vector<int64_t> slots;
    slots.reserve(static_cast<size_t>(n_tok));
    for (int32_t s = 0; s < n_seqs; ++s) {
      const int32_t* pt = h_page_tables + static_cast<int64_t>(h_rows ? h_rows[s] : s) * max_pages;
      for (int32_t pos = h_kv_len[s] - h_q_len[s]; pos < h_kv_len[s]; ++pos) {
        const int32_t page = pt[pos / kPageSize];
        if (page < 0 || page >= cache->n_pages) return NEXUS_ERANGE;
        slots.push_back(static_cast<int64_t>(page) * kPageSize + pos % kPageSize);
      }
    }
    std::sort(slots.begin(), slots.end());
    if (std::adjacent_find(slots.begin(), slots.end()) != slots.end()) return NEXUS_EOVERLAP;
  }
  if (n_tok == 0) return NEXUS_OK;

  std::unique_ptr<QkvLaunch> p(new QkvLaunch());
  std::memset(p.get(), 0, sizeof(QkvLaunch));
  p->page_tables = d_page_tables;
  p->bias = b_qkv;
  p->q_out = static_cast<uint16_t*>(q_out);
  p->k_pool = static_cast<uint16_t*>(cache->k_pool);
  p->v_pool = static_cast<uint16_t*>(cache->v_pool);
  p->n_pages = cache->n_pages;
  p->max_pages = max_pages;
  p->n_q_heads = n_q_heads;
  p->n_kv_heads = cache->n_kv_heads;
  p->n_heads = n_heads;
  p->layer = layer;
  p->v_transposed = cache->v_transposed;
  p->rope_gptj = cache->rope_type == NEXUS_ROPE_GPTJ;
  p->n_tok = static_cast<int32_t>(n_tok);
  p->k_blocks = (hidden + 63) / 64;
  p->n_tiles = static_cast<int32_t>(n_tiles);
  p->m_tiles = static_cast<int32_t>((n_tok + 127) / 128);
  // A band of token tiles and the weight tiles it meets stay in L2: up to 18
  // token tiles (1.25 MiB of rows each at hidden 5120) and, across 152 SMs,
  // about 8 weight tiles (2.5 MiB each) in flight.
  // Bands of 24 token tiles: a sweep at 32768 tokens (6 / 9 / 12 / 18 / 24 / 36 tiles:
  // 1.51 / 1.44 / 1.44 / 1.41 / 1.39 / 1.44 ms) put the optimum here.
  p->group_m = std::min<int32_t>(p->m_tiles, 24);
  p->total_tiles = static_cast<int32_t>(total);
  p->n_seqs = n_seqs;
  p->short_tiles = short_tiles ? 1 : 0;
  // A short re-decode streams the weight through few stages per CTA when each
  // tile's hidden dimension is split over a pair of CTAs (one tile per pair).
  // Each CTA of a pair needs at least one stage (two 64-feature boxes); more
  // than three boxes in all leave each at least one.
  p->pair_split = short_tiles && 2 * n_tiles <= num_sms() && (hidden + 63) / 64 > 3 ? 1 : 0;
  double inv[kHeadDim / 2];
  fill_inv_freq_over_pi(cache, inv);
  for (int i = 0; i < kHeadDim / 2; ++i) {
    p->inv_freq_hi[i] = static_cast<float>(inv[i]);
    p->inv_freq_lo[i] = static_cast<float>(inv[i] - static_cast<double>(p->inv_freq_hi[i]));
  }
  int32_t off = 0;
  for (int32_t s = 0; s < n_seqs; ++s) {
    p->seq[s].kv_len = h_kv_len[s];
    p->seq[s].q_len = h_q_len[s];
    p->seq[s].q_off = off;
    p->seq[s].pt_row = h_rows ? h_rows[s] : s;
    off += h_q_len[s];
  }
  QkvMaps maps;
  if (!encode_2d_sw128(&maps.x, x, static_cast<uint64_t>(hidden), static_cast<uint64_t>(n_tok),
                       short_tiles ? 64 : 128) ||
      !encode_2d_sw128(&maps.w, w_qkv, static_cast<uint64_t>(hidden),
                       static_cast<uint64_t>(n_heads) * kHeadDim, short_tiles ? 128 : 256))
    return NEXUS_ECUDA;
  const int grid = static_cast<int>(std::min<int64_t>(total, num_sms()));
  return launch_qkv(*p, maps, grid, static_cast<cudaStream_t>(stream)) == cudaSuccess ? NEXUS_OK
                                                                                      : NEXUS_ECUDA;
}

size_t nexus_slb_workspace_size(int32_t n_tools) {
  if (n_tools < 1) return 0;
  const int grid = std::max(slb_grid(n_tools, 1, nullptr), slb_grid(n_tools, kSlbMaxQueries, nullptr));
  return kSlbPartOffset + static_cast<size_t>(grid) * kSlbMaxQueries * 2 * (sizeof(float) + sizeof(int32_t));
}

nexus_status nexus_slb_route(const int8_t* d_tools, const float* d_tool_scales, int32_t n_tools,
                             int32_t dim, const int8_t* d_queries, const float* d_query_scales,
                             int32_t n_queries, float tau, int32_t* d_top_idx, float* d_top_score,
                             int32_t* d_route, void* workspace, size_t workspace_bytes,
                             nexus_stream stream) {
  if (!d_tools || !d_tool_scales || n_tools < 1 || n_queries < 0 || !std::isfinite(tau))
    return NEXUS_EINVAL;
  if (n_queries > 0 && (!d_queries || !d_query_scales || !d_top_idx || !d_top_score || !d_route))
    return NEXUS_EINVAL;
  if (dim < 4 || dim > 4096) return NEXUS_EINVAL;
  if (dim % 4 != 0 || !aligned16(d_tools) || (d_queries && !aligned16(d_queries)))
    return NEXUS_ELAYOUT;
  if (reinterpret_cast<uintptr_t>(d_tool_scales) % 4 || reinterpret_cast<uintptr_t>(d_top_idx) % 4 ||
      reinterpret_cast<uintptr_t>(d_top_score) % 4 || reinterpret_cast<uintptr_t>(d_route) % 4 ||
      reinterpret_cast<uintptr_t>(d_query_scales) % 4)
    return NEXUS_ELAYOUT;
  if (n_queries == 0) return NEXUS_OK;
  if (!workspace || !aligned16(workspace) || workspace_bytes < nexus_slb_workspace_size(n_tools))
    return NEXUS_ENOMEM;
  const int grid_max = std::max(slb_grid(n_tools, 1, nullptr),
                                slb_grid(n_tools, kSlbMaxQueries, nullptr));
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  SlbLaunch p;
  p.tools = d_tools;
  p.tool_scales = d_tool_scales;
  p.n_tools = n_tools;
  p.dim = dim;
  p.tau = tau;
  p.counter = reinterpret_cast<unsigned int*>(ws);
  p.part_score = reinterpret_cast<float*>(ws + kSlbPartOffset);
  p.part_idx = reinterpret_cast<int32_t*>(ws + kSlbPartOffset +
                                          static_cast<size_t>(grid_max) * kSlbMaxQueries * 2 * sizeof(float));
  for (int32_t q0 = 0; q0 < n_queries; q0 += kSlbMaxQueries) {
    p.n_queries = std::min(kSlbMaxQueries, n_queries - q0);
    int32_t per = 0;
    int grid = slb_grid(n_tools, p.n_queries, &per);
    p.chunk_tools = 0;
    p.stages = 0;
    if (p.n_queries <= kSlbSmallQueries && n_tools >= kSlbStreamMinTools &&
        aligned16(d_tool_scales)) {
      // Streamed scan: stages of 8 m tools, m the largest power of two (at most
      // 32) with about 8 KiB of codes per warp and stage, halved until two
      // stages and the queries fit a CTA's share of the SM's shared memory
      // (two CTAs per SM); as many stages as fit; contiguous ranges per CTA
      // that are whole stages but the last.
      const int kq = p.n_queries == 1 ? 1 : kSlbSmallQueries;
      const int budget = kSlbStreamSmemPerCta - kq * dim;
      int m = 1;
      while (m < 32 && 2 * m * dim <= 8192) m *= 2;
      while (m > 1 && 2 * 8 * m * (dim + 4) > budget) m /= 2;
      const int T = 8 * m;
      p.chunk_tools = T;
      p.stages = std::min(8, std::max(2, budget / (T * (dim + 4))));
      const int64_t g = std::min<int64_t>((n_tools + T - 1) / T, 2 * num_sms());
      per = static_cast<int32_t>(((n_tools + g - 1) / g + T - 1) / T * T);
      grid = (n_tools + per - 1) / per;
    }
    p.tools_per_cta = per;
    p.queries = d_queries + static_cast<int64_t>(q0) * dim;
    p.query_scales = d_query_scales + q0;
    p.top_idx = d_top_idx + 2 * static_cast<int64_t>(q0);
    p.top_score = d_top_score + 2 * static_cast<int64_t>(q0);
    p.route = d_route + q0;
    if (p.n_queries > kSlbSmallQueries && n_tools >= kSlbStreamMinTools && dim % 64 == 0 &&
        dim <= kSlbTcMaxDim) {
      // A batch over a large registry: the exact bf16 tensor-core scan, one CTA
      // per SM walking tiles of 128 tools.
      CUtensorMap tmap;
      if (!encode_2d_u8(&tmap, d_tools, static_cast<uint64_t>(dim),
                        static_cast<uint64_t>(n_tools), 128))
        return NEXUS_ECUDA;
      grid = static_cast<int>(std::min<int64_t>((n_tools + 127) / 128, num_sms()));
      if (launch_slb_tc(p, tmap, grid, static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return NEXUS_ECUDA;
      continue;
    }
    if (launch_slb(p, grid, static_cast<cudaStream_t>(stream)) != cudaSuccess) return NEXUS_ECUDA;
  }
  return NEXUS_OK;
}

nexus_status nexus_slb_quantize(const float* h_x, int32_t n, int32_t dim, int8_t* h_codes,
                                float* h_scales) {
  if (n < 0 || dim < 1 || (n > 0 && (!h_x || !h_codes || !h_scales))) return NEXUS_EINVAL;
  for (int32_t i = 0; i < n; ++i) {
    const float* x = h_x + static_cast<int64_t>(i) * dim;
    int8_t* c = h_codes + static_cast<int64_t>(i) * dim;
    float amax = 0.f;
    for (int32_t j = 0; j < dim; ++j) {
      if (!std::isfinite(x[j])) return NEXUS_EINVAL;
      amax = std::max(amax, std::fabs(x[j]));
    }
    if (amax == 0.f) {
      std::memset(c, 0, static_cast<size_t>(dim));
      h_scales[i] = 0.f;
      continue;
    }
    const float scale = amax / 127.0f;
    for (int32_t j = 0; j < dim; ++j) {
      const float q = std::nearbyint(x[j] / scale);   // ties to even in the default rounding mode
      c[j] = static_cast<int8_t>(std::min(127.f, std::max(-127.f, q)));
    }
    h_scales[i] = scale;
  }
  return NEXUS_OK;
}

// Page-locked staging memory: fresh anonymous pages registered with the driver.
// Mappings of at least a quarter of the transparent huge page size are rounded
// up to whole huge pages, aligned to them and advised to use them: DMA from
// scattered small pages ran at a few GB/s on Grace hosts, from huge pages at
// the link rate.
static size_t host_base_page() {
  const long pg = sysconf(_SC_PAGESIZE);
  return pg > 0 ? static_cast<size_t>(pg) : 4096;
}

static size_t host_huge_page() {
  static const size_t hp = [] {
    size_t v = 0;
    if (FILE* f = std::fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r")) {
      unsigned long long x = 0;
      if (std::fscanf(f, "%llu", &x) == 1) v = static_cast<size_t>(x);
      std::fclose(f);
    }
    const size_t base = host_base_page();
    return (v >= base && (v & (v - 1)) == 0) ? v : 0;
  }();
  return hp;
}

// Mappings handed out by nexus_host_alloc (address -> length), so that
// nexus_host_free unmaps only what this library mapped, at the length it mapped.
static std::mutex g_host_maps_mu;
static std::map<void*, size_t>& host_maps() {
  static std::map<void*, size_t> m;
  return m;
}

static size_t host_mapping_len(size_t bytes, size_t* align) {
  const size_t hp = host_huge_page();
  const size_t unit = (hp && bytes >= hp / 4) ? hp : host_base_page();
  *align = unit;
  return (bytes + unit - 1) / unit * unit;
}

nexus_status nexus_host_alloc(size_t bytes, void** out) {
  if (!out) return NEXUS_EINVAL;
  *out = nullptr;
  if (bytes == 0 || bytes > (static_cast<size_t>(1) << 48)) return NEXUS_EINVAL;
  size_t align = 0;
  const size_t len = host_mapping_len(bytes, &align);
  const size_t extra = align > host_base_page() ? align : 0;
  void* raw = mmap(nullptr, len + extra, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
  if (raw == MAP_FAILED) return NEXUS_ENOMEM;
  uint8_t* p = static_cast<uint8_t*>(raw);
  if (extra) {
    // keep the aligned [p, p + len) and return the rest
    const uintptr_t a = reinterpret_cast<uintptr_t>(raw);
    p = reinterpret_cast<uint8_t*>((a + align - 1) / align * align);
    const size_t head = static_cast<size_t>(p - static_cast<uint8_t*>(raw));
    if (head) munmap(raw, head);
    if (extra - head) munmap(p + len, extra - head);
#ifdef MADV_HUGEPAGE
    madvise(p, len, MADV_HUGEPAGE);   // advice only; small pages if the kernel declines
#endif
  }
  // Fault every page in (zero-filled) before the driver pins them.
  const size_t base = host_base_page();
  for (size_t off = 0; off < len; off += base) static_cast<volatile uint8_t*>(p)[off] = 0;
  if (extra) {
    // Where the faults fell back to base pages (memory too fragmented at that
    // moment), ask the kernel to collapse the range into huge pages now (Linux
    // 6.1 and later; best effort, an older kernel or a refusal changes nothing).
    constexpr int kMadvCollapse = 25;
    madvise(p, len, kMadvCollapse);
  }
  if (cudaHostRegister(p, len, cudaHostRegisterDefault) != cudaSuccess) {
    cudaGetLastError();
    munmap(p, len);
    return NEXUS_ECUDA;
  }
  {
    std::lock_guard<std::mutex> lock(g_host_maps_mu);
    host_maps()[p] = len;
  }
  *out = p;
  return NEXUS_OK;
}

nexus_status nexus_host_free(void* p, size_t bytes) {
  if (!p) return NEXUS_OK;
  if (bytes == 0) return NEXUS_EINVAL;
  size_t align = 0;
  const size_t len = host_mapping_len(bytes, &align);
  std::lock_guard<std::mutex> lock(g_host_maps_mu);
  auto it = host_maps().find(p);
  if (it == host_maps().end() || it->second != len) return NEXUS_EINVAL;
  if (cudaHostUnregister(p) != cudaSuccess) {
    // Still registered: leave it mapped (and recorded) rather than unmap pages
    // the driver may still reach.
    cudaGetLastError();
    return NEXUS_ECUDA;
  }
  munmap(p, len);
  host_maps().erase(it);
  return NEXUS_OK;
}

size_t nexus_attention_workspace_size(int32_t n_seqs, const int32_t* h_kv_len,
                                      const int32_t* h_q_len, int32_t n_q_heads,
                                      int32_t n_kv_heads, int32_t n_layers_call, int32_t split_kv,
                                      int32_t* splits_out) {
  AttnPlan pl;
  if (plan_attention(n_seqs, h_kv_len, h_q_len, n_q_heads, n_kv_heads, n_layers_call, split_kv,
                     &pl) != NEXUS_OK) {
    if (splits_out) *splits_out = 0;
    return 0;
  }
  if (splits_out) *splits_out = pl.splits;
  return workspace_bytes_for(pl, n_q_heads, n_layers_call);
}

}  // extern "C"
