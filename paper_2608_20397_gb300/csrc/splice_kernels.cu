// Splice scatter fused with RoPE delta re-rotation (Sec. III-B reanchoring,
// Sec. V-A splice at the cursor, Sec. V-B transposed V), the in-place
// re-rotation pass, and whole-page copies (Sec. V-D).
//
// Work unit: one CTA moves the rows of one segment that land in one
// destination page, for one layer (at most 16 rows x 8 KiB of K+V). Every K/V
// row is read and written once with 16-byte vector accesses; a warp covers
// four heads of one row (1 KiB contiguous), so both sides are fully coalesced.
// K is rotated pair-wise in float32 with cos/sin of float64-reduced angles
// and stored round-to-nearest-even; delta = 0 moves the bits untouched.
#include <cuda_bf16.h>

#include "internal.h"

namespace nexus {

// Set when a page id read from a device page table lies outside the pool; the
// piece that met it is skipped whole (nothing read or written through it).
__device__ unsigned int g_splice_bad_page = 0;

namespace {

constexpr int kThreads = 256;
constexpr int kItemsPerThread = 4;   // 16 rows x 8 heads x 8 chunk-pairs / 256 threads

__device__ __forceinline__ float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }
__device__ __forceinline__ uint32_t pack2(float lo, float hi) {
  __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);   // .x = lo (low half), .y = hi
  return *reinterpret_cast<uint32_t*>(&v);
}

__device__ __forceinline__ int find_segment(const SpliceLaunch& p, int piece) {
  int lo = 0, hi = p.n_segments - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.seg[mid].piece_begin <= piece) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// Rotates the 8 elements of `lo` (features 8c..8c+7) against the 8 of `hi`
// (features 64+8c..) for NeoX pairs (i, i+64), or rotates the 4 interleaved
// pairs inside each chunk for GPT-J pairs (2i, 2i+1).
__device__ __forceinline__ void rotate_chunks(uint4& lo, uint4& hi, int c, bool gptj,
                                              const float* cs, const float* sn) {
  uint32_t a[4] = {lo.x, lo.y, lo.z, lo.w};
  uint32_t b[4] = {hi.x, hi.y, hi.z, hi.w};
  if (!gptj) {
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      const int i0 = c * 8 + 2 * w;
      const float a0 = bf16_lo(a[w]), a1 = bf16_hi(a[w]);
      const float b0 = bf16_lo(b[w]), b1 = bf16_hi(b[w]);
      const float c0 = cs[i0], s0 = sn[i0], c1 = cs[i0 + 1], s1 = sn[i0 + 1];
      const float ra0 = fmaf(a0, c0, -(b0 * s0)), rb0 = fmaf(a0, s0, b0 * c0);
      const float ra1 = fmaf(a1, c1, -(b1 * s1)), rb1 = fmaf(a1, s1, b1 * c1);
      a[w] = pack2(ra0, ra1);
      b[w] = pack2(rb0, rb1);
    }
  } else {
#pragma unroll
    for (int w = 0; w < 4; ++w) {
      {
        const int i = c * 4 + w;   // pair (2i, 2i+1) inside the low chunk
        const float x = bf16_lo(a[w]), y = bf16_hi(a[w]);
        a[w] = pack2(fmaf(x, cs[i], -(y * sn[i])), fmaf(x, sn[i], y * cs[i]));
      }
      {
        const int i = 32 + c * 4 + w;
        const float x = bf16_lo(b[w]), y = bf16_hi(b[w]);
        b[w] = pack2(fmaf(x, cs[i], -(y * sn[i])), fmaf(x, sn[i], y * cs[i]));
      }
    }
  }
  lo = make_uint4(a[0], a[1], a[2], a[3]);
  hi = make_uint4(b[0], b[1], b[2], b[3]);
}

__device__ __forceinline__ void store_f32_chunk(float* dst, uint4 v) {
  float4 f0 = make_float4(bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y));
  float4 f1 = make_float4(bf16_lo(v.z), bf16_hi(v.z), bf16_lo(v.w), bf16_hi(v.w));
  reinterpret_cast<float4*>(dst)[0] = f0;
  reinterpret_cast<float4*>(dst)[1] = f1;
}

// Float32 (unrounded) variant of rotate_chunks, used only for the verification
// output of the re-rotation.
__device__ __forceinline__ void rotate_chunks_f32(const uint4& lo, const uint4& hi, int c, bool gptj,
                                                  const float* cs, const float* sn, float* out_lo,
                                                  float* out_hi) {
  const uint32_t a[4] = {lo.x, lo.y, lo.z, lo.w};
  const uint32_t b[4] = {hi.x, hi.y, hi.z, hi.w};
#pragma unroll
  for (int w = 0; w < 4; ++w) {
    const float a0 = bf16_lo(a[w]), a1 = bf16_hi(a[w]);
    const float b0 = bf16_lo(b[w]), b1 = bf16_hi(b[w]);
    if (!gptj) {
      const int i0 = c * 8 + 2 * w;
      out_lo[2 * w] = fmaf(a0, cs[i0], -(b0 * sn[i0]));
      out_hi[2 * w] = fmaf(a0, sn[i0], b0 * cs[i0]);
      out_lo[2 * w + 1] = fmaf(a1, cs[i0 + 1], -(b1 * sn[i0 + 1]));
      out_hi[2 * w + 1] = fmaf(a1, sn[i0 + 1], b1 * cs[i0 + 1]);
    } else {
      const int i = c * 4 + w, j = 32 + c * 4 + w;
      out_lo[2 * w] = fmaf(a0, cs[i], -(a1 * sn[i]));
      out_lo[2 * w + 1] = fmaf(a0, sn[i], a1 * cs[i]);
      out_hi[2 * w] = fmaf(b0, cs[j], -(b1 * sn[j]));
      out_hi[2 * w + 1] = fmaf(b0, sn[j], b1 * cs[j]);
    }
  }
}

__global__ void __launch_bounds__(kThreads) splice_kernel(const __grid_constant__ SpliceLaunch p) {
  extern __shared__ __align__(16) uint16_t s_vstage[];   // [16][Hkv][128] when V is transposed
  __shared__ float s_cos[kHeadDim / 2];
  __shared__ float s_sin[kHeadDim / 2];

  const int piece = blockIdx.x % p.n_pieces;
  const int layer_rel = blockIdx.x / p.n_pieces;
  const int layer = p.layer_begin + layer_rel;
  const int si = find_segment(p, piece);
  const DevSegment& sg = p.seg[si];
  const int H = p.n_kv_heads;

  // Destination rows of this piece: [r0, r1) relative to the segment start.
  const int page0 = sg.dst_start / kPageSize;
  const int dpage_idx = page0 + (piece - sg.piece_begin);
  const int r0 = max(sg.dst_start, dpage_idx * kPageSize) - sg.dst_start;
  const int r1 = min(sg.dst_start + sg.n_tokens, (dpage_idx + 1) * kPageSize) - sg.dst_start;
  const int ns = r1 - r0;
  if (ns <= 0) return;
  const int slot0 = (sg.dst_start + r0) % kPageSize;
  const int32_t dpage = p.page_tables[(int64_t)sg.dst_row * p.max_pages + dpage_idx];
  // Every page id this piece goes through (its destination page and, for a
  // cache source, the at most two pages its source rows span) is checked
  // against the pool before any access: the device table may hold ids the host
  // never saw. A bad id skips the piece and is recorded for nexus_device_status.
  {
    bool bad = dpage < 0 || dpage >= p.n_pages;
    if (sg.src_k == nullptr) {
      const int64_t srow = (int64_t)sg.src_row * p.max_pages;
      const int32_t sp0 = p.page_tables[srow + (sg.src_start + r0) / kPageSize];
      const int32_t sp1 = p.page_tables[srow + (sg.src_start + r1 - 1) / kPageSize];
      bad = bad || sp0 < 0 || sp0 >= p.n_pages || sp1 < 0 || sp1 >= p.n_pages;
    }
    if (bad) {
      if (threadIdx.x == 0) atomicOr(&g_splice_bad_page, 1u);
      return;
    }
  }

  const bool rotate = sg.delta != 0;
  if (rotate && threadIdx.x < kHeadDim / 2) {
    // angle / pi = delta * theta_i / pi, reduced exactly to [-1, 1] in float64
    double x = static_cast<double>(sg.delta) * p.inv_freq_over_pi[threadIdx.x];
    x = x - 2.0 * rint(0.5 * x);
    float s, c;
    sincospif(static_cast<float>(x), &s, &c);
    s_cos[threadIdx.x] = c;
    s_sin[threadIdx.x] = s;
  }
  __syncthreads();

  const bool from_block = sg.src_k != nullptr;
  const bool do_v = (sg.flags & NEXUS_SEG_K_ONLY) == 0 && p.out_mode == kOutPool;
  const int64_t page_elems = (int64_t)H * kPageSize * kHeadDim;
  const int items = ns * H * 8;
  // Block rows headed for a token-innermost V cache are loaded with K and staged
  // in shared memory from registers, so their loads overlap K's.
  const bool stage_from_regs = do_v && p.v_transposed && from_block &&
                               items <= kItemsPerThread * kThreads;

  // ---- K (always row-major), and row-major V, through registers
  uint4 klo[kItemsPerThread], khi[kItemsPerThread], vlo[kItemsPerThread], vhi[kItemsPerThread];
  int64_t dst_off[kItemsPerThread];
  int src_pos_of[kItemsPerThread];
#pragma unroll
  for (int u = 0; u < kItemsPerThread; ++u) {
    const int it = threadIdx.x + u * kThreads;
    dst_off[u] = -1;
    if (it >= items) continue;
    const int c = it & 7;
    const int h = (it >> 3) % H;
    const int rl = it / (8 * H);
    const int r = r0 + rl;
    const uint16_t* sk;
    const uint16_t* sv;
    if (from_block) {
      const int64_t off = layer * sg.src_layer_stride +
                          ((int64_t)(sg.src_start + r) * H + h) * kHeadDim;
      sk = sg.src_k + off;
      sv = sg.src_v + off;
    } else {
      const int spos = sg.src_start + r;
      const int32_t spage = p.page_tables[(int64_t)sg.src_row * p.max_pages + spos / kPageSize];
      const int64_t off = ((int64_t)layer * p.n_pages + spage) * page_elems +
                          ((int64_t)h * kPageSize + spos % kPageSize) * kHeadDim;
      sk = p.k_pool + off;
      sv = p.v_pool + off;
    }
    src_pos_of[u] = sg.src_start + r;
    klo[u] = *reinterpret_cast<const uint4*>(sk + c * 8);
    khi[u] = *reinterpret_cast<const uint4*>(sk + 64 + c * 8);
    if ((do_v && !p.v_transposed) || stage_from_regs) {
      vlo[u] = *reinterpret_cast<const uint4*>(sv + c * 8);
      vhi[u] = *reinterpret_cast<const uint4*>(sv + 64 + c * 8);
    }
    const int slot = slot0 + rl;
    dst_off[u] = ((int64_t)layer * p.n_pages + dpage) * page_elems +
                 ((int64_t)h * kPageSize + slot) * kHeadDim + c * 8;
  }
#pragma unroll
  for (int u = 0; u < kItemsPerThread; ++u) {
    if (dst_off[u] < 0) continue;
    const int it = threadIdx.x + u * kThreads;
    const int c = it & 7;
    if (p.out_mode == kOutF32) {
      const int h = (it >> 3) % H;
      const int tok = src_pos_of[u] - p.out_pos_begin;
      float* o = p.out_f32 + (((int64_t)layer_rel * sg.n_tokens + tok) * H + h) * kHeadDim + c * 8;
      if (rotate) {
        float lo[8], hi[8];
        rotate_chunks_f32(klo[u], khi[u], c, p.rope_gptj != 0, s_cos, s_sin, lo, hi);
        reinterpret_cast<float4*>(o)[0] = make_float4(lo[0], lo[1], lo[2], lo[3]);
        reinterpret_cast<float4*>(o)[1] = make_float4(lo[4], lo[5], lo[6], lo[7]);
        reinterpret_cast<float4*>(o + 64)[0] = make_float4(hi[0], hi[1], hi[2], hi[3]);
        reinterpret_cast<float4*>(o + 64)[1] = make_float4(hi[4], hi[5], hi[6], hi[7]);
      } else {
        store_f32_chunk(o, klo[u]);
        store_f32_chunk(o + 64, khi[u]);
      }
      continue;
    }
    if (rotate) rotate_chunks(klo[u], khi[u], c, p.rope_gptj != 0, s_cos, s_sin);
    uint16_t* dk = p.k_pool + dst_off[u];
    *reinterpret_cast<uint4*>(dk) = klo[u];
    *reinterpret_cast<uint4*>(dk + 64) = khi[u];
    if (do_v && !p.v_transposed) {
      uint16_t* dv = p.v_pool + dst_off[u];
      *reinterpret_cast<uint4*>(dv) = vlo[u];
      *reinterpret_cast<uint4*>(dv + 64) = vhi[u];
    } else if (stage_from_regs) {
      const int h = (it >> 3) % H;
      const int rl = it / (8 * H);
      uint16_t* st = s_vstage + (slot0 + rl) * H * kHeadDim + h * kHeadDim + c * 8;
      *reinterpret_cast<uint4*>(st) = vlo[u];
      *reinterpret_cast<uint4*>(st + 64) = vhi[u];
    }
  }
  // Items past kItemsPerThread * kThreads (more than 8 KV heads) take a plain loop.
  for (int it = threadIdx.x + kItemsPerThread * kThreads; it < items; it += kThreads) {
    const int c = it & 7;
    const int h = (it >> 3) % H;
    const int rl = it / (8 * H);
    const int r = r0 + rl;
    const uint16_t* sk;
    const uint16_t* sv;
    if (from_block) {
      const int64_t off = layer * sg.src_layer_stride +
                          ((int64_t)(sg.src_start + r) * H + h) * kHeadDim;
      sk = sg.src_k + off;
      sv = sg.src_v + off;
    } else {
      const int spos = sg.src_start + r;
      const int32_t spage = p.page_tables[(int64_t)sg.src_row * p.max_pages + spos / kPageSize];
      const int64_t off = ((int64_t)layer * p.n_pages + spage) * page_elems +
                          ((int64_t)h * kPageSize + spos % kPageSize) * kHeadDim;
      sk = p.k_pool + off;
      sv = p.v_pool + off;
    }
    uint4 lo = *reinterpret_cast<const uint4*>(sk + c * 8);
    uint4 hi = *reinterpret_cast<const uint4*>(sk + 64 + c * 8);
    if (p.out_mode == kOutF32) {
      const int tok = sg.src_start + r - p.out_pos_begin;
      float* o = p.out_f32 + (((int64_t)layer_rel * sg.n_tokens + tok) * H + h) * kHeadDim + c * 8;
      if (rotate) {
        float fl[8], fh[8];
        rotate_chunks_f32(lo, hi, c, p.rope_gptj != 0, s_cos, s_sin, fl, fh);
        for (int e = 0; e < 8; ++e) { o[e] = fl[e]; o[64 + e] = fh[e]; }
      } else {
        store_f32_chunk(o, lo);
        store_f32_chunk(o + 64, hi);
      }
      continue;
    }
    if (rotate) rotate_chunks(lo, hi, c, p.rope_gptj != 0, s_cos, s_sin);
    const int64_t doff = ((int64_t)layer * p.n_pages + dpage) * page_elems +
                         ((int64_t)h * kPageSize + slot0 + rl) * kHeadDim + c * 8;
    *reinterpret_cast<uint4*>(p.k_pool + doff) = lo;
    *reinterpret_cast<uint4*>(p.k_pool + doff + 64) = hi;
    if (do_v && !p.v_transposed) {
      *reinterpret_cast<uint4*>(p.v_pool + doff) = *reinterpret_cast<const uint4*>(sv + c * 8);
      *reinterpret_cast<uint4*>(p.v_pool + doff + 64) =
          *reinterpret_cast<const uint4*>(sv + 64 + c * 8);
    }
  }

  if (!(do_v && p.v_transposed)) return;

  // ---- token-innermost V: stage [slot][head][d] in shared memory, then write
  // each (head, d) row of 16 slots as 32 contiguous bytes (Sec. V-B).
  const int hd_rows = H * kHeadDim;
  if (!from_block && (sg.src_start + r0) % kPageSize == slot0) {
    // Source and destination slots coincide (the rows moved by a multiple of
    // 16): the piece is one page-to-page copy of token-innermost rows.
    const int32_t spage =
        p.page_tables[(int64_t)sg.src_row * p.max_pages + (sg.src_start + r0) / kPageSize];
    const uint16_t* src = p.v_pool + ((int64_t)layer * p.n_pages + spage) * page_elems;
    uint16_t* dst = p.v_pool + ((int64_t)layer * p.n_pages + dpage) * page_elems;
    if (ns == kPageSize) {
      const int vecs = (int)(page_elems / 8);
      uint4 buf[4];
      for (int i0 = threadIdx.x; i0 < vecs; i0 += 4 * kThreads) {
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (i0 + u * kThreads < vecs) buf[u] = reinterpret_cast<const uint4*>(src)[i0 + u * kThreads];
#pragma unroll
        for (int u = 0; u < 4; ++u)
          if (i0 + u * kThreads < vecs) reinterpret_cast<uint4*>(dst)[i0 + u * kThreads] = buf[u];
      }
    } else {
      for (int hd = threadIdx.x; hd < hd_rows; hd += kThreads)
        for (int s2 = slot0; s2 < slot0 + ns; ++s2)
          dst[(int64_t)hd * kPageSize + s2] = src[(int64_t)hd * kPageSize + s2];
    }
    return;
  }
  if (stage_from_regs) {
    // already staged by the register loop
  } else if (from_block) {
    const int chunks = ns * H * 16;   // 16-byte chunks of the source rows
    for (int it = threadIdx.x; it < chunks; it += kThreads) {
      const int cc = it % (H * 16);
      const int rl = it / (H * 16);
      const int64_t off = layer * sg.src_layer_stride +
                          (int64_t)(sg.src_start + r0 + rl) * H * kHeadDim + cc * 8;
      const uint4 v = *reinterpret_cast<const uint4*>(sg.src_v + off);
      *reinterpret_cast<uint4*>(s_vstage + (slot0 + rl) * hd_rows + cc * 8) = v;
    }
  } else {
    // Source rows span at most two source pages; read each page's 16-slot
    // rows whole and keep the slots this piece needs.
    const int spos0 = sg.src_start + r0;
    const int spos1 = sg.src_start + r1;   // exclusive
    for (int sp = spos0 / kPageSize; sp * kPageSize < spos1; ++sp) {
      const int32_t spage = p.page_tables[(int64_t)sg.src_row * p.max_pages + sp];
      const int lo_pos = max(spos0, sp * kPageSize);
      const int hi_pos = min(spos1, (sp + 1) * kPageSize);
      for (int hd = threadIdx.x; hd < hd_rows; hd += kThreads) {
        const uint16_t* src = p.v_pool + ((int64_t)layer * p.n_pages + spage) * page_elems +
                              (int64_t)hd * kPageSize;
        uint4 w[2];
        w[0] = reinterpret_cast<const uint4*>(src)[0];
        w[1] = reinterpret_cast<const uint4*>(src)[1];
        const uint16_t* e = reinterpret_cast<const uint16_t*>(w);
        for (int pos = lo_pos; pos < hi_pos; ++pos) {
          const int dslot = slot0 + (pos - spos0);
          s_vstage[dslot * hd_rows + hd] = e[pos % kPageSize];
        }
      }
    }
  }
  __syncthreads();
  for (int hd = threadIdx.x; hd < hd_rows; hd += kThreads) {
    uint16_t* dst = p.v_pool + ((int64_t)layer * p.n_pages + dpage) * page_elems +
                    (int64_t)hd * kPageSize;
    if (ns == kPageSize) {
      uint32_t w[kPageSize / 2];
#pragma unroll
      for (int s = 0; s < kPageSize / 2; ++s)
        w[s] = (uint32_t)s_vstage[(2 * s) * hd_rows + hd] |
               ((uint32_t)s_vstage[(2 * s + 1) * hd_rows + hd] << 16);
      reinterpret_cast<uint4*>(dst)[0] = make_uint4(w[0], w[1], w[2], w[3]);
      reinterpret_cast<uint4*>(dst)[1] = make_uint4(w[4], w[5], w[6], w[7]);
    } else {
      for (int s = slot0; s < slot0 + ns; ++s) dst[s] = s_vstage[s * hd_rows + hd];
    }
  }
}

// Whole-page copies (K and V, every layer of the call). One CTA moves two heads
// of one page pair in one layer (16 KiB of K and V in, 16 KiB out), so even a
// single pair spreads over layers x heads / 2 CTAs. The pair list travels in the
// kernel arguments; a short list uses a small argument block, which launches faster.
template <int kCap>
struct PageCopyArgs {
  uint16_t* k_pool;
  uint16_t* v_pool;
  int64_t n_pages;
  int32_t n_kv_heads;
  int32_t layer_begin;
  int32_t n_layers_call;
  int32_t n;
  int32_t src[kCap];
  int32_t dst[kCap];
};

template <int kCap>
__global__ void __launch_bounds__(kThreads) page_copy_kernel(const __grid_constant__ PageCopyArgs<kCap> p) {
  constexpr int kHeadVec = kPageSize * kHeadDim / 8;   // uint4 per head of a page
  const int head_pairs = (p.n_kv_heads + 1) / 2;
  int b = blockIdx.x;
  const int hp = b % head_pairs;
  b /= head_pairs;
  const int pair = b % p.n;
  const int layer = p.layer_begin + b / p.n;
  const int64_t page_vec = (int64_t)p.n_kv_heads * kHeadVec;
  const int64_t so = ((int64_t)layer * p.n_pages + p.src[pair]) * page_vec + hp * 2 * kHeadVec;
  const int64_t d_o = ((int64_t)layer * p.n_pages + p.dst[pair]) * page_vec + hp * 2 * kHeadVec;
  const int nvec = min(2, p.n_kv_heads - 2 * hp) * kHeadVec;
  const uint4* sk = reinterpret_cast<const uint4*>(p.k_pool) + so;
  const uint4* sv = reinterpret_cast<const uint4*>(p.v_pool) + so;
  uint4* dk = reinterpret_cast<uint4*>(p.k_pool) + d_o;
  uint4* dv = reinterpret_cast<uint4*>(p.v_pool) + d_o;
  uint4 a[2], c[2];
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int j = threadIdx.x + u * kThreads;
    if (j < nvec) { a[u] = sk[j]; c[u] = sv[j]; }
  }
#pragma unroll
  for (int u = 0; u < 2; ++u) {
    const int j = threadIdx.x + u * kThreads;
    if (j < nvec) { dk[j] = a[u]; dv[j] = c[u]; }
  }
}

template <int kCap>
cudaError_t launch_page_copy_as(const PageCopyLaunch& p, cudaStream_t stream) {
  PageCopyArgs<kCap> a;
  a.k_pool = p.k_pool;
  a.v_pool = p.v_pool;
  a.n_pages = p.n_pages;
  a.n_kv_heads = p.n_kv_heads;
  a.layer_begin = p.layer_begin;
  a.n_layers_call = p.n_layers_call;
  a.n = p.n;
  for (int i = 0; i < p.n; ++i) {
    a.src[i] = p.src[i];
    a.dst[i] = p.dst[i];
  }
  const int64_t blocks = (int64_t)p.n * p.n_layers_call * ((p.n_kv_heads + 1) / 2);
  if (blocks > 0x7FFFFFFFLL) return cudaErrorInvalidValue;
  page_copy_kernel<kCap><<<(unsigned)blocks, kThreads, 0, stream>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_splice(const SpliceLaunch& p, cudaStream_t stream) {
  if (p.n_pieces <= 0 || p.n_layers_call <= 0) return cudaSuccess;
  const int64_t blocks = (int64_t)p.n_pieces * p.n_layers_call;
  if (blocks > 0x7FFFFFFFLL) return cudaErrorInvalidValue;
  const size_t smem = p.v_transposed ? (size_t)kPageSize * p.n_kv_heads * kHeadDim * 2 : 0;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(splice_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
  }
  splice_kernel<<<(unsigned)blocks, kThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

cudaError_t splice_take_status(unsigned int* bad_page, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(bad_page, g_splice_bad_page, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_splice_bad_page, &zero, sizeof(unsigned int));
}

cudaError_t launch_page_copy(const PageCopyLaunch& p, cudaStream_t stream) {
  if (p.n <= 0 || p.n_layers_call <= 0) return cudaSuccess;
  if (p.n <= 8) return launch_page_copy_as<8>(p, stream);
  return launch_page_copy_as<kMaxPageCopies>(p, stream);
}

}  // namespace nexus
