// Fresh Q, K, V of the re-decoded suffix tokens (Sec. V-A): the QKV projection
// y = x W^T + b of every invalidated token, RoPE at the token's new position
// for the Q and K heads (Sec. III-B), Q written to its output and K, V written
// into the token's slot of the paged cache (either V layout, Sec. V-B).
//
// Persistent CTAs, one per SM, walk output tiles of 128 tokens x 256 features
// (two heads) in bands of group_m token tiles, the token tile fastest inside a
// band: the tiles in flight at any time share a few weight tiles and the
// band's token rows, which stay in L2, so DRAM sees each weight tile once per
// band rather than once per wave. Up to 64 tokens (a short re-decoded suffix)
// the launch only streams the weight: tiles are one head wide (twice the
// CTAs), only 64 token rows are copied per box (the products' rows 64-127
// belong to no token and are never stored), and a stage holds three boxes of
// consecutive hidden features, so each weight row is read 384 contiguous bytes
// at a time:
//   warp 0     TMA producer: X and W tiles of 64 hidden features per stage,
//              128-byte swizzle, 4-stage ring (48 KiB a stage)
//   warp 1     tcgen05.mma issuer (one lane): 128x256x16 bf16 products into
//              one of two 256-column TMEM accumulators, so the epilogue of a
//              tile overlaps the main loop of the next
//   warps 2-5  epilogue, thread = token row: TMEM -> registers, + bias,
//              rotation of Q and K heads, bf16 stores
// RoPE angles: pos * theta_i / pi with theta_i / pi split into two floats; the
// high product is reduced modulo 2 exactly and the low terms added after it, so
// the reduced angle is good to a float ulp for any position below 2^24.
// Every wait is bounded; on expiry the CTA records a timeout, lets its copies
// and products in flight finish, frees TMEM and exits.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace nexus {

__device__ unsigned int g_qkv_timeout = 0;
__device__ unsigned int g_qkv_bad_page = 0;

namespace {
using namespace ptx;

constexpr int BM = 128;   // token rows of a product
constexpr int BK = 64;    // hidden features per stage
constexpr int kThreads = 192;
constexpr int kProducerWarp = 0;
constexpr int kMmaWarp = 1;
constexpr uint64_t kBudgetNs = 2000000000ull;   // 2 s per wait
constexpr uint64_t kDrainNs = 200000000ull;     // 0.2 s to drain

// Tile shape: kBN output features (kBN / 128 heads), kXRows token rows copied
// per stage, kStages stages. The A operand always spans BM = 128 rows of the
// stage; with kXRows = 64 its rows 64-127 overlap the stage's W tile and
// produce rows of the accumulator that no token owns.
template <int kBN, int kXRows, int kStages, int kSub = 1>
struct QkvShape {
  static constexpr int BN = kBN;
  static constexpr int STAGES = kStages;
  static constexpr int SUB = kSub;   // 64-feature boxes per stage (consecutive columns)
  static constexpr int HEADS = kBN / 128;
  static constexpr uint32_t kABytes = kXRows * BK * 2;      // one x box
  static constexpr uint32_t kBBytes = kBN * BK * 2;         // one W box
  static constexpr uint32_t kSubBytes = kABytes + kBBytes;
  static constexpr uint32_t kStageBytes = kSub * kSubBytes;
  static constexpr int B_FULL = 0, B_EMPTY = kStages, B_AFULL = 2 * kStages,
                       B_AEMPTY = 2 * kStages + 2, B_FIN = 2 * kStages + 4,
                       kNumBars = 2 * kStages + 5;
  static constexpr uint32_t OFF_BAR = kStages * kStageBytes;
  static constexpr uint32_t OFF_MISC = OFF_BAR + kNumBars * 8;
  static constexpr uint32_t kSmemBytes = OFF_MISC + 16 + 1024;   // + slack for 1024-byte alignment
  static_assert(kXRows == BM || (kXRows == 64 && kSubBytes >= BM * BK * 2),
                "the A operand's 128 rows must lie inside the sub-stage");
  static_assert(kSubBytes % 1024 == 0 && kABytes % 1024 == 0, "128-byte swizzle atoms");
};
using LongTiles = QkvShape<256, 128, 4, 1>;   // 128 tokens x two heads, 4 stages of 48 KiB
// Up to 64 tokens x one head: 3 stages of three consecutive 64-feature boxes
// (72 KiB), so each weight row is read 384 contiguous bytes at a time and a
// third stage is in flight while the products consume one (two stages of four
// boxes: 8 % slower; one box per stage, 128 bytes per row and stage: 23 %
// slower even with 9 stages).
using ShortTiles = QkvShape<128, 64, 3, 3>;

__device__ __forceinline__ void record_timeout(volatile int* abort) {
  *abort = 1;
  atomicOr(&g_qkv_timeout, 1u);
}

__device__ __forceinline__ void load_bias(const float* b, float (&f)[32]) {
  const float4* b4 = reinterpret_cast<const float4*>(b);
#pragma unroll
  for (int i = 0; i < 8; ++i) {
    const float4 v = __ldg(b4 + i);
    f[4 * i] += v.x; f[4 * i + 1] += v.y; f[4 * i + 2] += v.z; f[4 * i + 3] += v.w;
  }
}

__device__ __forceinline__ void store_row32(uint16_t* dst, const float (&f)[32]) {
  uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    d[i] = make_uint4(pack_bf16x2(f[8 * i], f[8 * i + 1]), pack_bf16x2(f[8 * i + 2], f[8 * i + 3]),
                      pack_bf16x2(f[8 * i + 4], f[8 * i + 5]), pack_bf16x2(f[8 * i + 6], f[8 * i + 7]));
}

// Column-strided store into a token-innermost V page: feature c at dst[c * 16].
__device__ __forceinline__ void store_col32(uint16_t* dst, const float (&f)[32]) {
#pragma unroll
  for (int i = 0; i < 32; ++i) dst[i * kPageSize] = __bfloat16_as_ushort(__float2bfloat16_rn(f[i]));
}

__device__ __forceinline__ void tile_coords(const QkvLaunch& p, int t, int& mt, int& nt) {
  const int per_band = p.group_m * p.n_tiles;
  const int band = t / per_band;
  const int first = band * p.group_m;
  const int gm = min(p.group_m, p.m_tiles - first);
  const int local = t - band * per_band;
  mt = first + local % gm;
  nt = local / gm;
}

template <class Sh>
__global__ void __launch_bounds__(kThreads, 1)
qkv_kernel(const __grid_constant__ QkvLaunch p, const __grid_constant__ QkvMaps maps) {
  constexpr int BN = Sh::BN;
  constexpr int kStages = Sh::STAGES;
  constexpr uint32_t kABytes = Sh::kABytes;
  constexpr uint32_t kStageBytes = Sh::kStageBytes;
  constexpr int kSub = Sh::SUB;
  constexpr uint32_t kSubBytes = Sh::kSubBytes;
  const int kb_stages = (p.k_blocks + kSub - 1) / kSub;
  constexpr int B_FULL = Sh::B_FULL, B_EMPTY = Sh::B_EMPTY, B_AFULL = Sh::B_AFULL,
                B_AEMPTY = Sh::B_AEMPTY, B_FIN = Sh::B_FIN;
  constexpr uint32_t OFF_BAR = Sh::OFF_BAR, OFF_MISC = Sh::OFF_MISC;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sbase + OFF_BAR + 8u * i; };
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(smem + OFF_MISC);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + OFF_MISC + 4);
  volatile int* never = reinterpret_cast<volatile int*>(smem + OFF_MISC + 8);   // stays 0
  const volatile unsigned int* gabort = &g_qkv_timeout;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;

  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(B_FULL + s), 1);
      mbar_init(bar(B_EMPTY + s), 1);
    }
    for (int b = 0; b < 2; ++b) {
      mbar_init(bar(B_AFULL + b), 1);
      mbar_init(bar(B_AEMPTY + b), 4);   // one arrival per epilogue warp
    }
    mbar_init(bar(B_FIN), 1);
    *abort = 0;
    *never = 0;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    tmem_alloc(sbase + OFF_MISC, 512);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == kProducerWarp) {
    // ------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tmap(&maps.x);
      prefetch_tmap(&maps.w);
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < p.total_tiles && ok; t += gridDim.x) {
        int mt, nt;
        tile_coords(p, t, mt, nt);
        for (int kb = 0; kb < kb_stages; ++kb, ++it) {
          const int st = it % kStages;
          if (it >= kStages) {
            ok = mbar_wait(bar(B_EMPTY + st), ((it / kStages) - 1) & 1, kBudgetNs, abort, gabort);
            if (!ok) { record_timeout(abort); break; }
          }
          const uint32_t a = sbase + st * kStageBytes;
          mbar_arrive_expect_tx(bar(B_FULL + st), kStageBytes);
#pragma unroll
          for (int sub = 0; sub < kSub; ++sub) {
            tma_load_2d(a + sub * kSubBytes, &maps.x, bar(B_FULL + st), (kb * kSub + sub) * BK, mt * BM);
            tma_load_2d(a + sub * kSubBytes + kABytes, &maps.w, bar(B_FULL + st), (kb * kSub + sub) * BK,
                        nt * BN);
          }
        }
      }
      // The last copies issued land before the CTA can exit (at once when the
      // products have consumed them).
      for (int i = max(0, it - kStages); i < it; ++i)
        mbar_wait(bar(B_FULL + i % kStages), (i / kStages) & 1, kDrainNs, never);
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    // ------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(BM, BN, false);
      // Descriptors of stage 0 formed once; a stage and a k-step only add their
      // byte offset / 16 to the start-address field (no carry: shared memory
      // lies below 256 KiB), keeping the issuing thread off the critical path.
      const uint64_t da0 = smem_desc(sbase, 16, 1024, kSwizzle128B);
      const uint64_t db0 = smem_desc(sbase + kABytes, 16, 1024, kSwizzle128B);
      int it = 0, acc_it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < p.total_tiles && ok; t += gridDim.x, ++acc_it) {
        const int buf = acc_it & 1;
        if (acc_it >= 2) {
          ok = mbar_wait(bar(B_AEMPTY + buf), ((acc_it >> 1) - 1) & 1, kBudgetNs, abort, gabort);
          if (!ok) { record_timeout(abort); break; }
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * BN;
        for (int kb = 0; kb < kb_stages; ++kb, ++it) {
          const int st = it % kStages;
          ok = mbar_wait(bar(B_FULL + st), (it / kStages) & 1, kBudgetNs, abort, gabort);
          if (!ok) { record_timeout(abort); break; }
          tc_fence_after();
#pragma unroll
          for (int sub = 0; sub < kSub; ++sub) {
            const uint64_t so = static_cast<uint64_t>((st * kStageBytes + sub * kSubBytes) >> 4);
#pragma unroll
            for (int kk = 0; kk < BK / 16; ++kk)
              mma_bf16(d, da0 + so + (kk * 32 >> 4), db0 + so + (kk * 32 >> 4), idesc,
                       (kb | sub | kk) != 0 ? 1u : 0u);
          }
          mma_commit(bar(B_EMPTY + st));
        }
        if (ok) mma_commit(bar(B_AFULL + buf));
      }
      // Every product issued has completed before TMEM is freed.
      mma_commit(bar(B_FIN));
      mbar_wait(bar(B_FIN), 0, kDrainNs, never);
    }
    __syncwarp();
  } else {
    // ------------------------------------------------------ epilogue
    const int quad = warp & 3;   // TMEM lanes [32 quad, 32 quad + 32)
    const int row = quad * 32 + lane;
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    const bool gptj = p.rope_gptj != 0;
    const int64_t page_elems = (int64_t)p.n_kv_heads * kPageSize * kHeadDim;
    int acc_it = 0;
    for (int t = blockIdx.x; t < p.total_tiles; t += gridDim.x, ++acc_it) {
      int mt, nt;
      tile_coords(p, t, mt, nt);
      const int buf = acc_it & 1;
      bool ok = mbar_wait(bar(B_AFULL + buf), (acc_it >> 1) & 1, kBudgetNs, abort, gabort);
      ok = __all_sync(0xffffffffu, ok);
      if (!ok) { if (lane == 0) record_timeout(abort); break; }
      tc_fence_after();

      // The token of this row: its sequence, new position and cache slot.
      const int tok = mt * BM + row;
      const bool valid = tok < p.n_tok;
      int pos = 0;
      int64_t page_off = -1;   // element offset of (layer, page) in a pool
      if (valid) {
        int lo = 0, hi = p.n_seqs - 1;
        while (lo < hi) {
          const int mid = (lo + hi + 1) >> 1;
          if (p.seq[mid].q_off <= tok) lo = mid; else hi = mid - 1;
        }
        const AttnSeq& s = p.seq[lo];
        pos = s.kv_len - s.q_len + (tok - s.q_off);
        const int32_t page = p.page_tables[(int64_t)s.pt_row * p.max_pages + pos / kPageSize];
        if (page >= 0 && page < p.n_pages)
          page_off = ((int64_t)p.layer * p.n_pages + page) * page_elems;
        else
          atomicOr(&g_qkv_bad_page, 1u);
      }
      const int slot = pos % kPageSize;
      const float pf = static_cast<float>(pos);
      const uint32_t t_acc = tmem + lane_base + buf * BN;
      const bool any_rot = Sh::HEADS * nt < p.n_q_heads + p.n_kv_heads;

#pragma unroll 1
      for (int c = 0; c < 2; ++c) {
        // cos / sin of pairs [32 c, 32 c + 32) at this token's position
        float cs[32], sn[32];
        if (any_rot) {
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const float fh = p.inv_freq_hi[c * 32 + j];
            const float ph = pf * fh;
            const float e = fmaf(pf, fh, -ph);
            const float r = ph - 2.f * rintf(0.5f * ph);
            sincospif(r + fmaf(pf, p.inv_freq_lo[c * 32 + j], e), &sn[j], &cs[j]);
          }
        }
        // neox: pair i = (i, i + 64), chunk c holds columns [32c, 32c+32) and
        // [64+32c, 96+32c); gptj: pair i = (2i, 2i + 1), chunk c holds [64c, 64c+64)
        const int col_a = gptj ? c * 64 : c * 32;
        const int col_b = gptj ? c * 64 + 32 : 64 + c * 32;
#pragma unroll 1
        for (int h = 0; h < Sh::HEADS; ++h) {
          const int head = Sh::HEADS * nt + h;
          if (head >= p.n_heads) break;
          __syncwarp();
          uint32_t ra[32], rb[32];
          tmem_ld32(t_acc + h * kHeadDim + col_a, ra);
          tmem_ld32(t_acc + h * kHeadDim + col_b, rb);
          tmem_ld_wait();
          float fa[32], fb[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            fa[j] = __uint_as_float(ra[j]);
            fb[j] = __uint_as_float(rb[j]);
          }
          if (p.bias) {
            load_bias(p.bias + head * kHeadDim + col_a, fa);
            load_bias(p.bias + head * kHeadDim + col_b, fb);
          }
          const bool is_v = head >= p.n_q_heads + p.n_kv_heads;
          if (!is_v) {
            if (!gptj) {
#pragma unroll
              for (int j = 0; j < 32; ++j) {
                const float x1 = fa[j], x2 = fb[j];
                fa[j] = fmaf(x1, cs[j], -(x2 * sn[j]));
                fb[j] = fmaf(x1, sn[j], x2 * cs[j]);
              }
            } else {
#pragma unroll
              for (int j = 0; j < 16; ++j) {
                float x1 = fa[2 * j], x2 = fa[2 * j + 1];
                fa[2 * j] = fmaf(x1, cs[j], -(x2 * sn[j]));
                fa[2 * j + 1] = fmaf(x1, sn[j], x2 * cs[j]);
                x1 = fb[2 * j]; x2 = fb[2 * j + 1];
                fb[2 * j] = fmaf(x1, cs[16 + j], -(x2 * sn[16 + j]));
                fb[2 * j + 1] = fmaf(x1, sn[16 + j], x2 * cs[16 + j]);
              }
            }
          }
          if (!valid) {
          } else if (head < p.n_q_heads) {
            uint16_t* dst = p.q_out + ((int64_t)tok * p.n_q_heads + head) * kHeadDim;
            store_row32(dst + col_a, fa);
            store_row32(dst + col_b, fb);
          } else if (page_off >= 0) {
            const int kvh = is_v ? head - p.n_q_heads - p.n_kv_heads : head - p.n_q_heads;
            const int64_t head_off = page_off + (int64_t)kvh * kPageSize * kHeadDim;
            if (is_v && p.v_transposed) {
              uint16_t* dst = p.v_pool + head_off + slot;
              store_col32(dst + col_a * kPageSize, fa);
              store_col32(dst + col_b * kPageSize, fb);
            } else {
              uint16_t* dst = (is_v ? p.v_pool : p.k_pool) + head_off + slot * kHeadDim;
              store_row32(dst + col_a, fa);
              store_row32(dst + col_b, fb);
            }
          }
        }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(bar(B_AEMPTY + buf));
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, 512);
}

template <class Sh>
cudaError_t launch_qkv_as(const QkvLaunch& p, const QkvMaps& maps, int grid, cudaStream_t stream) {
  static_assert(Sh::kSmemBytes <= 227 * 1024, "shared memory budget");
  cudaError_t e = cudaFuncSetAttribute(qkv_kernel<Sh>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)Sh::kSmemBytes);
  if (e != cudaSuccess) return e;
  qkv_kernel<Sh><<<(unsigned)grid, kThreads, Sh::kSmemBytes, stream>>>(p, maps);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_qkv(const QkvLaunch& p, const QkvMaps& maps, int grid, cudaStream_t stream) {
  if (p.total_tiles <= 0 || grid <= 0) return cudaSuccess;
  return p.short_tiles ? launch_qkv_as<ShortTiles>(p, maps, grid, stream)
                       : launch_qkv_as<LongTiles>(p, maps, grid, stream);
}

cudaError_t qkv_take_status(unsigned int* timeout, unsigned int* bad_page, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  if ((e = cudaMemcpyFromSymbol(timeout, g_qkv_timeout, sizeof(unsigned int))) != cudaSuccess)
    return e;
  if ((e = cudaMemcpyFromSymbol(bad_page, g_qkv_bad_page, sizeof(unsigned int))) != cudaSuccess)
    return e;
  const unsigned int zero = 0;
  if ((e = cudaMemcpyToSymbol(g_qkv_timeout, &zero, sizeof(unsigned int))) != cudaSuccess) return e;
  return cudaMemcpyToSymbol(g_qkv_bad_page, &zero, sizeof(unsigned int));
}

}  // namespace nexus
