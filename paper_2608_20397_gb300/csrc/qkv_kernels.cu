// Fresh Q, K, V of the re-decoded suffix tokens (Sec. V-A): the QKV projection
// y = x W^T + b of every invalidated token, RoPE at the token's new position
// for the Q and K heads (Sec. III-B), Q written to its output and K, V written
// into the token's slot of the paged cache (either V layout, Sec. V-B).
//
// Persistent CTAs, one per SM, walk output tiles of 128 tokens x 256 features
// (two heads) in bands of group_m (24) token tiles, the token tile fastest inside a
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
                       B_READY = 2 * kStages + 5,   // CTA pair: the peer's sum of my half is ready
                       B_DONE = 2 * kStages + 6,    // CTA pair: the peer has read my buffer
                       kNumBars = 2 * kStages + 7;
  static constexpr uint32_t OFF_BAR = kStages * kStageBytes;
  static constexpr uint32_t OFF_MISC = OFF_BAR + kNumBars * 8;
  static constexpr uint32_t kSmemBytes = OFF_MISC + 16 + 1024;   // + slack for 1024-byte alignment
  static_assert(kXRows == BM || (kXRows == 64 && kSubBytes >= BM * BK * 2),
                "the A operand's 128 rows must lie inside the sub-stage");
  static_assert(kSubBytes % 1024 == 0 && kABytes % 1024 == 0, "128-byte swizzle atoms");
};
using LongTiles = QkvShape<256, 128, 4, 1>;   // 128 tokens x two heads, 4 stages of 48 KiB
// Up to 64 tokens x one head: 4 stages of two consecutive 64-feature boxes
// (48 KiB), so each weight row is read 256 contiguous bytes at a time and
// several stages are in flight while the products consume one. A hidden size of
// 5120 is 40 such stages, which a CTA pair splits 20 / 20 (three-box stages
// left 14 / 13 with the last one partly past the end: 1.3 % slower; two stages of
// four boxes: 8 % slower; one box per stage, 128 bytes per row and stage: 23 %
// slower even with 9 stages).
using ShortTiles = QkvShape<128, 64, 4, 2>;

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

// Streaming stores (evict first): the outputs are not read again by this
// launch and would otherwise push the weight out of L2.
__device__ __forceinline__ void store_row32(uint16_t* dst, const float (&f)[32]) {
  uint4* d = reinterpret_cast<uint4*>(dst);
#pragma unroll
  for (int i = 0; i < 4; ++i)
    __stcs(d + i, make_uint4(pack_bf16x2(f[8 * i], f[8 * i + 1]), pack_bf16x2(f[8 * i + 2], f[8 * i + 3]),
                             pack_bf16x2(f[8 * i + 4], f[8 * i + 5]), pack_bf16x2(f[8 * i + 6], f[8 * i + 7])));
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

// kPair (short tiles only): a cluster of two CTAs shares each tile. CTA r of
// the pair multiplies the hidden features of the stages [r ? kb_half : 0,
// r ? kb_stages : kb_half) into its own accumulator, so each streams half of
// the weight slice and walks half of the stages. The epilogue is split by
// rotation half: CTA r finishes column half r (NeoX: features [32 r, 32 r + 32)
// and their partners 64 above; GPT-J: [64 r, 64 r + 64)). Each CTA leaves its
// partial sum of the other half in its own shared memory, signals the peer
// (remote mbarrier arrive), adds the peer's partial of its own half read over
// distributed shared memory, and waits until the peer has read its buffer
// before it exits. One tile per pair (the host launches two CTAs per tile).
template <class Sh, bool kPair = false>
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
                B_AEMPTY = Sh::B_AEMPTY, B_FIN = Sh::B_FIN, B_READY = Sh::B_READY,
                B_DONE = Sh::B_DONE;
  // CTA pair: this CTA's rank, its stages [kb0, kb1) and its tile stride
  const uint32_t rank = kPair ? cluster_ctarank() : 0u;
  const int kb_half = (kb_stages + 1) / 2;
  const int kb0 = kPair && rank ? kb_half : 0;
  const int kb1 = kPair && !rank ? kb_half : kb_stages;
  const int t_first = kPair ? static_cast<int>(blockIdx.x >> 1) : static_cast<int>(blockIdx.x);
  const int t_step = kPair ? static_cast<int>(gridDim.x >> 1) : static_cast<int>(gridDim.x);
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
    mbar_init(bar(B_READY), 128);   // one arrival per epilogue thread of the peer
    mbar_init(bar(B_DONE), 128);
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
  // The peer arrives remotely on this CTA's barriers only after both CTAs have
  // initialised theirs.
  if constexpr (kPair) cluster_sync_all();
  const uint32_t tmem = *tmem_slot;
  // Launched with programmatic stream serialization: the setup above overlaps
  // the previous kernel's tail, and no global memory this or an earlier kernel
  // writes is touched before that kernel has ended. The one exception is the
  // producer's first weight rows: the weights are read-only to every kernel of
  // this library, so they are requested before the wait.
  if (warp != kProducerWarp) griddep_wait();
  griddep_launch_dependents();

  if (warp == kProducerWarp) {
    // ------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tmap(&maps.x);
      prefetch_tmap(&maps.w);
      // Every band of token tiles reads the whole weight again: it is kept in L2
      // ahead of the activation rows and the outputs streaming past it.
      const uint64_t w_policy = l2_policy_evict_last();
      // the first tile's first stages: weight rows now (each stage's full
      // barrier expects its whole bytes), activation rows after the wait
      int n_pre = 0;
      if (t_first < p.total_tiles) {
        int mt, nt;
        tile_coords(p, t_first, mt, nt);
        n_pre = min(kStages, kb1 - kb0);
        for (int st = 0; st < n_pre; ++st) {
          const int kb = kb0 + st;
          const uint32_t a = sbase + st * kStageBytes;
          mbar_arrive_expect_tx(bar(B_FULL + st), kStageBytes);
#pragma unroll
          for (int sub = 0; sub < kSub; ++sub)
            tma_load_2d_hint(a + sub * kSubBytes + kABytes, &maps.w, bar(B_FULL + st),
                             (kb * kSub + sub) * BK, nt * BN, w_policy);
        }
      }
      griddep_wait();
      int it = 0;
      bool ok = true;
      for (int t = t_first; t < p.total_tiles && ok; t += t_step) {
        int mt, nt;
        tile_coords(p, t, mt, nt);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const int st = it % kStages;
          if (it >= kStages) {
            ok = mbar_wait(bar(B_EMPTY + st), ((it / kStages) - 1) & 1, kBudgetNs, abort, gabort);
            if (!ok) { record_timeout(abort); break; }
          }
          const uint32_t a = sbase + st * kStageBytes;
          const bool pre = it < n_pre;   // weight rows already requested
          if (!pre) mbar_arrive_expect_tx(bar(B_FULL + st), kStageBytes);
#pragma unroll
          for (int sub = 0; sub < kSub; ++sub) {
            tma_load_2d(a + sub * kSubBytes, &maps.x, bar(B_FULL + st), (kb * kSub + sub) * BK, mt * BM);
            if (!pre)
              tma_load_2d_hint(a + sub * kSubBytes + kABytes, &maps.w, bar(B_FULL + st),
                               (kb * kSub + sub) * BK, nt * BN, w_policy);
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
      for (int t = t_first; t < p.total_tiles && ok; t += t_step, ++acc_it) {
        const int buf = acc_it & 1;
        if (acc_it >= 2) {
          ok = mbar_wait(bar(B_AEMPTY + buf), ((acc_it >> 1) - 1) & 1, kBudgetNs, abort, gabort);
          if (!ok) { record_timeout(abort); break; }
        }
        tc_fence_after();
        const uint32_t d = tmem + buf * BN;
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
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
                       (kb != kb0 || sub != 0 || kk != 0) ? 1u : 0u);
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
    // The token of a row: its sequence, new position and cache slot.
    auto row_token = [&](int mt, int& tok, bool& valid, int& pos, int64_t& page_off) {
      tok = mt * BM + row;
      valid = tok < p.n_tok;
      pos = 0;
      page_off = -1;   // element offset of (layer, page) in a pool
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
    };
    // cos / sin of pairs [32 c, 32 c + 32) at position pf
    auto rope_cs = [&](int c, float pf, float (&cs)[32], float (&sn)[32]) {
#pragma unroll
      for (int j = 0; j < 32; ++j) {
        const float fh = p.inv_freq_hi[c * 32 + j];
        const float ph = pf * fh;
        const float e = fmaf(pf, fh, -ph);
        const float r = ph - 2.f * rintf(0.5f * ph);
        sincospif(r + fmaf(pf, p.inv_freq_lo[c * 32 + j], e), &sn[j], &cs[j]);
      }
    };
    // neox: pair i = (i, i + 64), half c holds columns [32c, 32c+32) and
    // [64+32c, 96+32c); gptj: pair i = (2i, 2i + 1), half c holds [64c, 64c+64)
    auto rotate = [&](float (&fa)[32], float (&fb)[32], const float (&cs)[32], const float (&sn)[32]) {
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
    };
    // One row's half (columns col_a.. and col_b..) of head `head` to its destination.
    auto store_half = [&](int head, int col_a, int col_b, bool valid, int tok, int64_t page_off,
                          int slot, const float (&fa)[32], const float (&fb)[32]) {
      const bool is_v = head >= p.n_q_heads + p.n_kv_heads;
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
    };
    if constexpr (kPair) {
      // One tile (one head, up to 64 tokens) per pair; this CTA finishes half
      // `rank` of it. Everything that does not need the products (the row's
      // token and slot, the rotation, the bias) is done while they run.
      const int t = t_first;
      bool ok = t < p.total_tiles;
      bool peer_read_me = false;
      if (ok) {
        int mt, nt;
        tile_coords(p, t, mt, nt);
        const int head = nt;   // one head per short tile
        const int c = static_cast<int>(rank);
        const int col_a = gptj ? c * 64 : c * 32, col_b = gptj ? c * 64 + 32 : 64 + c * 32;
        const int oc = gptj ? (1 - c) * 64 : (1 - c) * 32;   // the peer's half
        const int ocb = gptj ? oc + 32 : 64 + oc;
        int tok, pos;
        bool valid;
        int64_t page_off;
        row_token(mt, tok, valid, pos, page_off);
        const int slot = pos % kPageSize;
        const bool rot = head < p.n_q_heads + p.n_kv_heads;
        float cs[32], sn[32];
        if (rot && valid) rope_cs(c, static_cast<float>(pos), cs, sn);
        float ba[32], bb[32];
#pragma unroll
        for (int j = 0; j < 32; ++j) ba[j] = bb[j] = 0.f;
        if (p.bias && valid) {
          load_bias(p.bias + head * kHeadDim + col_a, ba);
          load_bias(p.bias + head * kHeadDim + col_b, bb);
        }
        ok = mbar_wait(bar(B_AFULL), 0, kBudgetNs, abort, gabort);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok && lane == 0) record_timeout(abort);
        if (ok) tc_fence_after();
        // The peer's half of this CTA's sums goes to this CTA's buffer (the stage
        // ring, free once every product has completed): 64 token rows x 64
        // float32 columns, 16-byte chunks XOR-swizzled by the row so that a
        // warp's rows fall on different banks.
        const uint32_t mine_buf = sbase;
        if (ok && row < 64) {
          uint32_t ra[32], rb[32];
          tmem_ld32(tmem + lane_base + oc, ra);
          tmem_ld32(tmem + lane_base + ocb, rb);
          tmem_ld_wait();
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            st_shared_v4(mine_buf + row * 256 + ((k ^ (row & 15)) << 4), ra[4 * k], ra[4 * k + 1],
                         ra[4 * k + 2], ra[4 * k + 3]);
            st_shared_v4(mine_buf + row * 256 + (((8 + k) ^ (row & 15)) << 4), rb[4 * k],
                         rb[4 * k + 1], rb[4 * k + 2], rb[4 * k + 3]);
          }
        }
        const uint32_t peer = 1u - rank;
        mbar_arrive_remote(map_to_rank(bar(B_READY), peer));
        peer_read_me = true;
        bool got = ok && mbar_wait_cluster(bar(B_READY), 0, kBudgetNs) && !*abort;
        got = __all_sync(0xffffffffu, got);
        if (ok && !got && lane == 0) record_timeout(abort);
        if (got && row < 64) {
          uint32_t ra[32], rb[32];
          tmem_ld32(tmem + lane_base + col_a, ra);
          tmem_ld32(tmem + lane_base + col_b, rb);
          tmem_ld_wait();
          float fa[32], fb[32];
          const uint32_t pbuf = map_to_rank(mine_buf, peer);
#pragma unroll
          for (int k = 0; k < 8; ++k) {
            const float4 va = ld_cluster_f4(pbuf + row * 256 + ((k ^ (row & 15)) << 4));
            const float4 vb = ld_cluster_f4(pbuf + row * 256 + (((8 + k) ^ (row & 15)) << 4));
            fa[4 * k] = __uint_as_float(ra[4 * k]) + va.x + ba[4 * k];
            fa[4 * k + 1] = __uint_as_float(ra[4 * k + 1]) + va.y + ba[4 * k + 1];
            fa[4 * k + 2] = __uint_as_float(ra[4 * k + 2]) + va.z + ba[4 * k + 2];
            fa[4 * k + 3] = __uint_as_float(ra[4 * k + 3]) + va.w + ba[4 * k + 3];
            fb[4 * k] = __uint_as_float(rb[4 * k]) + vb.x + bb[4 * k];
            fb[4 * k + 1] = __uint_as_float(rb[4 * k + 1]) + vb.y + bb[4 * k + 1];
            fb[4 * k + 2] = __uint_as_float(rb[4 * k + 2]) + vb.z + bb[4 * k + 2];
            fb[4 * k + 3] = __uint_as_float(rb[4 * k + 3]) + vb.w + bb[4 * k + 3];
          }
          // the loads above have returned their values: the peer may let its buffer go
          mbar_arrive_remote(map_to_rank(bar(B_DONE), peer));
          if (rot) rotate(fa, fb, cs, sn);
          store_half(head, col_a, col_b, valid, tok, page_off, slot, fa, fb);
        } else {
          mbar_arrive_remote(map_to_rank(bar(B_DONE), peer));
        }
      }
      // This CTA's buffer stays until the peer has read it (or given up: every
      // wait of the peer before its reads is bounded by 2 s, this one by 6 s).
      if (peer_read_me) mbar_wait_cluster(bar(B_DONE), 0, 3 * kBudgetNs);
    } else {
      int acc_it = 0;
      for (int t = t_first; t < p.total_tiles; t += t_step, ++acc_it) {
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
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, 512);
}

template <class Sh, bool kPair = false>
cudaError_t launch_qkv_as(const QkvLaunch& p, const QkvMaps& maps, int grid, cudaStream_t stream) {
  static_assert(Sh::kSmemBytes <= 227 * 1024, "shared memory budget");
  cudaError_t e = cudaFuncSetAttribute(qkv_kernel<Sh, kPair>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)Sh::kSmemBytes);
  if (e != cudaSuccess) return e;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  attr[1].id = cudaLaunchAttributeClusterDimension;
  attr[1].val.clusterDim.x = 2;   // kPair: one pair of CTAs per tile
  attr[1].val.clusterDim.y = 1;
  attr[1].val.clusterDim.z = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(kPair ? static_cast<unsigned>(2 * p.total_tiles) : static_cast<unsigned>(grid));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = Sh::kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = kPair ? 2 : 1;
  return cudaLaunchKernelEx(&cfg, qkv_kernel<Sh, kPair>, p, maps);
}

}  // namespace

cudaError_t launch_qkv(const QkvLaunch& p, const QkvMaps& maps, int grid, cudaStream_t stream) {
  if (p.total_tiles <= 0 || grid <= 0) return cudaSuccess;
  if (p.short_tiles && p.pair_split) return launch_qkv_as<ShortTiles, true>(p, maps, grid, stream);
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
