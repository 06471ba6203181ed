// Causal GQA suffix-redecode / re-prefill attention on sm_103a tensor cores
// (softmax(QK^T / sqrt(d)) V of Sec. III-A over the redecoded suffix of
// Sec. III-C / Sec. V-A), plus the split-KV partial merge.
//
// One CTA owns two 128-row query tiles (A and B) of one KV head. Rows are
// (token, head in the GQA group) pairs, 128 / group tokens x group heads, so
// every K/V tile brought into shared memory serves all query heads that read
// it, twice. Per CTA (352 threads):
//
//   warp 8     TMA producer: both Q tiles once, then K and V tiles of 128 keys
//              (eight 16-token pages each, through the page table) into a
//              two-stage ring; a tile whose eight page ids are consecutive is
//              one copy per 64-column half, any other one copy per page and half
//   warps 9,10 MMA issuers of tile A and tile B (tcgen05.mma, bf16 in, f32
//              accumulate in TMEM), taking turns: S_A(0) S_B(0), then batches
//              PV_A(j) S_A(j+1) | PV_B(j) S_B(j+1), in this order, so one
//              tile's products run while the other tile's softmax works. Each
//              waits for its tile's P of the first 80 keys and the K / V stages
//              (different lanes at once) while the other's batch is queued,
//              queues those keys' P V products, checks that the rest of P has
//              landed, and hands over two products before its own batch ends.
//   warps 0-3  softmax of tile A, warps 4-7 softmax of tile B: thread i of a
//              warpgroup owns TMEM lane i (= tile row i); online softmax in the
//              log2 domain, the running max moved only past 2^8 growth (then O
//              is rescaled in TMEM); P is written back as bf16 over the first 64
//              columns of the tile's own S, in two parts (keys 0-79, then
//              80-127, each released by its own barrier), and read from TMEM by
//              the P V product
//
// TMEM columns: S_A [0,128), S_B [128,256), O_A [256,384), O_B [384,512).
// The S-full barrier of tile X at step j is committed after PV_X(j-1), so it
// also certifies that O_X and the P columns are free. Every wait is bounded;
// on expiry the CTA records a timeout, drains its in-flight copies and MMAs,
// frees TMEM and exits.
#include <cuda_bf16.h>

#include <mutex>
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"

namespace nexus {

__device__ unsigned int g_attn_timeout = 0;

namespace {
using namespace ptx;

constexpr int BM = 128;   // query rows per tile
constexpr int BN = 128;   // keys per tile
constexpr int D = kHeadDim;
constexpr int kStages = 2;
constexpr int kThreads = 352;
constexpr int kProducerWarp = 8;
constexpr int kMmaWarp = 9;      // issues tile A's products (and owns TMEM)
constexpr int kMmaWarpB = 10;    // issues tile B's products
constexpr uint32_t kTileBytes = BM * D * 2;   // 32 KiB
constexpr uint32_t kHalf = 16384;             // one 64-column half of a tile
constexpr uint64_t kBudgetNs = 2000000000ull; // 2 s per wait
constexpr uint64_t kDrainNs = 200000000ull;   // 0.2 s to drain after an abort
constexpr float kRescaleThreshold = 8.0f;     // move the running max only past 2^8 growth
// The softmax releases P of a tile's first kLoKeys keys before the rest, so the
// issuer wakes and queues those P V products while the rest of P is computed.
constexpr int kLoKeys = 80;

constexpr uint32_t OFF_Q = 0;                          // tile A, tile B
constexpr uint32_t OFF_K = OFF_Q + 2 * kTileBytes;
constexpr uint32_t OFF_V = OFF_K + kStages * kTileBytes;
constexpr uint32_t OFF_BAR = OFF_V + kStages * kTileBytes;
enum {
  B_Q = 0,
  B_KF = 1,      // +stage: K tile landed
  B_VF = 3,      // +stage: V tile landed
  B_KE = 5,      // +stage: K tile consumed (every tile's S product done)
  B_VE = 7,      // +stage: V tile consumed (every tile's P V product done)
  B_SF = 9,      // +tile
  B_PF = 11,     // +tile: P of keys [0, kLoKeys) stored
  B_OD = 13,     // +tile
  B_FIN = 15,
  B_VZ = 16,     // last V tile's rows past kv_len are zeroed
  B_HA = 17,     // tile A's issuer has issued its batch (tile B's may issue)
  B_HB = 18,     // tile B's issuer has issued its batch
  B_FIN2 = 19,
  B_PH = 20,     // +tile: P of keys [kLoKeys, 128) stored
  B_PL = 22,     // +tile: the P V products of keys [0, kLoKeys) are done
  kNumBars = 24
};
constexpr uint32_t OFF_MISC = OFF_BAR + kNumBars * 8;
constexpr uint32_t kSmemUsed = OFF_MISC + 16;
constexpr uint32_t kSmemBytes = kSmemUsed + 1024;   // slack for 1024-byte alignment

constexpr uint32_t TM_S = 0;     // + 128 * tile
constexpr uint32_t TM_O = 256;   // + 128 * tile

__device__ __forceinline__ void record_timeout(volatile int* abort) {
  *abort = 1;
  atomicOr(&g_attn_timeout, 1u);
}

struct Work {
  int seq, kv, layer_rel, split;
  int tok0[2], ntok[2], pos0[2];
  bool has_b;
  bool skip;            // a split index past this pair's split count: no work, no writes
  int kt_begin, n_tiles;
};

// kKinds: pairs holding two query tiles and pairs holding one take their own
// split counts (splits_pair / splits_single, a split-KV plan); otherwise every
// pair takes `splits`. Kept apart at compile time: selecting the count per
// pair raised the register count of the whole kernel (166 -> 168) and slowed
// the re-prefill's loops by ~1.5 %.
template <bool kKinds>
__device__ __forceinline__ Work decode_work(const AttnLaunch& p);

// Split plans with per-kind counts: x enumerates exactly the (pair, split)
// CTAs of every sequence, deepest first, so no CTA is launched past its
// pair's split count.
template <>
__device__ __forceinline__ Work decode_work<true>(const AttnLaunch& p) {
  Work w;
  const int rev = p.cta_prefix[p.n_seqs] - 1 - (int)blockIdx.x;
  int lo = 0, hi = p.n_seqs - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.cta_prefix[mid] <= rev) lo = mid; else hi = mid - 1;
  }
  w.seq = lo;
  const AttnSeq& s = p.seq[lo];
  const int q_tiles = (s.q_len + p.tile_tokens - 1) / p.tile_tokens;
  const int local = rev - p.cta_prefix[lo];
  const int full = q_tiles / 2;
  int pair;
  if (local < full * p.splits_pair) {
    pair = local / p.splits_pair;
    w.split = local % p.splits_pair;
  } else {
    pair = full;
    w.split = local - full * p.splits_pair;
  }
  w.kv = blockIdx.y;
  w.layer_rel = blockIdx.z;
  w.has_b = 2 * pair + 1 < q_tiles;
  for (int x = 0; x < 2; ++x) {
    w.tok0[x] = (2 * pair + x) * p.tile_tokens;
    w.ntok[x] = max(0, min(p.tile_tokens, s.q_len - w.tok0[x]));
    w.pos0[x] = s.kv_len - s.q_len + w.tok0[x];
  }
  const int last = w.has_b ? 1 : 0;
  const int pos_last = w.pos0[last] + w.ntok[last] - 1;
  const int kt_total = pos_last / BN + 1;
  // key tiles spread evenly over the pair's own split count (split <= 32 and
  // kt_total <= 2^24 keep the products below 2^30)
  const int s_this = w.has_b ? p.splits_pair : p.splits_single;
  w.skip = false;
  w.kt_begin = w.split * kt_total / s_this;
  w.n_tiles = (w.split + 1) * kt_total / s_this - w.kt_begin;
  return w;
}

template <>
__device__ __forceinline__ Work decode_work<false>(const AttnLaunch& p) {
  constexpr bool kKinds = false;
  Work w;
  const int rev = p.total_tiles - 1 - (int)blockIdx.x;   // deepest query tiles first
  int lo = 0, hi = p.n_seqs - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.tile_prefix[mid] <= rev) lo = mid; else hi = mid - 1;
  }
  w.seq = lo;
  const int pair = rev - p.tile_prefix[lo] + p.pair0[lo];
  w.kv = blockIdx.y;
  w.layer_rel = blockIdx.z / p.splits;
  w.split = blockIdx.z % p.splits;
  const AttnSeq& s = p.seq[lo];
  const int q_tiles = (s.q_len + p.tile_tokens - 1) / p.tile_tokens;
  w.has_b = 2 * pair + 1 < q_tiles;
  for (int x = 0; x < 2; ++x) {
    w.tok0[x] = (2 * pair + x) * p.tile_tokens;
    w.ntok[x] = max(0, min(p.tile_tokens, s.q_len - w.tok0[x]));
    w.pos0[x] = s.kv_len - s.q_len + w.tok0[x];
  }
  const int last = w.has_b ? 1 : 0;
  const int pos_last = w.pos0[last] + w.ntok[last] - 1;
  const int kt_total = pos_last / BN + 1;
  // The pair's key tiles spread evenly over its split count (split <= 32 and
  // kt_total <= 2^24 keep the products below 2^30).
  if constexpr (kKinds) {
    const int s_this = w.has_b ? p.splits_pair : p.splits_single;
    w.skip = w.split >= s_this;
    w.kt_begin = w.split * kt_total / s_this;
    w.n_tiles = w.skip ? 0 : (w.split + 1) * kt_total / s_this - w.kt_begin;
  } else {
    w.skip = false;
    w.kt_begin = w.split * kt_total / p.splits;
    w.n_tiles = (w.split + 1) * kt_total / p.splits - w.kt_begin;
  }
  return w;
}

// Split count of the pair that owns packed token `tok` (the merge needs it per row).
__device__ __forceinline__ int splits_of_token(const AttnLaunch& p, int tok) {
  if (p.splits_pair == p.splits_single) return p.splits_pair;
  int lo = 0, hi = p.n_seqs - 1;   // last sequence starting at or before tok
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (p.seq[mid].q_off <= tok) lo = mid; else hi = mid - 1;
  }
  const AttnSeq& s = p.seq[lo];
  const int pair = (tok - s.q_off) / p.tile_tokens / 2;
  const int q_tiles = (s.q_len + p.tile_tokens - 1) / p.tile_tokens;
  return 2 * pair + 1 < q_tiles ? p.splits_pair : p.splits_single;
}

// Zeroes V rows of keys [r0, 128) of one stage, so cache slots past kv_len
// (whatever bits they hold) contribute exactly 0 to P V.
__device__ __forceinline__ void zero_v_rows(uint8_t* vbuf, int r0, bool vt, int lane) {
  if (!vt) {
    for (int i = lane; i < 2 * (BN - r0) * 8; i += 32) {
      const int half = i / ((BN - r0) * 8);
      const int rem = i % ((BN - r0) * 8);
      const int row = r0 + rem / 8;
      reinterpret_cast<uint4*>(vbuf + half * kHalf + row * 128)[rem % 8] = make_uint4(0, 0, 0, 0);
    }
  } else {
    // eight pages of [128 d][16 keys] with the 32-byte swizzle (16-byte chunk
    // index XOR bit 2 of the row)
    for (int i = lane; i < 8 * D; i += 32) {
      const int pg = i / D, d = i % D;
      const int k0 = pg * 16;
      if (k0 + 16 <= r0) continue;
      uint16_t* row = reinterpret_cast<uint16_t*>(vbuf + pg * 4096 + d * 32);
      for (int s = max(0, r0 - k0); s < 16; ++s) {
        const int chunk = (s >> 3) ^ ((d >> 2) & 1);
        row[chunk * 8 + (s & 7)] = 0;
      }
    }
  }
}

__device__ __forceinline__ float fmax3(float a, float b, float c) {
  float d;
  asm("max.f32 %0, %1, %2, %3;" : "=f"(d) : "f"(a), "f"(b), "f"(c));
  return d;
}

// D[tmem] (+)= A[tmem] * B[smem]: A is read from tensor memory (P, packed
// bf16 pairs along K, row i in lane i).
__device__ __forceinline__ void mma_bf16_ts(uint32_t d_tmem, uint32_t a_tmem, uint64_t b_desc,
                                            uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n"
      " .reg .pred p;\n"
      " setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], [%1], %2, %3, p;\n"
      "}\n" ::"r"(d_tmem),
      "r"(a_tmem), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}

__device__ __forceinline__ void tmem_st4(uint32_t taddr, const uint32_t (&r)[4]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x4.b32 [%0], {%1,%2,%3,%4};" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3])
               : "memory");
}

__device__ __forceinline__ void tmem_st8(uint32_t taddr, const uint32_t (&r)[8]) {
  asm volatile("tcgen05.st.sync.aligned.32x32b.x8.b32 [%0], {%1,%2,%3,%4,%5,%6,%7,%8};" ::"r"(taddr),
               "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]),
               "r"(r[7])
               : "memory");
}

// Packed two-wide float32 arithmetic (one instruction for two lanes of work):
// the softmax shares its SM sub-partitions with the thread issuing the tensor
// core products, so every instruction it saves is an issue slot for that thread.
__device__ __forceinline__ float2 ffma2(float2 a, float2 b, float2 c) {
  float2 d;
  asm("{\n"
      " .reg .b64 ra, rb, rc, rd;\n"
      " mov.b64 ra, {%2, %3};\n"
      " mov.b64 rb, {%4, %5};\n"
      " mov.b64 rc, {%6, %7};\n"
      " fma.rn.f32x2 rd, ra, rb, rc;\n"
      " mov.b64 {%0, %1}, rd;\n"
      "}\n"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y), "f"(c.x), "f"(c.y));
  return d;
}
__device__ __forceinline__ float2 fadd2(float2 a, float2 b) {
  float2 d;
  asm("{\n"
      " .reg .b64 ra, rb, rd;\n"
      " mov.b64 ra, {%2, %3};\n"
      " mov.b64 rb, {%4, %5};\n"
      " add.rn.f32x2 rd, ra, rb;\n"
      " mov.b64 {%0, %1}, rd;\n"
      "}\n"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}

__device__ __forceinline__ float2 fmul2(float2 a, float2 b) {
  float2 d;
  asm("{\n"
      " .reg .b64 ra, rb, rd;\n"
      " mov.b64 ra, {%2, %3};\n"
      " mov.b64 rb, {%4, %5};\n"
      " mul.rn.f32x2 rd, ra, rb;\n"
      " mov.b64 {%0, %1}, rd;\n"
      "}\n"
      : "=f"(d.x), "=f"(d.y)
      : "f"(a.x), "f"(a.y), "f"(b.x), "f"(b.y));
  return d;
}
__device__ __forceinline__ float rcp_approx(float x) {
  float r;
  asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(r) : "f"(x));
  return r;
}

// S = Q K^T over one 128-key tile: 8 products along d, then S-full committed.
// Descriptors come in formed; a k-step adds its byte offset / 16 to the
// start-address field (no carry: shared memory lies below 256 KiB), so a product
// costs one 64-bit add per operand to issue.
__device__ __forceinline__ void issue_s(uint32_t t_s, uint64_t dq, uint64_t dk, uint32_t idesc,
                                        uint32_t s_full) {
#pragma unroll
  for (int kk = 0; kk < D / 16; ++kk) {
    const uint64_t o = static_cast<uint64_t>(((kk >> 2) * kHalf + (kk & 3) * 32) >> 4);
    mma_bf16(t_s, dq + o, dk + o, idesc, kk > 0 ? 1u : 0u);
  }
  mma_commit(s_full);
}

// O += P V over keys [16 kk0, 16 kk1) of a 128-key tile: P from TMEM (16 keys
// = 8 columns per step).
template <int kk0, int kk1>
__device__ __forceinline__ void issue_pv(uint32_t t_o, uint32_t t_s, uint64_t dv, uint64_t v_step,
                                         uint32_t idesc, bool first) {
#pragma unroll
  for (int kk = kk0; kk < kk1; ++kk)
    mma_bf16_ts(t_o, t_s + kk * 8, dv + kk * v_step, idesc, (!first || kk > 0) ? 1u : 0u);
}

// The first P V product of a tile pair with short rows: O = P V over key tile
// 0 with P read twice, as bf16 from columns 0..63 and as its bf16 remainder
// P - bf16(P) from columns 64..127, so O accumulates P at about 16 bits.
__device__ __forceinline__ void issue_pv_rem(uint32_t t_o, uint32_t t_s, uint64_t dv,
                                             uint64_t v_step, uint32_t idesc) {
#pragma unroll
  for (int kk = 0; kk < BN / 16; ++kk)
    mma_bf16_ts(t_o, t_s + kk * 8, dv + kk * v_step, idesc, kk > 0 ? 1u : 0u);
#pragma unroll
  for (int kk = 0; kk < BN / 16; ++kk)
    mma_bf16_ts(t_o, t_s + BN / 2 + kk * 8, dv + kk * v_step, idesc, 1u);
}

// kSoftcap: attention-logit soft-capping (Sec. V-B): the scaled score s becomes
// cap * tanh(s / cap) before the softmax. kShort: the launch covers the tile
// pairs holding rows that see fewer than 128 keys (see short_rows below); the
// host gives all other pairs to the kShort = false kernel, which carries none of
// that code (its presence alone slowed the loops of every step by 1-2 %).
template <bool kSoftcap, bool kShort, bool kKinds>
__global__ void __launch_bounds__(kThreads, 1)
attention_kernel(const __grid_constant__ AttnLaunch p, const __grid_constant__ AttnMaps maps) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sbase + OFF_BAR + 8u * i; };
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(smem + OFF_MISC);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + OFF_MISC + 4);
  volatile int* never = reinterpret_cast<volatile int*>(smem + OFF_MISC + 8);   // stays 0
  const volatile unsigned int* gabort = &g_attn_timeout;

  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const Work w = decode_work<kKinds>(p);
  if (w.skip) return;   // before any barrier, TMEM or global memory use
  const AttnSeq sq = p.seq[w.seq];
  const int G = p.group;
  const int layer = p.layer_begin + w.layer_rel;
  const int n_tiles = w.n_tiles;
  const int n_q = w.has_b ? 2 : 1;
  // Rows that see fewer than 128 keys (positions below 127, all their keys in
  // the sequence's key tile 0) take P at about 16 bits in that tile: bf16
  // rounding of a few large weights would otherwise show in O (up to 2^-9 of
  // |v| per weight). Only a CTA starting at key tile 0 whose first row lies
  // there has such rows; every other CTA runs exactly the plain bf16 path.
  const bool short_rows = kShort && w.kt_begin == 0 && w.pos0[0] < BN - 1;

  // ---- setup: zero the Q rows no TMA box writes, init barriers, alloc TMEM
  {
    const int rows_loaded = G * p.tile_tokens;
    const int per_half = (BM - rows_loaded) * 8;
    for (int i = threadIdx.x; i < 4 * per_half; i += kThreads) {
      const int qh = i / per_half;   // tile * 2 + half
      const int rem = i % per_half;
      reinterpret_cast<uint4*>(smem + OFF_Q + (qh >> 1) * kTileBytes + (qh & 1) * kHalf +
                               (rows_loaded + rem / 8) * 128)[rem % 8] = make_uint4(0, 0, 0, 0);
    }
    fence_proxy_async_smem();
  }
  if (threadIdx.x == 0) {
    mbar_init(bar(B_Q), 1);
    for (int s = 0; s < kStages; ++s) {
      mbar_init(bar(B_KF + s), 1);
      mbar_init(bar(B_VF + s), 1);
      mbar_init(bar(B_KE + s), n_q);   // one commit per issuing warp
      mbar_init(bar(B_VE + s), n_q);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(bar(B_SF + x), 1);
      mbar_init(bar(B_PF + x), 128);
      mbar_init(bar(B_PH + x), 128);
      mbar_init(bar(B_PL + x), 1);
      mbar_init(bar(B_OD + x), 1);
    }
    mbar_init(bar(B_FIN), 1);
    mbar_init(bar(B_FIN2), 1);
    mbar_init(bar(B_HA), 1);
    mbar_init(bar(B_HB), 1);
    mbar_init(bar(B_VZ), 1);
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
  const bool vt = p.v_transposed != 0;
  // Launched with programmatic stream serialization: the setup above (shared
  // memory, barriers, TMEM) overlaps the previous kernel's tail; nothing in
  // global memory is touched before that kernel has completed (the partials a
  // previous merge still reads, the Q / K / V it wrote).
  griddep_wait();
  griddep_launch_dependents();

  if (warp == kProducerWarp) {
    // ------------------------------------------------------ TMA producer
    const int32_t* pt = p.page_tables + (int64_t)sq.pt_row * p.max_pages;
    const int pg_max = (sq.kv_len - 1) / kPageSize;
    int issued = 0, issued_k = 0;
    if (n_tiles > 0) {
      if (lane == 0) {
        prefetch_tmap(&maps.q);
        prefetch_tmap(&maps.k);
        prefetch_tmap(&maps.v);
        prefetch_tmap(&maps.k8);
        prefetch_tmap(&maps.v8);
        mbar_arrive_expect_tx(bar(B_Q), 2u * n_q * G * p.tile_tokens * 128u);
        for (int x = 0; x < n_q; ++x)
          for (int half = 0; half < 2; ++half)
            tma_load_4d(sbase + OFF_Q + x * kTileBytes + half * kHalf, &maps.q, bar(B_Q),
                        half * 64, w.kv * G, sq.q_off + (x ? w.tok0[1] : w.tok0[0]), w.layer_rel);
      }
      // K and V stages are released separately: K_j is free once both S
      // products of tile j are done, an iteration before V_j, so K tiles are
      // fetched a full iteration ahead of their use.
      for (int it = 0; it < n_tiles; ++it) {
        const int st = it & 1;
        const int kt = w.kt_begin + it;
        int page = 0;
        if (lane < 8) page = pt[min(kt * 8 + lane, pg_max)];
        const int gp = layer * p.n_pages + page;
        // Eight consecutive page ids (the clamped ids of a ragged last tile
        // repeat, so it never qualifies): each 64-column half of the tile is one
        // copy of eight pages, which lands in the same rows as eight copies.
        const int gp0 = __shfl_sync(0xffffffffu, gp, 0);
        const bool run8 = __all_sync(0xffffffffu, lane >= 8 || gp == gp0 + lane);
        bool ok = true;
        if (it >= 2) ok = mbar_wait(bar(B_KE + st), ((it >> 1) - 1) & 1, kBudgetNs, abort, gabort);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) { if (lane == 0) record_timeout(abort); break; }
        if (lane == 0) mbar_arrive_expect_tx(bar(B_KF + st), kTileBytes);
        __syncwarp();
        if (run8) {
          if (lane == 0) {
            const uint32_t kdst = sbase + OFF_K + st * kTileBytes;
            tma_load_4d(kdst, &maps.k8, bar(B_KF + st), 0, 0, w.kv, gp0);
            tma_load_4d(kdst + kHalf, &maps.k8, bar(B_KF + st), 64, 0, w.kv, gp0);
          }
        } else if (lane < 8) {
          const uint32_t kdst = sbase + OFF_K + st * kTileBytes + lane * 2048;
          tma_load_4d(kdst, &maps.k, bar(B_KF + st), 0, 0, w.kv, gp);
          tma_load_4d(kdst + kHalf, &maps.k, bar(B_KF + st), 64, 0, w.kv, gp);
        }
        if (it >= 2) ok = mbar_wait(bar(B_VE + st), ((it >> 1) - 1) & 1, kBudgetNs, abort, gabort);
        ok = __all_sync(0xffffffffu, ok);
        if (!ok) { if (lane == 0) record_timeout(abort); issued_k = it + 1; break; }
        if (lane == 0) mbar_arrive_expect_tx(bar(B_VF + st), kTileBytes);
        __syncwarp();
        if (run8) {
          if (lane == 0) {
            const uint32_t vdst = sbase + OFF_V + st * kTileBytes;
            if (!vt) {
              tma_load_4d(vdst, &maps.v8, bar(B_VF + st), 0, 0, w.kv, gp0);
              tma_load_4d(vdst + kHalf, &maps.v8, bar(B_VF + st), 64, 0, w.kv, gp0);
            } else {
              tma_load_4d(vdst, &maps.v8, bar(B_VF + st), 0, 0, w.kv, gp0);
            }
          }
        } else if (lane < 8) {
          const uint32_t vdst = sbase + OFF_V + st * kTileBytes;
          if (!vt) {
            tma_load_4d(vdst + lane * 2048, &maps.v, bar(B_VF + st), 0, 0, w.kv, gp);
            tma_load_4d(vdst + lane * 2048 + kHalf, &maps.v, bar(B_VF + st), 64, 0, w.kv, gp);
          } else {
            tma_load_4d(vdst + lane * 4096, &maps.v, bar(B_VF + st), 0, 0, w.kv, gp);
          }
        }
        issued = it + 1;
        issued_k = it + 1;
        const int key0 = kt * BN;
        if (key0 + BN > sq.kv_len) {
          // The tile holding the last key: cache slots past kv_len may hold any
          // bits, so their V rows are zeroed before any P V product reads them.
          ok = mbar_wait(bar(B_VF + st), (it >> 1) & 1, kBudgetNs, abort, gabort);
          ok = __all_sync(0xffffffffu, ok);
          if (!ok) { if (lane == 0) record_timeout(abort); break; }
          zero_v_rows(smem + OFF_V + st * kTileBytes, sq.kv_len - key0, vt, lane);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) mbar_arrive(bar(B_VZ));
        }
      }
      if (*abort) {
        // Let the copies still in flight land before the CTA exits.
        for (int it = max(0, issued_k - 2); it < issued_k; ++it)
          mbar_wait(bar(B_KF + (it & 1)), (it >> 1) & 1, kDrainNs, never);
        for (int it = max(0, issued - 2); it < issued; ++it)
          mbar_wait(bar(B_VF + (it & 1)), (it >> 1) & 1, kDrainNs, never);
      }
    }
  } else if (warp == kMmaWarp || warp == kMmaWarpB) {
    // ------------------------------------------------------ MMA issuer
    constexpr uint32_t idesc_qk = idesc_bf16_f32(BM, BN, false);
    const uint32_t idesc_pv = idesc_bf16_f32(BM, D, !vt);
    // Shared-memory descriptors are formed once per CTA; a k-step only adds its
    // byte offset / 16 to the start-address field (no carry out of the field:
    // shared memory lies below 256 KiB). Forming descriptors per product made
    // the issuing thread too slow to keep the tensor core fed.
    const uint64_t dq0 = smem_desc(sbase + OFF_Q, 16, 1024, kSwizzle128B);
    const uint64_t dq1 = smem_desc(sbase + OFF_Q + kTileBytes, 16, 1024, kSwizzle128B);
    const uint64_t dk0 = smem_desc(sbase + OFF_K, 16, 1024, kSwizzle128B);
    const uint64_t dk1 = smem_desc(sbase + OFF_K + kTileBytes, 16, 1024, kSwizzle128B);
    // row-major V: MN-major, 64-wide d halves 16 KiB apart (LBO), 8-key groups
    // 1 KiB apart (SBO), 16 keys = 2 KiB per k-step; token-innermost V: K-major
    // pages of [128 d][16 keys], 8-row groups 256 B apart, one 4 KiB page per step
    const uint64_t dv0 = vt ? smem_desc(sbase + OFF_V, 16, 256, kSwizzle32B)
                            : smem_desc(sbase + OFF_V, kHalf, 1024, kSwizzle128B);
    const uint64_t dv1 = vt ? smem_desc(sbase + OFF_V + kTileBytes, 16, 256, kSwizzle32B)
                            : smem_desc(sbase + OFF_V + kTileBytes, kHalf, 1024, kSwizzle128B);
    const uint64_t v_step = vt ? (4096 >> 4) : (2048 >> 4);
    // The whole warp waits on up to four barriers with one try-wait per lane:
    // lane l polls barrier l % 4, and a lane without one (0 = none) polls the Q
    // barrier, complete by then. In the usual case, every barrier already
    // complete, that is one instruction and one vote.
    auto wait4 = [&](uint32_t b0, uint32_t p0, uint32_t b1, uint32_t p1, uint32_t b2, uint32_t p2,
                     uint32_t b3, uint32_t p3) -> bool {
      const int l4 = lane & 3;
      uint32_t br = l4 == 0 ? b0 : l4 == 1 ? b1 : l4 == 2 ? b2 : b3;
      uint32_t par = l4 == 0 ? p0 : l4 == 1 ? p1 : l4 == 2 ? p2 : p3;
      if (br == 0) { br = bar(B_Q); par = 0; }
      bool done = mbar_try_wait(br, par);
      if (__all_sync(0xffffffffu, done)) return true;
      const bool wt = done || mbar_wait(br, par, kBudgetNs, abort, gabort);
      return __all_sync(0xffffffffu, wt);
    };
    // Two issuing warps, one per query tile, in strict alternation: each waits
    // for the first part of its own tile's P (and the K / V stages) and for the
    // other's hand-off while the other's batch is queued, so the tensor pipe
    // sees the single ordered stream PV_A S_A PV_B S_B ... with the waits taken
    // off its path.
    // (One warp issuing both tiles spent ~1200 cycles per batch on its commits,
    // barrier polls and fence while the short product queue ran dry.) The
    // hand-off orders the issue and keeps the two tiles within one batch of each
    // other, which the K / V release barriers (one commit per tile a phase) rely
    // on; every product still waits for its own data through the barriers above.
    const int x = warp == kMmaWarp ? 0 : 1;
    bool ok = true;
    if (n_tiles > 0 && x < n_q) {
      const uint32_t t_s = tmem + TM_S + x * 128, t_o = tmem + TM_O + x * 128;
      const uint64_t dq = x ? dq1 : dq0;
      const uint32_t h_own = bar(x ? B_HB : B_HA), h_other = bar(x ? B_HA : B_HB);
      const bool pair = n_q == 2;
      // tile B's first S follows tile A's (hand-off phase 0)
      ok = wait4(bar(B_Q), 0, bar(B_KF), 0, x ? h_other : 0u, 0, 0, 0);
      if (ok && lane == 0) {
        tc_fence_after();
        issue_s(t_s, dq, dk0, idesc_qk, bar(B_SF + x));
        mma_commit(bar(B_KE + 0));
        if (pair) mbar_arrive(h_own);
      }
      __syncwarp();
      for (int j = 0; ok && j < n_tiles; ++j) {
        const int st = j & 1;
        const int nst = (j + 1) & 1;
        const bool more = j + 1 < n_tiles;
        const bool ragged = (w.kt_begin + j) * BN + BN > sq.kv_len;
        // A's batch j follows B's batch j - 1 (B's hand-off phase j); B's batch j
        // follows A's batch j (A's hand-off phase j + 1).
        ok = wait4(bar(B_PF + x), j & 1, bar(B_VF + st), (j >> 1) & 1,
                   more ? bar(B_KF + nst) : (ragged ? bar(B_VZ) : 0u), more ? ((j + 1) >> 1) & 1 : 0u,
                   pair ? h_other : 0u, x ? (j + 1) & 1 : j & 1);
        if (!ok) break;
        // short rows: key tile 0 also reads the remainder of P, all after the
        // whole of P (the softmax releases both parts at once there)
        bool rem0 = false;
        if constexpr (kShort) rem0 = short_rows && j == 0;
        const uint64_t dv = st ? dv1 : dv0;
        bool got = true;
        if (lane == 0) {
          tc_fence_after();
          if (!rem0) issue_pv<0, kLoKeys / 16>(t_o, t_s, dv, v_step, idesc_pv, j == 0);
          mma_commit(bar(B_PL + x));
          // The rest of P has usually landed while those products were queued:
          // the issuing thread checks in place (a warp-wide wait here stalled
          // the product stream for ~200 cycles and drained the queue).
          got = mbar_test_wait(bar(B_PH + x), j & 1) ||
                mbar_wait(bar(B_PH + x), j & 1, kBudgetNs, abort, gabort);
        }
        if (lane == 0 && got) {
          tc_fence_after();
          if (rem0)
            issue_pv_rem(t_o, t_s, dv, v_step, idesc_pv);
          else
            issue_pv<kLoKeys / 16, BN / 16>(t_o, t_s, dv, v_step, idesc_pv, false);
          // The hand-off comes two products before the batch ends, so that the
          // other issuer's wait ends as the queue runs out (c5 re-prefill per
          // layer, by products left at the hand-off: 0 7.31 ms, 2 7.16-7.20,
          // 4 7.17-7.23, 6 7.27, 8 7.51, 12 8.12); the commits follow it.
          if (more) {
            const uint64_t dk = nst ? dk1 : dk0;
#pragma unroll
            for (int kk = 0; kk < D / 16; ++kk) {
              if (kk == D / 16 - 2 && pair) mbar_arrive(h_own);
              const uint64_t o = static_cast<uint64_t>(((kk >> 2) * kHalf + (kk & 3) * 32) >> 4);
              mma_bf16(t_s, dq + o, dk + o, idesc_qk, kk > 0 ? 1u : 0u);
            }
          } else if (pair) {
            mbar_arrive(h_own);
          }
          mma_commit(bar(B_VE + st));
          if (more) {
            mma_commit(bar(B_SF + x));
            mma_commit(bar(B_KE + nst));
          } else {
            mma_commit(bar(B_OD + x));
          }
        }
        ok = __shfl_sync(0xffffffffu, got ? 1 : 0, 0) != 0;
      }
      if (!ok && lane == 0) record_timeout(abort);
      // Every MMA this thread issued has finished before TMEM is released.
      if (lane == 0) mma_commit(bar(x ? B_FIN2 : B_FIN));
      __syncwarp();
      mbar_wait(bar(x ? B_FIN2 : B_FIN), 0, kDrainNs, never);
    }
  } else {
    // ------------------------------------------------------ softmax warpgroups
    const int x = warp >> 2;                   // query tile of this warpgroup
    const int r = threadIdx.x & 127;           // tile row == TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t t_s = tmem + lane_base + TM_S + x * 128;
    const uint32_t t_o = tmem + lane_base + TM_O + x * 128;
    const int tr = r / G;                      // token within the tile
    const int pos_r = (x ? w.pos0[1] : w.pos0[0]) + tr;
    const int ntok_x = x ? w.ntok[1] : w.ntok[0];
    const int tok0_x = x ? w.tok0[1] : w.tok0[0];
    const bool active = x < n_q && n_tiles > 0;
    const bool row_valid = x < n_q && (r < G * p.tile_tokens) && (tr < ntok_x);
    // log2-domain multiplier of a score (or of its tanh when soft-capped)
    const float sc = kSoftcap ? p.softcap_out : p.scale_log2;
    float m_run = -INFINITY;                   // running max, log2-scaled units
    float l_run = 0.f;
    bool ok = true;
    for (int j = 0; active && j < n_tiles; ++j) {
      bool wt = mbar_wait(bar(B_SF + x), j & 1, kBudgetNs, abort, gabort);
      ok = __all_sync(0xffffffffu, wt);
      if (!ok) break;
      tc_fence_after();
      float s[BN];
      {
        uint32_t v[4][32];
#pragma unroll
        for (int q = 0; q < 4; ++q) tmem_ld32(t_s + q * 32, v[q]);
        tmem_ld_wait();
#pragma unroll
        for (int q = 0; q < 4; ++q)
#pragma unroll
          for (int e = 0; e < 32; ++e) s[q * 32 + e] = __uint_as_float(v[q][e]);
      }
      const int lim = pos_r - (w.kt_begin + j) * BN;   // keys c <= lim are visible
      // Columns [c0, c1) made ready for the exponentials: soft-capped, then
      // masked. The row is prepared in two parts, [0, kLoKeys) first.
      auto prep = [&](auto c0c, auto c1c) {
        constexpr int c0 = decltype(c0c)::value, c1 = decltype(c1c)::value;
        if constexpr (kSoftcap) {
          // tanh(x) = 2 / (2 z) - 1 with 2 z = 1 + u, u = 2^(-2 x log2 e); the
          // argument is clamped at 30 so that u stays finite (and a NaN score of
          // an unused slot, masked below, becomes a finite number). The
          // reciprocals of a group of four z come from one: 1 / z_i = (product
          // of the other three) / (product of all four).
          const float2 nci = make_float2(-p.softcap_in, -p.softcap_in);
          const float2 half = make_float2(0.5f, 0.5f), mone = make_float2(-1.f, -1.f);
#pragma unroll
          for (int c = c0; c < c1; c += 4) {
            float2 a = fmul2(make_float2(s[c], s[c + 1]), nci);
            float2 b = fmul2(make_float2(s[c + 2], s[c + 3]), nci);
            a.x = ex2_approx(fminf(a.x, 30.f));
            a.y = ex2_approx(fminf(a.y, 30.f));
            b.x = ex2_approx(fminf(b.x, 30.f));
            b.y = ex2_approx(fminf(b.y, 30.f));
            const float2 za = ffma2(a, half, half);
            const float2 zb = ffma2(b, half, half);
            const float2 zp = fmul2(za, zb);
            const float r = rcp_approx(zp.x * zp.y);
            const float2 rp = fmul2(make_float2(r, r), make_float2(zp.y, zp.x));
            const float2 ta = ffma2(rp, zb, mone);
            const float2 tb = ffma2(rp, za, mone);
            s[c] = ta.x;
            s[c + 1] = ta.y;
            s[c + 2] = tb.x;
            s[c + 3] = tb.y;
          }
        }
        if (lim < c1 - 1) {
#pragma unroll
          for (int c = c0; c < c1; ++c) s[c] = (c <= lim) ? s[c] : -INFINITY;
        }
      };
      // Exponentials 2^(s sc - m) of columns [16 q0, 16 q1), written to TMEM as
      // bf16 P over the first 64 columns of S; returns their row sum (four pair
      // chains).
      float2 sum[4];
      auto pass = [&](auto q0c, auto q1c, float neg_m) -> float {
        constexpr int q0 = decltype(q0c)::value, q1 = decltype(q1c)::value;
        const float2 sc2 = make_float2(sc, sc);
        const float2 nm2 = make_float2(neg_m, neg_m);
#pragma unroll
        for (int k = 0; k < 4; ++k) sum[k] = make_float2(0.f, 0.f);
#pragma unroll
        for (int q = q0; q < q1; ++q) {
          uint32_t pk[8];
#pragma unroll
          for (int e = 0; e < 16; e += 2) {
            const int c = q * 16 + e;
            float2 ab = ffma2(make_float2(s[c], s[c + 1]), sc2, nm2);
            ab.x = ex2_approx(ab.x);
            ab.y = ex2_approx(ab.y);
            sum[(e >> 1) & 3] = fadd2(sum[(e >> 1) & 3], ab);
            pk[e / 2] = pack_bf16x2(ab.x, ab.y);
          }
          tmem_st8(t_s + q * 8, pk);   // P over the first 64 columns of S
        }
        return ((sum[0].x + sum[0].y) + (sum[1].x + sum[1].y)) +
               ((sum[2].x + sum[2].y) + (sum[3].x + sum[3].y));
      };
      // The same pass over the whole row for short rows' key tile 0, which also
      // writes the bf16 remainder P - bf16(P) over columns 64..127, four columns
      // of each at a time (the score row already holds 128 of the thread's
      // registers).
      auto pass_rem = [&](float neg_m) -> float {
        const float2 sc2 = make_float2(sc, sc);
        const float2 nm2 = make_float2(neg_m, neg_m);
#pragma unroll
        for (int k = 0; k < 4; ++k) sum[k] = make_float2(0.f, 0.f);
#pragma unroll
        for (int q = 0; q < 16; ++q) {
          uint32_t pk[4], pl[4];
#pragma unroll
          for (int e = 0; e < 8; e += 2) {
            const int c = q * 8 + e;
            float2 ab = ffma2(make_float2(s[c], s[c + 1]), sc2, nm2);
            ab.x = ex2_approx(ab.x);
            ab.y = ex2_approx(ab.y);
            sum[(e >> 1) & 3] = fadd2(sum[(e >> 1) & 3], ab);
            pk[e / 2] = pack_bf16x2(ab.x, ab.y);
            // exact differences: bf16(p) keeps p's leading 8 bits
            pl[e / 2] = pack_bf16x2(ab.x - __uint_as_float(pk[e / 2] << 16),
                                    ab.y - __uint_as_float(pk[e / 2] & 0xFFFF0000u));
          }
          tmem_st4(t_s + q * 4, pk);
          tmem_st4(t_s + BN / 2 + q * 4, pl);
        }
        return ((sum[0].x + sum[0].y) + (sum[1].x + sum[1].y)) +
               ((sum[2].x + sum[2].y) + (sum[3].x + sum[3].y));
      };
      // max over columns [c0, 128)
      auto row_max = [&](auto c0c) -> float {
        constexpr int c0 = decltype(c0c)::value;
        float mxa[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) mxa[k] = -INFINITY;
#pragma unroll
        for (int c = c0; c < BN; c += 16)
#pragma unroll
          for (int k = 0; k < 8; ++k) mxa[k] = fmax3(mxa[k], s[c + k], s[c + 8 + k]);
        return fmaxf(fmax3(mxa[0], mxa[1], mxa[2]),
                     fmaxf(fmax3(mxa[3], mxa[4], mxa[5]), fmaxf(mxa[6], mxa[7])));
      };
      // O of this tile's rows scaled by alpha (warps whose rows all keep their
      // max skip it).
      auto rescale_o = [&](float alpha) {
#pragma unroll 1
        for (int q = 0; q < 4; ++q) {
          uint32_t v[32];
          tmem_ld32(t_o + q * 32, v);
          tmem_ld_wait();
#pragma unroll
          for (int e = 0; e < 32; ++e) v[e] = __float_as_uint(__uint_as_float(v[e]) * alpha);
          tmem_st32(t_o + q * 32, v);
        }
      };
      // The running max moves only when a tile's max exceeds it by more than
      // 2^8, which after a row's first tile is rare. So once every row of the
      // warp has a running max, the exponentials are taken with it straight
      // away, part by part: a part's sum below 2^8 proves that none of its
      // exponentials exceeds 2^8, i.e. the max would not have moved for them.
      // P of keys [0, kLoKeys) is released as soon as that holds for them, and
      // the issuer queues their P V products while the rest is computed. If the
      // rest moves the max (its own max is then the row's), the softmax waits
      // for those products, scales O (which then holds them) like any moved max
      // does, and redoes the rest of P with the new max; a warp with a row whose
      // first part already moves it (and every row's first tile) takes the max
      // over the whole row first.
      prep(std::integral_constant<int, 0>{}, std::integral_constant<int, kLoKeys>{});
      const bool have_max = __all_sync(0xffffffffu, m_run != -INFINITY);
      bool fast = false;
      float rs_lo = 0.f;
      if (have_max) {
        rs_lo = pass(std::integral_constant<int, 0>{}, std::integral_constant<int, kLoKeys / 16>{},
                     -m_run);
        fast = !__any_sync(0xffffffffu, !(rs_lo < 256.f));
      }
      if (fast) {
        tmem_st_wait();
        tc_fence_before();
        mbar_arrive(bar(B_PF + x));
        prep(std::integral_constant<int, kLoKeys>{}, std::integral_constant<int, BN>{});
        float rs_hi = pass(std::integral_constant<int, kLoKeys / 16>{},
                           std::integral_constant<int, BN / 16>{}, -m_run);
        float alpha = 1.f;
        if (__any_sync(0xffffffffu, !(rs_lo + rs_hi < 256.f))) {
          const bool wt = mbar_wait(bar(B_PL + x), j & 1, kBudgetNs, abort, gabort);
          ok = __all_sync(0xffffffffu, wt);
          if (!ok) break;
          tc_fence_after();
          const float mxs = row_max(std::integral_constant<int, kLoKeys>{}) * sc;
          const bool move = mxs > m_run + kRescaleThreshold;
          if (move) {
            alpha = ex2_approx(m_run - mxs);
            m_run = mxs;
          }
          if (__any_sync(0xffffffffu, move)) {
            rescale_o(alpha);
            rs_hi = pass(std::integral_constant<int, kLoKeys / 16>{},
                         std::integral_constant<int, BN / 16>{}, -m_run);
          }
        }
        tmem_st_wait();
        l_run = alpha * (l_run + rs_lo) + rs_hi;
        tc_fence_before();
        mbar_arrive(bar(B_PH + x));
      } else {
        prep(std::integral_constant<int, kLoKeys>{}, std::integral_constant<int, BN>{});
        const float mx = row_max(std::integral_constant<int, 0>{});
        const float mxs = mx * sc;
        const bool move = mx > -INFINITY && (m_run == -INFINITY || mxs > m_run + kRescaleThreshold);
        float alpha = 1.f;
        bool rescale = false;
        if (move) {
          if (m_run != -INFINITY) {
            alpha = ex2_approx(m_run - mxs);
            rescale = true;
          }
          m_run = mxs;
        }
        const float neg_m = m_run == -INFINITY ? 0.f : -m_run;
        float rs;
        if constexpr (kShort) {
          if (short_rows && j == 0)
            rs = pass_rem(neg_m);
          else
            rs = pass(std::integral_constant<int, 0>{}, std::integral_constant<int, BN / 16>{}, neg_m);
        } else {
          rs = pass(std::integral_constant<int, 0>{}, std::integral_constant<int, BN / 16>{}, neg_m);
        }
        // PV_x(j-1) is complete: this step's S-full barrier was committed after it.
        if (__any_sync(0xffffffffu, rescale)) rescale_o(alpha);
        tmem_st_wait();
        l_run = l_run * alpha + rs;
        tc_fence_before();
        mbar_arrive(bar(B_PF + x));
        mbar_arrive(bar(B_PH + x));
      }
    }
    if (!ok && r == 0) record_timeout(abort);

    // ---- epilogue: O / l and LSE, 32 columns at a time
    bool have_o = false;
    if (active && ok) {
      bool wt = mbar_wait(bar(B_OD + x), 0, kBudgetNs, abort, gabort);
      have_o = __all_sync(0xffffffffu, wt);
      if (!have_o && r == 0) record_timeout(abort);
      if (have_o) tc_fence_after();
    }
    const bool good = have_o && l_run > 0.f;
    const float inv_l = good ? 1.f / l_run : 0.f;
    const float lse = good ? (m_run + log2f(l_run)) * 0.69314718055994531f : -INFINITY;
    const int tok = sq.q_off + tok0_x + tr;
    const int head = w.kv * G + (r % G);
    const int64_t row = ((int64_t)w.layer_rel * p.n_tok + tok) * p.n_q_heads + head;
    const int64_t rows_per_split = (int64_t)p.n_layers_call * p.n_tok * p.n_q_heads;
    if constexpr (kKinds) {
      // Split plans: the float32 partial rows go through shared memory so that
      // each is written as one coalesced 512-byte store; a thread storing its
      // own row scattered every warp store over 32 rows (half sectors), and a
      // two-tile CTA spent ~6 us on it. Each warp stages its own 32 rows (16 KB,
      // 16-byte chunks XOR-swizzled by the row): tile A in the K ring (free once
      // its last P V product completed: every S product precedes it), tile B in
      // the V ring (free once its own last P V completed).
      if (x < n_q) {
        const int lw = r & 31;
        const uint32_t stage = sbase + (x == 0 ? OFF_K : OFF_V) + (warp & 3) * 16384;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          uint32_t v[32];
          if (have_o) {
            tmem_ld32(t_o + q * 32, v);
            tmem_ld_wait();
          }
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const int chunk = q * 8 + c;
            const float4 f = have_o ? make_float4(__uint_as_float(v[4 * c]) * inv_l,
                                                  __uint_as_float(v[4 * c + 1]) * inv_l,
                                                  __uint_as_float(v[4 * c + 2]) * inv_l,
                                                  __uint_as_float(v[4 * c + 3]) * inv_l)
                                    : make_float4(0.f, 0.f, 0.f, 0.f);
            st_shared_v4(stage + lw * 512 + ((chunk ^ lw) & 31) * 16, __float_as_uint(f.x),
                         __float_as_uint(f.y), __float_as_uint(f.z), __float_as_uint(f.w));
          }
        }
        __syncwarp();
        // row i of the warp: lane i's row index and validity, broadcast
        float* const base = p.part_o + (int64_t)w.split * rows_per_split * D + lane * 4;
        const unsigned valid_mask = __ballot_sync(0xffffffffu, row_valid);
        const uint32_t row_lo = static_cast<uint32_t>(row), row_hi = static_cast<uint32_t>(row >> 32);
#pragma unroll 4
        for (int i = 0; i < 32; ++i) {
          const uint32_t lo = __shfl_sync(0xffffffffu, row_lo, i);
          const uint32_t hi = __shfl_sync(0xffffffffu, row_hi, i);
          if (!((valid_mask >> i) & 1u)) continue;   // the same for the whole warp
          const int64_t row_i = static_cast<int64_t>((static_cast<uint64_t>(hi) << 32) | lo);
          const float4 val = ld_shared_v4f(stage + i * 512 + ((lane ^ i) & 31) * 16);
          __stcg(reinterpret_cast<float4*>(base + row_i * D), val);
        }
        if (row_valid) p.part_lse[(int64_t)w.split * rows_per_split + row] = lse;
      }
    } else {
#pragma unroll
    for (int q = 0; q < 4; ++q) {
      uint32_t v[32];
      if (have_o) {
        tmem_ld32(t_o + q * 32, v);
        tmem_ld_wait();
      }
      if (!row_valid) continue;
      if (p.splits == 1) {
        uint4* dst = reinterpret_cast<uint4*>(p.out + row * D + q * 32);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
          float f[8];
#pragma unroll
          for (int e = 0; e < 8; ++e) f[e] = have_o ? __uint_as_float(v[c * 8 + e]) * inv_l : 0.f;
          dst[c] = make_uint4(pack_bf16x2(f[0], f[1]), pack_bf16x2(f[2], f[3]),
                              pack_bf16x2(f[4], f[5]), pack_bf16x2(f[6], f[7]));
        }
      } else {
        float4* dst = reinterpret_cast<float4*>(
            p.part_o + ((int64_t)w.split * rows_per_split + row) * D + q * 32);
#pragma unroll
        for (int c = 0; c < 8; ++c)
          dst[c] = have_o ? make_float4(__uint_as_float(v[4 * c]) * inv_l,
                                        __uint_as_float(v[4 * c + 1]) * inv_l,
                                        __uint_as_float(v[4 * c + 2]) * inv_l,
                                        __uint_as_float(v[4 * c + 3]) * inv_l)
                          : make_float4(0.f, 0.f, 0.f, 0.f);
      }
    }
    if (row_valid) {
      if (p.splits == 1) {
        if (p.lse) p.lse[row] = lse;
      } else {
        p.part_lse[(int64_t)w.split * rows_per_split + row] = lse;
      }
    }
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == kMmaWarp) tmem_dealloc(tmem, 512);
}

// Merge of split-KV partials: one warp per (layer, token, head) row. Lane s
// holds split s's LSE; the max and the weight sum are warp-shuffle
// reductions, then every lane accumulates its four columns over the splits.
// Every split writes every row it owns (zeros and an LSE of -inf where it saw
// no key), so the first 16 splits' partial rows are loaded together with the
// LSE, before the weights are known: one memory round trip for up to 16 splits.
__global__ void __launch_bounds__(128) combine_kernel(const __grid_constant__ AttnLaunch p) {
  griddep_wait();   // the attention grid's partials are complete and visible
  griddep_launch_dependents();
  const int64_t rows = (int64_t)p.n_layers_call * p.n_tok * p.n_q_heads;
  const int64_t row = (int64_t)blockIdx.x * 4 + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (row >= rows) return;
  const int splits = splits_of_token(p, static_cast<int>((row / p.n_q_heads) % p.n_tok));
  constexpr int kBatch = 16;
  float4 v[kBatch];
  const float l_s = lane < splits ? __ldcg(p.part_lse + (int64_t)lane * rows + row) : -INFINITY;
#pragma unroll
  for (int k = 0; k < kBatch; ++k)
    v[k] = k < splits
               ? __ldcg(reinterpret_cast<const float4*>(p.part_o + ((int64_t)k * rows + row) * D) + lane)
               : make_float4(0.f, 0.f, 0.f, 0.f);
  float mx = l_s;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  const float w = (mx == -INFINITY || l_s == -INFINITY) ? 0.f : expf(l_s - mx);
  float wsum = w;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) wsum += __shfl_xor_sync(0xffffffffu, wsum, o);
  float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
  for (int s0 = 0; s0 < splits; s0 += kBatch) {
    if (s0 > 0) {
#pragma unroll
      for (int k = 0; k < kBatch; ++k)
        v[k] = s0 + k < splits
                   ? __ldcg(reinterpret_cast<const float4*>(p.part_o + ((int64_t)(s0 + k) * rows + row) * D) + lane)
                   : make_float4(0.f, 0.f, 0.f, 0.f);
    }
#pragma unroll
    for (int k = 0; k < kBatch; ++k) {
      const float ws = __shfl_sync(0xffffffffu, w, (s0 + k) & 31);
      if (s0 + k < splits && ws != 0.f) {
        acc.x += ws * v[k].x; acc.y += ws * v[k].y; acc.z += ws * v[k].z; acc.w += ws * v[k].w;
      }
    }
  }
  const float inv = wsum > 0.f ? 1.f / wsum : 0.f;
  uint2 outv = make_uint2(pack_bf16x2(acc.x * inv, acc.y * inv), pack_bf16x2(acc.z * inv, acc.w * inv));
  reinterpret_cast<uint2*>(p.out + row * D)[lane] = outv;
  if (p.lse && lane == 0) p.lse[row] = wsum > 0.f ? mx + logf(wsum) : -INFINITY;
}

// The failure path on its own: a bounded wait on a barrier that nothing
// arrives on gives up and records a timeout like any kernel's wait would.
__global__ void wait_selftest_kernel(uint64_t budget_ns) {
  __shared__ uint64_t bar_word;
  __shared__ int abort_flag;
  const uint32_t b = smem_u32(&bar_word);
  mbar_init(b, 1);
  abort_flag = 0;
  fence_mbar_init();
  if (!mbar_wait(b, 0, budget_ns, &abort_flag)) record_timeout(&abort_flag);
}

}  // namespace

cudaError_t launch_wait_selftest(uint64_t budget_ns, cudaStream_t stream) {
  wait_selftest_kernel<<<1, 1, 0, stream>>>(budget_ns);
  return cudaGetLastError();
}

cudaError_t launch_attention(const AttnLaunch& p, const AttnMaps& maps, cudaStream_t stream) {
  if (p.total_tiles <= 0 || p.n_layers_call <= 0) return cudaSuccess;
  static_assert(kSmemBytes <= 227 * 1024, "shared memory budget");
  const bool kinds = p.splits > 1 && !p.short_rows && p.cta_prefix[p.n_seqs] > 0;
  // (short-row launches never take a kinds plan)
  void (*kernel)(const AttnLaunch, const AttnMaps);
  if (p.softcap_out > 0.f)
    kernel = p.short_rows ? attention_kernel<true, true, false>
                          : (kinds ? attention_kernel<true, false, true> : attention_kernel<true, false, false>);
  else
    kernel = p.short_rows ? attention_kernel<false, true, false>
                          : (kinds ? attention_kernel<false, false, true> : attention_kernel<false, false, false>);
  cudaError_t e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kSmemBytes);
  if (e != cudaSuccess) return e;
  const dim3 grid = kinds ? dim3((unsigned)p.cta_prefix[p.n_seqs], (unsigned)p.n_kv_heads,
                                 (unsigned)p.n_layers_call)
                         : dim3((unsigned)p.total_tiles, (unsigned)p.n_kv_heads,
                                (unsigned)(p.n_layers_call * p.splits));
  // Programmatic stream serialization: the CTAs may start (and set up) while
  // the previous kernel of the stream finishes; they wait for it before any
  // global memory access.
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemBytes;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, p, maps);
}

cudaError_t launch_attn_combine(const AttnLaunch& p, cudaStream_t stream) {
  const int64_t rows = (int64_t)p.n_layers_call * p.n_tok * p.n_q_heads;
  if (rows <= 0) return cudaSuccess;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)((rows + 3) / 4));
  cfg.blockDim = dim3(128);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, combine_kernel, p);
}

cudaError_t attention_take_timeout(unsigned int* flag, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  e = cudaMemcpyFromSymbol(flag, g_attn_timeout, sizeof(unsigned int));
  if (e != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_attn_timeout, &zero, sizeof(unsigned int));
}

}  // namespace nexus

// ---------------------------------------------------------------------------
// Attention without any device allocation by the caller.
//
// Some callers cannot obtain device memory for the split-KV partials: code
// running while a stream is being captured (cudaMalloc is not allowed there),
// plug-ins that only ever receive their input and output buffers from a host
// framework, or processes whose memory pool is fixed up front. For them the
// partials live in one file-scope array that the module owns; every GPU that
// loads this library keeps it until the process exits.
// ---------------------------------------------------------------------------
namespace nexus {
namespace {
constexpr size_t kStaticScratchBytes = size_t(32) << 20;   // 32 MiB
static __device__ __align__(256) unsigned char g_static_split_scratch[kStaticScratchBytes];

// A __device__ array's address belongs to the CUDA context that loaded the
// module, not to the device: after cudaDeviceReset, or under a context a
// plug-in made current itself, the array may sit elsewhere. The address is
// therefore remembered per context, keyed by the context's unique id (ids are
// never reused within a process, unlike context handles).
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);
struct ScratchEntry {
  unsigned long long ctx_id;
  void* addr;
};
constexpr int kMaxScratchContexts = 64;
std::mutex g_scratch_mu;
ScratchEntry g_scratch[kMaxScratchContexts] = {};
int g_scratch_n = 0, g_scratch_next = 0;

template <typename Fn>
Fn driver_entry(const char* name) {
  void* f = nullptr;
  cudaDriverEntryPointQueryResult q;
  if (cudaGetDriverEntryPointByVersion(name, &f, 12000, cudaEnableDefault, &q) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess) {
    cudaGetLastError();
    return nullptr;
  }
  return reinterpret_cast<Fn>(f);
}

// Unique id of the current context; false if none is current or the driver
// cannot tell.
bool current_context_id(unsigned long long* id) {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    get_current = driver_entry<CtxGetCurrentFn>("cuCtxGetCurrent");
    get_id = driver_entry<CtxGetIdFn>("cuCtxGetId");
  });
  if (!get_current || !get_id) return false;
  CUcontext ctx = nullptr;
  if (get_current(&ctx) != CUDA_SUCCESS || !ctx) return false;
  return get_id(ctx, id) == CUDA_SUCCESS;
}

// Device address of the array in the current context. Host code cannot use the
// array's name as a device pointer, so the address is looked up once per
// context (cudaGetSymbolAddress, with that context current) and remembered.
cudaError_t static_scratch_address(void** out) {
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  unsigned long long id = 0;
  if (current_context_id(&id)) {
    for (int i = 0; i < g_scratch_n; ++i)
      if (g_scratch[i].ctx_id == id) {
        *out = g_scratch[i].addr;
        return cudaSuccess;
      }
  }
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_static_split_scratch);
  if (e != cudaSuccess) return e;
  // The lookup may have made the runtime's primary context current.
  if (current_context_id(&id)) {
    ScratchEntry& slot = g_scratch_n < kMaxScratchContexts ? g_scratch[g_scratch_n++]
                                                           : g_scratch[g_scratch_next];
    if (g_scratch_n == kMaxScratchContexts)
      g_scratch_next = (g_scratch_next + 1) % kMaxScratchContexts;
    slot.ctx_id = id;
    slot.addr = p;
  }
  *out = p;
  return cudaSuccess;
}
}  // namespace
}  // namespace nexus

extern "C" nexus_status nexus_suffix_attention_noalloc(
    const nexus_kv_cache* cache, const int32_t* d_page_tables, int32_t n_rows, int32_t max_pages,
    int32_t n_seqs, const int32_t* h_rows, const int32_t* h_kv_len, const int32_t* h_q_len,
    const void* q, void* out, float* lse, int32_t n_q_heads, int32_t layer_begin,
    int32_t layer_end, int32_t split_kv, nexus_stream stream) {
  // Arguments are validated by nexus_suffix_attention, which also returns
  // NEXUS_ENOMEM (before any launch) when the partials need more than the array.
  void* scratch = nullptr;
  if (nexus::static_scratch_address(&scratch) != cudaSuccess) {
    cudaGetLastError();
    return NEXUS_ECUDA;
  }
  return nexus_suffix_attention(cache, d_page_tables, n_rows, max_pages, n_seqs, h_rows, h_kv_len,
                                h_q_len, q, out, lse, n_q_heads, layer_begin, layer_end, split_kv,
                                scratch, nexus::kStaticScratchBytes, stream);
}
