// INT8 tool scan with the top-2 margin gate (Sec. IV-A).
//
// scores[q][t] = float(dot(codes_q, codes_t)) * (scale_q * scale_t); per query
// the two best tools (score, then lower index); routed to the best one when the
// margin top1 - top2 exceeds tau, else escalated (-1).
//
// One warp scores one tool at a time: lane l reads 4-byte words l, l + 32, ... of
// the tool row (coalesced) and multiplies them with the same words of each query
// by dp4a. Batches of 5..32 queries (slb_kernel) keep the queries in shared
// memory and reduce with a 31-shuffle butterfly that leaves lane q with the exact
// integer dot of query q, so lane q keeps query q's running top two; over large
// registries they run on the tensor cores instead (slb_tc_kernel, below). Up to 4
// queries (slb_small_kernel, the routing of single requests) read the query
// words straight into registers, load all of a tool's words at once and run
// with one or two tools per warp, for latency; over large registries they
// stream through shared memory instead (slb_stream_kernel, below). Warps merge in shared memory,
// CTAs write their top two per query to the workspace, and the CTA that
// finishes last (an atomic ticket; nothing waits) merges them, applies the gate
// and resets the ticket for the next call. The merge uses a total order (score,
// then index), so the result does not depend on the CTAs' timing.
#include <cstdint>

#include "internal.h"
#include "ptx.cuh"

namespace nexus {

__device__ unsigned int g_slb_timeout = 0;

namespace {
using namespace ptx;

constexpr int kSlbThreads = 256;
constexpr int kSlbWarps = kSlbThreads / 32;

struct Top2 {
  float s1, s2;
  int32_t i1, i2;
};

__device__ __forceinline__ bool better(float s, int32_t i, float t, int32_t j) {
  return s > t || (s == t && i < j);
}

__device__ __forceinline__ void push(Top2& a, float s, int32_t i) {
  if (better(s, i, a.s1, a.i1)) {
    a.s2 = a.s1; a.i2 = a.i1;
    a.s1 = s; a.i1 = i;
  } else if (better(s, i, a.s2, a.i2)) {
    a.s2 = s; a.i2 = i;
  }
}

__device__ __forceinline__ Top2 empty_top2() {
  Top2 a;
  a.s1 = a.s2 = -INFINITY;
  a.i1 = a.i2 = INT32_MAX;
  return a;
}

__device__ __forceinline__ Top2 shfl_top2(const Top2& a, int off) {
  Top2 b;
  b.s1 = __shfl_xor_sync(0xffffffffu, a.s1, off);
  b.s2 = __shfl_xor_sync(0xffffffffu, a.s2, off);
  b.i1 = __shfl_xor_sync(0xffffffffu, a.i1, off);
  b.i2 = __shfl_xor_sync(0xffffffffu, a.i2, off);
  return b;
}

// Run by every thread of the CTA that finished last: warp w merges the CTA
// partials of queries w, w + 8, ..., its lanes striding over the CTAs (their
// loads are independent, so they overlap), then a shuffle merge of the lanes'
// top twos; applies the gate and resets the ticket.
__device__ void final_merge(const SlbLaunch& p, int warp, int lane) {
  __threadfence();
  for (int q = warp; q < p.n_queries; q += kSlbWarps) {
    Top2 m = empty_top2();
    for (int b = lane; b < (int)gridDim.x; b += 32) {
      const int64_t k = (int64_t)b * 32 + q;
      push(m, __ldcg(p.part_score + 2 * k), __ldcg(p.part_idx + 2 * k));
      push(m, __ldcg(p.part_score + 2 * k + 1), __ldcg(p.part_idx + 2 * k + 1));
    }
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      const Top2 o = shfl_top2(m, off);
      push(m, o.s1, o.i1);
      push(m, o.s2, o.i2);
    }
    if (lane == 0) {
      const bool has2 = m.i2 != INT32_MAX;
      const float s2 = has2 ? m.s2 : -INFINITY;
      p.top_idx[2 * q] = m.i1;
      p.top_idx[2 * q + 1] = has2 ? m.i2 : -1;
      p.top_score[2 * q] = m.s1;
      p.top_score[2 * q + 1] = s2;
      p.route[q] = (m.s1 - s2) > p.tau ? m.i1 : -1;
    }
  }
  if (threadIdx.x == 0) *p.counter = 0u;
}

template <int kQ>
__global__ void __launch_bounds__(kSlbThreads) slb_kernel(const __grid_constant__ SlbLaunch p) {
  extern __shared__ int32_t s_q[];   // [kQ][words] query codes as 4-byte words
  __shared__ Top2 s_top[kSlbWarps][32];
  __shared__ bool s_last;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int words = p.dim / 4;
  const int nq = p.n_queries;

  const int32_t* qsrc = reinterpret_cast<const int32_t*>(p.queries);
  for (int i = threadIdx.x; i < kQ * words; i += kSlbThreads)
    s_q[i] = i < nq * words ? qsrc[i] : 0;
  __syncthreads();
  const float qscale = lane < nq ? p.query_scales[lane] : 0.f;

  Top2 top = empty_top2();
  const int t0 = blockIdx.x * p.tools_per_cta;
  const int t1 = min(p.n_tools, t0 + p.tools_per_cta);
  // Two tools per step: each query word read from shared memory feeds two dp4a.
  for (int ta = t0 + 2 * warp; ta < t1; ta += 2 * kSlbWarps) {
    const bool has_b = ta + 1 < t1;
    const int32_t* row_a = reinterpret_cast<const int32_t*>(p.tools + (int64_t)ta * p.dim);
    const int32_t* row_b = row_a + (has_b ? words : 0);
    int acc[2][32];
#pragma unroll
    for (int q = 0; q < 32; ++q) acc[0][q] = acc[1][q] = 0;
    for (int w0 = lane; w0 < words; w0 += 32 * 8) {
      int32_t wa[8], wb[8];
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int w = w0 + 32 * k;
        wa[k] = w < words ? __ldg(row_a + w) : 0;
        wb[k] = w < words ? __ldg(row_b + w) : 0;
      }
#pragma unroll
      for (int k = 0; k < 8; ++k) {
        const int w = w0 + 32 * k;
        if (w >= words) break;
#pragma unroll
        for (int q = 0; q < kQ; ++q) {
          const int32_t qw = s_q[q * words + w];
          acc[0][q] = __dp4a(wa[k], qw, acc[0][q]);
          acc[1][q] = __dp4a(wb[k], qw, acc[1][q]);
        }
      }
    }
#pragma unroll
    for (int x = 0; x < 2; ++x) {
      // Butterfly: at the step of width `off`, this lane's bit `off` picks which
      // half of the remaining queries it keeps summing; lane l ends with query l.
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) {
        const bool upper = (lane & off) != 0;
#pragma unroll
        for (int j = 0; j < off; ++j) {
          const int send = upper ? acc[x][j] : acc[x][j + off];
          const int keep = upper ? acc[x][j + off] : acc[x][j];
          acc[x][j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
        }
      }
    }
    if (lane < nq) {
      push(top, __int2float_rn(acc[0][0]) * (qscale * __ldg(p.tool_scales + ta)), ta);
      if (has_b)
        push(top, __int2float_rn(acc[1][0]) * (qscale * __ldg(p.tool_scales + ta + 1)), ta + 1);
    }
  }
  s_top[warp][lane] = top;
  __syncthreads();
  if (warp == 0) {
    Top2 m = s_top[0][lane];
    for (int w = 1; w < kSlbWarps; ++w) {
      const Top2 o = s_top[w][lane];
      push(m, o.s1, o.i1);
      push(m, o.s2, o.i2);
    }
    if (lane < nq) {
      const int64_t k = (int64_t)blockIdx.x * 32 + lane;
      p.part_score[2 * k] = m.s1;
      p.part_score[2 * k + 1] = m.s2;
      p.part_idx[2 * k] = m.i1;
      p.part_idx[2 * k + 1] = m.i2;
    }
    __threadfence();
  }
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(p.counter, 1u) == gridDim.x - 1;
  __syncthreads();
  if (s_last) final_merge(p, warp, lane);
}

// Few queries (the routing of one request): the latency path. Query words are
// read straight into registers (no shared-memory staging before the scan can
// start), each warp takes one tool at a time with all of its words loaded at
// once, and the host gives it enough CTAs that a warp sees one or two tools.
template <int kQ, int kT>
__global__ void __launch_bounds__(kSlbThreads) slb_small_kernel(const __grid_constant__ SlbLaunch p) {
  __shared__ Top2 s_top[kSlbWarps][kQ];
  __shared__ bool s_last;
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int words = p.dim / 4;
  const int nq = p.n_queries;
  const int32_t* qsrc = reinterpret_cast<const int32_t*>(p.queries);

  Top2 top[kQ];
#pragma unroll
  for (int q = 0; q < kQ; ++q) top[q] = empty_top2();
  const int t0 = blockIdx.x * p.tools_per_cta;
  const int t1 = min(p.n_tools, t0 + p.tools_per_cta);
  // kT tools per warp step, every word of the step loaded before any product.
  for (int ta = t0 + kT * warp; ta < t1; ta += kT * kSlbWarps) {
    int acc[kT][kQ];
#pragma unroll
    for (int x = 0; x < kT; ++x)
#pragma unroll
      for (int q = 0; q < kQ; ++q) acc[x][q] = 0;
    for (int w0 = lane; w0 < words; w0 += 32 * 8) {
      int32_t tw[kT][8];
#pragma unroll
      for (int x = 0; x < kT; ++x) {
        const int32_t* row = reinterpret_cast<const int32_t*>(p.tools + (int64_t)(ta + x) * p.dim);
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int w = w0 + 32 * k;
          tw[x][k] = (ta + x < t1 && w < words) ? __ldg(row + w) : 0;
        }
      }
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
#pragma unroll
        for (int k = 0; k < 8; ++k) {
          const int w = w0 + 32 * k;
          const int32_t qw = (q < nq && w < words) ? __ldg(qsrc + q * words + w) : 0;
#pragma unroll
          for (int x = 0; x < kT; ++x) acc[x][q] = __dp4a(tw[x][k], qw, acc[x][q]);
        }
      }
    }
#pragma unroll
    for (int x = 0; x < kT; ++x) {
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
#pragma unroll
        for (int off = 16; off >= 1; off >>= 1)
          acc[x][q] += __shfl_xor_sync(0xffffffffu, acc[x][q], off);
        if (q < nq && ta + x < t1) {
          const float c = __ldg(p.query_scales + q) * __ldg(p.tool_scales + ta + x);
          push(top[q], __int2float_rn(acc[x][q]) * c, ta + x);
        }
      }
    }
  }
  if (lane == 0) {
#pragma unroll
    for (int q = 0; q < kQ; ++q) s_top[warp][q] = top[q];
  }
  __syncthreads();
  if (warp == 0) {
    if (lane < nq) {
      Top2 m = s_top[0][lane];
      for (int w = 1; w < kSlbWarps; ++w) {
        const Top2 o = s_top[w][lane];
        push(m, o.s1, o.i1);
        push(m, o.s2, o.i2);
      }
      const int64_t k = (int64_t)blockIdx.x * 32 + lane;
      p.part_score[2 * k] = m.s1;
      p.part_score[2 * k + 1] = m.s2;
      p.part_idx[2 * k] = m.i1;
      p.part_idx[2 * k + 1] = m.i2;
    }
    __threadfence();
  }
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(p.counter, 1u) == gridDim.x - 1;
  __syncthreads();
  if (s_last) final_merge(p, warp, lane);
}

// A large registry with few queries is a pure stream of HBM reads (each code
// byte is used once per query). Each CTA owns a contiguous range of tools and
// streams it through a ring of shared-memory stages: one thread issues a bulk
// copy per stage as soon as the stage is free, so the copies run ahead of the
// products without holding registers; eight warps split the stage's tools,
// groups of lanes per tool striding over its 4-byte words, dp4a against the
// query words held in shared memory, and a butterfly sum within the group. The stage also
// carries the tools' scales (the scale array must be 16-byte aligned). A CTA's last,
// partial stage is read straight from global memory (its size need not be a
// multiple of 16 bytes). Waits are bounded; on expiry the CTA records a
// timeout, lets its copies land and finishes the merge with what it has.
constexpr int kStreamWarps = 8;                          // product warps
constexpr int kStreamThreads = (kStreamWarps + 1) * 32;  // + the copy warp
constexpr uint64_t kSlbBudgetNs = 2000000000ull;
constexpr uint64_t kSlbDrainNs = 200000000ull;

template <int kQ>
__global__ void __launch_bounds__(kStreamThreads, 2) slb_stream_kernel(const __grid_constant__ SlbLaunch p) {
  extern __shared__ uint8_t s_dyn[];
  __shared__ Top2 s_top[kStreamWarps][kQ];
  __shared__ bool s_last;
  __shared__ int s_abort;
  __shared__ int s_never;
  uint8_t* s_base = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(s_dyn) + 127) &
                                               ~static_cast<uintptr_t>(127));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int words = p.dim / 4;
  const int nq = p.n_queries;
  const int T = p.chunk_tools;
  const int S = p.stages;
  const uint32_t chunk_bytes = static_cast<uint32_t>(T) * p.dim;
  const uint32_t scale_bytes = static_cast<uint32_t>(T) * 4u;
  uint8_t* s_tools = s_base;                                                       // [S][T][dim]
  float* s_scale = reinterpret_cast<float*>(s_base + (size_t)S * chunk_bytes);     // [S][T]
  int32_t* s_q = reinterpret_cast<int32_t*>(s_base + (size_t)S * (chunk_bytes + scale_bytes));
  const uint32_t bar0 = smem_u32(reinterpret_cast<uint8_t*>(s_q) + ((kQ * p.dim + 15) & ~15));
  auto full = [&](int s) -> uint32_t { return bar0 + 8u * s; };
  auto empty = [&](int s) -> uint32_t { return bar0 + 8u * (S + s); };
  const volatile unsigned int* gabort = &g_slb_timeout;

  const int t0 = blockIdx.x * p.tools_per_cta;
  const int t1 = min(p.n_tools, t0 + p.tools_per_cta);
  const int n_own = max(0, t1 - t0);
  const int n_full = n_own / T;                 // stages copied into shared memory
  const int n_chunks = (n_own + T - 1) / T;

  const int32_t* qsrc = reinterpret_cast<const int32_t*>(p.queries);
  for (int i = threadIdx.x; i < kQ * words; i += kStreamThreads)
    s_q[i] = i < nq * words ? qsrc[i] : 0;
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full(s), 1);
      mbar_init(empty(s), kStreamWarps);
    }
    s_abort = 0;
    s_never = 0;
    fence_mbar_init();
  }
  __syncthreads();
  volatile int* abort = &s_abort;

  Top2 top[kQ];
  float qscale[kQ];
#pragma unroll
  for (int q = 0; q < kQ; ++q) {
    top[q] = empty_top2();
    qscale[q] = q < nq ? __ldg(p.query_scales + q) : 0.f;
  }

  if (warp == kStreamWarps) {
    // ---- copy warp: one thread fills the ring
    if (lane == 0) {
      int issued = 0;
      for (int c = 0; c < n_full; ++c) {
        const int s = c % S;
        if (c >= S && !mbar_wait(empty(s), ((c / S) - 1) & 1, kSlbBudgetNs, abort, gabort)) {
          *abort = 1;
          atomicOr(&g_slb_timeout, 1u);
          break;
        }
        mbar_arrive_expect_tx(full(s), chunk_bytes + scale_bytes);
        bulk_load(smem_u32(s_tools + (size_t)s * chunk_bytes), p.tools + (int64_t)(t0 + c * T) * p.dim,
                  chunk_bytes, full(s));
        bulk_load(smem_u32(s_scale + (size_t)s * T), p.tool_scales + t0 + c * T, scale_bytes, full(s));
        issued = c + 1;
      }
      // The copies issued here land before the CTA can exit.
      for (int c = max(0, issued - S); c < issued; ++c)
        mbar_wait(full(c % S), (c / S) & 1, kSlbDrainNs, &s_never);
    }
  } else {
    // ---- product warps: warp w takes tools [w m, w m + m) of every stage,
    // L = 32 / m lanes per tool striding over its words; each lane keeps the
    // top two of the tools its lane group saw, merged across lanes at the end.
    const int m = T / kStreamWarps;            // a power of two, 1..32
    const int L = 32 / m;
    const bool vec = (p.dim & 15) == 0;        // rows and queries in 16-byte words
    const int n4 = p.dim / 16;
    const int sub = lane % L;
    const int x = warp * m + lane / L;         // this lane group's tool within a stage
    for (int c = 0; c < n_chunks; ++c) {
      const bool staged = c < n_full;
      const int s = c % S;
      if (staged) {
        const bool ok = __all_sync(0xffffffffu, mbar_wait(full(s), (c / S) & 1, kSlbBudgetNs, abort,
                                                          gabort));
        if (!ok) {
          if (lane == 0) {
            *abort = 1;
            atomicOr(&g_slb_timeout, 1u);
          }
          break;
        }
      }
      const bool valid = x < min(T, n_own - c * T);
      int acc[kQ];
#pragma unroll
      for (int q = 0; q < kQ; ++q) acc[q] = 0;
      if (valid) {
        if (staged && vec) {
          // 16-byte words of the row and the queries, four independent chains
          const int4* row = reinterpret_cast<const int4*>(s_tools + (size_t)s * chunk_bytes +
                                                          (size_t)x * p.dim);
          const int4* q4 = reinterpret_cast<const int4*>(s_q);
          int a1[kQ], a2[kQ], a3[kQ];
#pragma unroll
          for (int q = 0; q < kQ; ++q) a1[q] = a2[q] = a3[q] = 0;
#pragma unroll 2
          for (int v = sub; v < n4; v += L) {
            const int4 t = row[v];
#pragma unroll
            for (int q = 0; q < kQ; ++q) {
              const int4 u = q4[q * n4 + v];
              acc[q] = __dp4a(t.x, u.x, acc[q]);
              a1[q] = __dp4a(t.y, u.y, a1[q]);
              a2[q] = __dp4a(t.z, u.z, a2[q]);
              a3[q] = __dp4a(t.w, u.w, a3[q]);
            }
          }
#pragma unroll
          for (int q = 0; q < kQ; ++q) acc[q] += (a1[q] + a2[q]) + a3[q];
        } else if (staged) {
          const int32_t* row =
              reinterpret_cast<const int32_t*>(s_tools + (size_t)s * chunk_bytes + (size_t)x * p.dim);
#pragma unroll 4
          for (int w = sub; w < words; w += L) {
            const int32_t tw = row[w];
#pragma unroll
            for (int q = 0; q < kQ; ++q) acc[q] = __dp4a(tw, s_q[q * words + w], acc[q]);
          }
        } else {
          const int32_t* row =
              reinterpret_cast<const int32_t*>(p.tools + ((int64_t)(t0 + c * T) + x) * p.dim);
#pragma unroll 4
          for (int w = sub; w < words; w += L) {
            const int32_t tw = __ldg(row + w);
#pragma unroll
            for (int q = 0; q < kQ; ++q) acc[q] = __dp4a(tw, s_q[q * words + w], acc[q]);
          }
        }
      }
      const int tool = t0 + c * T + x;
      const float ts = !valid ? 0.f : staged ? s_scale[s * T + x] : __ldg(p.tool_scales + tool);
#pragma unroll
      for (int q = 0; q < kQ; ++q) {
        for (int off = L >> 1; off >= 1; off >>= 1) acc[q] += __shfl_xor_sync(0xffffffffu, acc[q], off);
        if (valid && q < nq) push(top[q], __int2float_rn(acc[q]) * (qscale[q] * ts), tool);
      }
      if (staged) {
        __syncwarp();
        if (lane == 0) mbar_arrive(empty(s));
      }
    }
    // The lanes of a group hold the same top two: one lane per group enters
    // the merge, so every tool is counted once.
#pragma unroll
    for (int q = 0; q < kQ; ++q) {
      if (sub != 0) top[q] = empty_top2();
#pragma unroll
      for (int off = 16; off >= 1; off >>= 1) {
        const Top2 o = shfl_top2(top[q], off);
        push(top[q], o.s1, o.i1);
        push(top[q], o.s2, o.i2);
      }
    }
    if (lane == 0) {
#pragma unroll
      for (int q = 0; q < kQ; ++q) s_top[warp][q] = top[q];
    }
  }
  __syncthreads();
  if (warp == 0) {
    if (lane < nq) {
      Top2 m = s_top[0][lane];
      for (int w = 1; w < kStreamWarps; ++w) {
        const Top2 o = s_top[w][lane];
        push(m, o.s1, o.i1);
        push(m, o.s2, o.i2);
      }
      const int64_t k = (int64_t)blockIdx.x * 32 + lane;
      p.part_score[2 * k] = m.s1;
      p.part_score[2 * k + 1] = m.s2;
      p.part_idx[2 * k] = m.i1;
      p.part_idx[2 * k + 1] = m.i2;
    }
    __threadfence();
  }
  __syncthreads();
  if (threadIdx.x == 0) s_last = atomicAdd(p.counter, 1u) == gridDim.x - 1;
  __syncthreads();
  if (s_last) final_merge(p, warp, lane);
}

size_t stream_smem_bytes(const SlbLaunch& p, int kq) {
  return (size_t)p.stages * p.chunk_tools * (p.dim + 4) + ((kq * p.dim + 15) & ~15) +
         16u * p.stages + 128;
}

template <int kQ>
cudaError_t launch_stream_as(const SlbLaunch& p, int grid, cudaStream_t stream) {
  const size_t smem = stream_smem_bytes(p, kQ);
  cudaError_t e = cudaFuncSetAttribute(slb_stream_kernel<kQ>,
                                       cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  // all of the SM's unified L1 / shared storage as shared memory: two CTAs per SM
  e = cudaFuncSetAttribute(slb_stream_kernel<kQ>, cudaFuncAttributePreferredSharedMemoryCarveout,
                           (int)cudaSharedmemCarveoutMaxShared);
  if (e != cudaSuccess) return e;
  slb_stream_kernel<kQ><<<(unsigned)grid, kStreamThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

// ---------------------------------------------------------------------------
// Batches of 5..32 queries over a large registry on the tensor cores. The
// integer dot products are computed exactly by bf16 products with float32
// accumulation: every int8 code (-128 included) is exact in bf16, and for
// dim <= 1024 every partial sum is an integer of magnitude at most
// 1024 * 128 * 128 = 2^24, which float32 holds exactly, so the order of the
// additions does not matter and the scores equal those of the dp4a kernels bit
// for bit. A CTA walks tiles of 128 tools; per 64-dimension chunk of a tile:
//   warp 0     TMA copy of the chunk's int8 codes (128 x 64 bytes) into an
//              8-stage ring
//   warps 2-4, 6-8, 10-11
//              convert the codes to bf16 in the 128-byte-swizzled K-major
//              layout of the MMA's A operand (4-slot ring): a code v becomes
//              the float 2^23 + (v + 128), minus 2^23 + 128, packed to bf16
//              (eight warps, none on the issuing thread's sub-partition; warps
//              5 and 9 stay idle)
//   warp 1     tcgen05.mma 128 x 32 x 16 against the queries (bf16, resident,
//              rows past the batch zero), four per chunk, into one of two
//              32-column TMEM accumulators
//   warps 12-15 read the accumulator (thread = tool), scale, and keep per-query
//              top twos through a shared-memory transpose
// Every wait is bounded; on expiry the CTA records a timeout and winds down.
constexpr int kTcThreads = 512;
constexpr int kTcTools = 128;
constexpr int kTcStaging = 8;                  // int8 chunk ring
constexpr int kTcASlots = 4;                   // bf16 A ring
constexpr uint32_t kTcStBytes = kTcTools * 64;        // 8 KiB
constexpr uint32_t kTcABytes = kTcTools * 128;        // 16 KiB
constexpr uint32_t kTcOffB = 0;                       // queries: dim / 64 chunks of 4 KiB
constexpr uint32_t kTcOffSt = 64 * 1024;
constexpr uint32_t kTcOffA = kTcOffSt + kTcStaging * kTcStBytes;
constexpr uint32_t kTcOffSc = kTcOffA + kTcASlots * kTcABytes;   // scores [128][33]
constexpr uint32_t kTcOffTop = kTcOffSc + kTcTools * 33 * 4;
constexpr uint32_t kTcOffQs = kTcOffTop + 4 * 32 * sizeof(Top2);
constexpr uint32_t kTcOffBar = kTcOffQs + 32 * 4;
constexpr int kTcBars = 2 * kTcStaging + 2 * kTcASlots + 4 + 1;
constexpr uint32_t kTcOffMisc = kTcOffBar + kTcBars * 8;
constexpr uint32_t kTcSmem = kTcOffMisc + 32 + 1024;
static_assert(kTcSmem <= 227 * 1024, "shared memory budget");
constexpr uint64_t kTcBudgetNs = 2000000000ull;
constexpr uint64_t kTcDrainNs = 200000000ull;

__device__ __forceinline__ void record_timeout(volatile int* abort) {
  *abort = 1;
  atomicOr(&g_slb_timeout, 1u);
}

// 16 codes -> 16 bf16 (8 words), exactly.
__device__ __forceinline__ void codes_to_bf16(const uint4& c, uint32_t (&o)[8]) {
  const uint32_t w[4] = {c.x, c.y, c.z, c.w};
  // __byte_perm selector 0x765k: byte k of u, then bytes 1-3 of 0x4B000000
  const float off = 8388736.f;   // 2^23 + 128
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    const uint32_t u = w[k] ^ 0x80808080u;   // bytes v + 128
    const float f0 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7650)) - off;
    const float f1 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7651)) - off;
    const float f2 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7652)) - off;
    const float f3 = __uint_as_float(__byte_perm(u, 0x4B000000u, 0x7653)) - off;
    o[2 * k] = pack_bf16x2(f0, f1);
    o[2 * k + 1] = pack_bf16x2(f2, f3);
  }
}

__device__ __forceinline__ void named_sync_128(int id) {
  asm volatile("bar.sync %0, 128;" ::"r"(id) : "memory");
}

__global__ void __launch_bounds__(kTcThreads, 1)
slb_tc_kernel(const __grid_constant__ SlbLaunch p, const __grid_constant__ CUtensorMap tmap) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  auto bar = [&](int i) -> uint32_t { return sbase + kTcOffBar + 8u * i; };
  const int B_FST = 0, B_EST = kTcStaging, B_FA = 2 * kTcStaging, B_EA = B_FA + kTcASlots,
            B_AF = B_EA + kTcASlots, B_AE = B_AF + 2, B_FIN = B_AE + 2;
  volatile uint32_t* tmem_slot = reinterpret_cast<volatile uint32_t*>(smem + kTcOffMisc);
  volatile int* abort = reinterpret_cast<volatile int*>(smem + kTcOffMisc + 4);
  volatile int* never = reinterpret_cast<volatile int*>(smem + kTcOffMisc + 8);
  volatile int* last = reinterpret_cast<volatile int*>(smem + kTcOffMisc + 12);
  float* s_sc = reinterpret_cast<float*>(smem + kTcOffSc);
  Top2* s_top = reinterpret_cast<Top2*>(smem + kTcOffTop);
  float* s_qs = reinterpret_cast<float*>(smem + kTcOffQs);
  const volatile unsigned int* gabort = &g_slb_timeout;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int nq = p.n_queries;
  const int n_chunks = p.dim / 64;
  const int n_tiles = (p.n_tools + kTcTools - 1) / kTcTools;

  if (threadIdx.x == 0) {
    for (int i = 0; i < kTcBars; ++i) {
      uint32_t count = 1;
      if ((i >= B_EST && i < B_EST + kTcStaging) || (i >= B_FA && i < B_FA + kTcASlots))
        count = 8;   // one arrival per converter warp
      if (i >= B_AE && i < B_AE + 2) count = 4;   // one per epilogue warp
      mbar_init(bar(i), count);
    }
    *abort = 0;
    *never = 0;
    fence_mbar_init();
  }
  if (threadIdx.x < 32) s_qs[threadIdx.x] = threadIdx.x < nq ? p.query_scales[threadIdx.x] : 0.f;
  // queries -> bf16 B operand: chunk c holds rows 0..31 (queries; zero past the batch)
  for (int i = threadIdx.x; i < n_chunks * 32 * 4; i += kTcThreads) {
    const int c = i / 128, row = (i / 4) % 32, q16 = i % 4;
    uint4 v = make_uint4(0, 0, 0, 0);
    if (row < nq)
      v = *reinterpret_cast<const uint4*>(p.queries + (int64_t)row * p.dim + c * 64 + q16 * 16);
    uint32_t o[8];
    codes_to_bf16(v, o);
    const uint32_t rb = sbase + kTcOffB + c * 4096 + row * 128;
    st_shared_v4(rb + (((2 * q16) ^ (row & 7)) << 4), o[0], o[1], o[2], o[3]);
    st_shared_v4(rb + (((2 * q16 + 1) ^ (row & 7)) << 4), o[4], o[5], o[6], o[7]);
  }
  fence_proxy_async_smem();
  if (warp == 1) {
    tmem_alloc(sbase + kTcOffMisc, 64);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  if (warp == 0) {
    // ------------------------------------------------------ TMA producer
    if (lane == 0) {
      prefetch_tmap(&tmap);
      int it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
        for (int c = 0; c < n_chunks; ++c, ++it) {
          const int s = it % kTcStaging;
          if (it >= kTcStaging &&
              !mbar_wait(bar(B_EST + s), ((it / kTcStaging) - 1) & 1, kTcBudgetNs, abort, gabort)) {
            ok = false;
            record_timeout(abort);
            break;
          }
          mbar_arrive_expect_tx(bar(B_FST + s), kTcStBytes);
          tma_load_2d(sbase + kTcOffSt + s * kTcStBytes, &tmap, bar(B_FST + s), c * 64,
                      t * kTcTools);
        }
      }
      for (int i = max(0, it - kTcStaging); i < it; ++i)
        mbar_wait(bar(B_FST + i % kTcStaging), (i / kTcStaging) & 1, kTcDrainNs, never);
    }
    __syncwarp();
  } else if (warp == 1) {
    // ------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_bf16_f32(kTcTools, 32, false);
      const uint64_t da0 = smem_desc(sbase + kTcOffA, 16, 1024, kSwizzle128B);
      const uint64_t db0 = smem_desc(sbase + kTcOffB, 16, 1024, kSwizzle128B);
      int it = 0, acc_it = 0;
      bool ok = true;
      for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x, ++acc_it) {
        const int b = acc_it & 1;
        if (acc_it >= 2 &&
            !mbar_wait(bar(B_AE + b), ((acc_it >> 1) - 1) & 1, kTcBudgetNs, abort, gabort)) {
          ok = false;
          record_timeout(abort);
          break;
        }
        tc_fence_after();
        for (int c = 0; c < n_chunks; ++c, ++it) {
          const int a = it % kTcASlots;
          if (!mbar_wait(bar(B_FA + a), (it / kTcASlots) & 1, kTcBudgetNs, abort, gabort)) {
            ok = false;
            record_timeout(abort);
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int kk = 0; kk < 4; ++kk)
            mma_bf16(tmem + b * 32, da0 + ((a * kTcABytes + kk * 32) >> 4),
                     db0 + ((c * 4096 + kk * 32) >> 4), idesc, (c | kk) != 0 ? 1u : 0u);
          mma_commit(bar(B_EA + a));
        }
        if (ok) mma_commit(bar(B_AF + b));
      }
      mma_commit(bar(B_FIN));
      mbar_wait(bar(B_FIN), 0, kTcDrainNs, never);
    }
    __syncwarp();
  } else if (warp < 12 && (warp & 3) != 1) {
    // ------------------------------------------------------ converters
    // converters sit on warps 2, 3, 4, 6, 7, 8, 10, 11: none shares the issuing
    // thread's sub-partition (warps 5 and 9 stay idle)
    const int cw = warp - 2 - (warp > 5 ? 1 : 0) - (warp > 9 ? 1 : 0);
    const int ct = cw * 32 + lane;
    int it = 0;
    bool ok = true;
    for (int t = blockIdx.x; t < n_tiles && ok; t += gridDim.x) {
      for (int c = 0; c < n_chunks; ++c, ++it) {
        const int s = it % kTcStaging, a = it % kTcASlots;
        bool w = mbar_wait(bar(B_FST + s), (it / kTcStaging) & 1, kTcBudgetNs, abort, gabort);
        if (w && it >= kTcASlots)
          w = mbar_wait(bar(B_EA + a), ((it / kTcASlots) - 1) & 1, kTcBudgetNs, abort, gabort);
        ok = __all_sync(0xffffffffu, w);
        if (!ok) {
          if (lane == 0) record_timeout(abort);
          break;
        }
        const uint8_t* st = smem + kTcOffSt + s * kTcStBytes;
        const uint32_t ab = sbase + kTcOffA + a * kTcABytes;
#pragma unroll
        for (int k = 0; k < 2; ++k) {
          const int i = ct + 256 * k, row = i >> 2, q16 = i & 3;
          const uint4 v = *reinterpret_cast<const uint4*>(st + row * 64 + q16 * 16);
          uint32_t o[8];
          codes_to_bf16(v, o);
          st_shared_v4(ab + row * 128 + (((2 * q16) ^ (row & 7)) << 4), o[0], o[1], o[2], o[3]);
          st_shared_v4(ab + row * 128 + (((2 * q16 + 1) ^ (row & 7)) << 4), o[4], o[5], o[6], o[7]);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
          mbar_arrive(bar(B_EST + s));
          mbar_arrive(bar(B_FA + a));
        }
      }
    }
  } else if (warp >= 12) {
    // ------------------------------------------------------ epilogue
    const int quad = warp & 3;                  // TMEM lanes [32 quad, 32 quad + 32)
    const int r = quad * 32 + lane;             // this thread's tool row of the tile
    const int et = threadIdx.x - 384;
    const int q = et & 31, part = et >> 5;      // transposed role: query q, rows of `part`
    const uint32_t lane_base = static_cast<uint32_t>(quad * 32) << 16;
    Top2 top = empty_top2();
    bool ok = true;
    int acc_it = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++acc_it) {
      const int b = acc_it & 1;
      if (ok) {
        const bool w = mbar_wait(bar(B_AF + b), (acc_it >> 1) & 1, kTcBudgetNs, abort, gabort);
        ok = __all_sync(0xffffffffu, w);
        if (!ok && lane == 0) record_timeout(abort);
      }
      if (ok) {
        tc_fence_after();
        uint32_t v[32];
        tmem_ld32(tmem + lane_base + b * 32, v);
        tmem_ld_wait();
        tc_fence_before();
        __syncwarp();
        if (lane == 0) mbar_arrive(bar(B_AE + b));
        const int tool = t * kTcTools + r;
        const float st = tool < p.n_tools ? __ldg(p.tool_scales + tool) : 0.f;
#pragma unroll
        for (int j = 0; j < 32; ++j) s_sc[r * 33 + j] = __uint_as_float(v[j]) * (s_qs[j] * st);
      }
      named_sync_128(1);
      if (ok && q < nq) {
        const int row0 = part * 32;
        const int n_valid = min(32, p.n_tools - (t * kTcTools + row0));
        for (int rr = 0; rr < n_valid; ++rr)
          push(top, s_sc[(row0 + rr) * 33 + q], t * kTcTools + row0 + rr);
      }
      named_sync_128(1);
    }
    s_top[part * 32 + q] = top;
    named_sync_128(1);
    if (part == 0 && q < nq) {
      Top2 m = s_top[q];
      for (int w = 1; w < 4; ++w) {
        const Top2 o = s_top[w * 32 + q];
        push(m, o.s1, o.i1);
        push(m, o.s2, o.i2);
      }
      const int64_t k = (int64_t)blockIdx.x * 32 + q;
      p.part_score[2 * k] = m.s1;
      p.part_score[2 * k + 1] = m.s2;
      p.part_idx[2 * k] = m.i1;
      p.part_idx[2 * k + 1] = m.i2;
      __threadfence();
    }
  }

  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  if (warp == 1) tmem_dealloc(tmem, 64);
  if (threadIdx.x == 0) *last = atomicAdd(p.counter, 1u) == gridDim.x - 1;
  __syncthreads();
  if (*last && warp < kSlbWarps) final_merge(p, warp, lane);
}

template <int kQ>
cudaError_t launch_slb_as(const SlbLaunch& p, int grid, cudaStream_t stream) {
  const size_t smem = (size_t)kQ * p.dim;
  if (smem > 48 * 1024) {
    cudaError_t e = cudaFuncSetAttribute(slb_kernel<kQ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
  }
  slb_kernel<kQ><<<(unsigned)grid, kSlbThreads, smem, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_slb(const SlbLaunch& p, int grid, cudaStream_t stream) {
  if (p.n_queries <= 0 || grid <= 0) return cudaSuccess;
  if (p.chunk_tools > 0) {
    if (p.n_queries == 1) return launch_stream_as<1>(p, grid, stream);
    return launch_stream_as<kSlbSmallQueries>(p, grid, stream);
  }
  if (p.n_queries <= kSlbSmallQueries) {
    // Many tools per warp: four per step for more loads in flight; otherwise one
    // per warp, so a small registry spreads over every warp.
    const bool tiled = p.tools_per_cta >= 4 * 2 * kSlbWarps;
    if (p.n_queries == 1) {
      if (tiled) slb_small_kernel<1, 4><<<(unsigned)grid, kSlbThreads, 0, stream>>>(p);
      else slb_small_kernel<1, 1><<<(unsigned)grid, kSlbThreads, 0, stream>>>(p);
    } else {
      if (tiled) slb_small_kernel<kSlbSmallQueries, 4><<<(unsigned)grid, kSlbThreads, 0, stream>>>(p);
      else slb_small_kernel<kSlbSmallQueries, 1><<<(unsigned)grid, kSlbThreads, 0, stream>>>(p);
    }
    return cudaGetLastError();
  }
  if (p.n_queries <= 8) return launch_slb_as<8>(p, grid, stream);
  if (p.n_queries <= 16) return launch_slb_as<16>(p, grid, stream);
  return launch_slb_as<32>(p, grid, stream);
}

cudaError_t launch_slb_tc(const SlbLaunch& p, const CUtensorMap& tools, int grid,
                          cudaStream_t stream) {
  if (p.n_queries <= 0 || grid <= 0) return cudaSuccess;
  cudaError_t e = cudaFuncSetAttribute(slb_tc_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)kTcSmem);
  if (e != cudaSuccess) return e;
  slb_tc_kernel<<<(unsigned)grid, kTcThreads, kTcSmem, stream>>>(p, tools);
  return cudaGetLastError();
}

cudaError_t slb_take_timeout(unsigned int* flag, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  if ((e = cudaMemcpyFromSymbol(flag, g_slb_timeout, sizeof(unsigned int))) != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_slb_timeout, &zero, sizeof(unsigned int));
}

}  // namespace nexus
