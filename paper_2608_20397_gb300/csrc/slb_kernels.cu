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
// integer dot of query q, so lane q keeps query q's running top two. Up to 4
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

cudaError_t slb_take_timeout(unsigned int* flag, cudaStream_t stream) {
  cudaError_t e = cudaStreamSynchronize(stream);
  if (e != cudaSuccess) return e;
  if ((e = cudaMemcpyFromSymbol(flag, g_slb_timeout, sizeof(unsigned int))) != cudaSuccess) return e;
  const unsigned int zero = 0;
  return cudaMemcpyToSymbol(g_slb_timeout, &zero, sizeof(unsigned int));
}

}  // namespace nexus
