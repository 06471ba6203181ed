// INT8 tool scan with the top-2 margin gate (Sec. IV-A).
//
// scores[q][t] = float(dot(codes_q, codes_t)) * (scale_q * scale_t); per query
// the two best tools (score, then lower index); routed to the best one when the
// margin top1 - top2 exceeds tau, else escalated (-1).
//
// One warp scores one tool against every query of the launch (up to 32): lane l
// reads 4-byte words l, l + 32, ... of the tool row (coalesced), multiplies them
// with the same words of each query (shared memory) by dp4a, and a 31-shuffle
// butterfly leaves lane q with the exact integer dot of query q. Lane q keeps
// query q's running top two, so no further shuffles are needed. Warps merge in
// shared memory, CTAs write their top two per query to the workspace, and the
// CTA that finishes last (an atomic ticket; nothing waits) merges them, applies
// the gate and resets the ticket for the next call. The merge uses a total order
// (score, then index), so the result does not depend on the CTAs' timing.
#include <cstdint>

#include "internal.h"

namespace nexus {
namespace {

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
  for (int t = t0 + warp; t < t1; t += kSlbWarps) {
    const int32_t* row = reinterpret_cast<const int32_t*>(p.tools + (int64_t)t * p.dim);
    int acc[32];
#pragma unroll
    for (int q = 0; q < 32; ++q) acc[q] = 0;
    for (int w = lane; w < words; w += 32) {
      const int32_t tw = __ldg(row + w);
#pragma unroll
      for (int q = 0; q < kQ; ++q) acc[q] = __dp4a(tw, s_q[q * words + w], acc[q]);
    }
    // Butterfly: after the step of width `off`, lane bit b of `off` selects
    // which half of the remaining queries this lane sums; lane l ends with query l.
#pragma unroll
    for (int off = 16; off >= 1; off >>= 1) {
      const bool upper = (lane & off) != 0;
#pragma unroll
      for (int j = 0; j < off; ++j) {
        const int send = upper ? acc[j] : acc[j + off];
        const int keep = upper ? acc[j + off] : acc[j];
        acc[j] = keep + __shfl_xor_sync(0xffffffffu, send, off);
      }
    }
    if (lane < nq) {
      const float c = qscale * __ldg(p.tool_scales + t);
      push(top, __int2float_rn(acc[0]) * c, t);
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
  if (!s_last || warp != 0) return;
  __threadfence();
  if (lane < nq) {
    Top2 m = empty_top2();
    for (int b = 0; b < (int)gridDim.x; ++b) {
      const int64_t k = (int64_t)b * 32 + lane;
      push(m, __ldcg(p.part_score + 2 * k), __ldcg(p.part_idx + 2 * k));
      push(m, __ldcg(p.part_score + 2 * k + 1), __ldcg(p.part_idx + 2 * k + 1));
    }
    const bool has2 = m.i2 != INT32_MAX;
    const float s2 = has2 ? m.s2 : -INFINITY;
    p.top_idx[2 * lane] = m.i1;
    p.top_idx[2 * lane + 1] = has2 ? m.i2 : -1;
    p.top_score[2 * lane] = m.s1;
    p.top_score[2 * lane + 1] = s2;
    p.route[lane] = (m.s1 - s2) > p.tau ? m.i1 : -1;
  }
  if (lane == 0) *p.counter = 0u;
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
  if (p.n_queries <= 1) return launch_slb_as<1>(p, grid, stream);
  if (p.n_queries <= 4) return launch_slb_as<4>(p, grid, stream);
  if (p.n_queries <= 8) return launch_slb_as<8>(p, grid, stream);
  if (p.n_queries <= 16) return launch_slb_as<16>(p, grid, stream);
  return launch_slb_as<32>(p, grid, stream);
}

}  // namespace nexus
