// Exact combination of partial attention results over disjoint key sets
// (the log-sum-exp algebra behind split-KV and the two-level prefix/suffix
// attention): with c_i = e^(lse_i - M), M = max_i lse_i,
//   o = sum_i c_i o_i / sum_i c_i,   lse = M + ln sum_i c_i.
// Used by the kernels that finish the last partial of a (token, kv head).
#pragma once
#include <cuda_runtime.h>
#include <math.h>
#include <stdint.h>

namespace tpa {

// One thread's share of the merge of `n` partials of one row: 4*NV
// consecutive dims.  lse[i] is partial i's log-sum-exp, o + i*o_stride its
// first dim of the share.  B partials are loaded at once (independent
// loads: one memory latency per batch rather than per partial) and folded
// into a running maximum m; on return acc = sum_i e^(lse_i - m) o_i and
// tot = sum_i e^(lse_i - m) (m = -inf, tot = 0 when no partial is finite).
// Partials are read from L2 (__ldcg): other CTAs wrote them.
template <int NV, int B>
__device__ __forceinline__ void merge_partials(const float* lse, const float* o, int n,
                                               int64_t o_stride, float (&acc)[4 * NV], float& m,
                                               float& tot) {
  constexpr float kLog2e = 1.4426950408889634f;
  m = -INFINITY;
  tot = 0.f;
#pragma unroll
  for (int c = 0; c < 4 * NV; ++c) acc[c] = 0.f;
  for (int i0 = 0; i0 < n; i0 += B) {
    float l[B];
    float4 v[B][NV];
#pragma unroll
    for (int b = 0; b < B; ++b) {
      const bool in = i0 + b < n;
      const float4* src = reinterpret_cast<const float4*>(o + static_cast<int64_t>(i0 + b) * o_stride);
      l[b] = in ? __ldcg(lse + i0 + b) : -INFINITY;
#pragma unroll
      for (int u = 0; u < NV; ++u) v[b][u] = in ? __ldcg(src + u) : make_float4(0.f, 0.f, 0.f, 0.f);
    }
    float mb = m;
#pragma unroll
    for (int b = 0; b < B; ++b) mb = fmaxf(mb, l[b]);
    if (mb == -INFINITY) continue;
    const float r = m == -INFINITY ? 0.f : exp2f((m - mb) * kLog2e);
    tot *= r;
#pragma unroll
    for (int c = 0; c < 4 * NV; ++c) acc[c] *= r;
#pragma unroll
    for (int b = 0; b < B; ++b) {
      const float w = l[b] == -INFINITY ? 0.f : exp2f((l[b] - mb) * kLog2e);
      tot += w;
#pragma unroll
      for (int u = 0; u < NV; ++u) {
        acc[4 * u + 0] += w * v[b][u].x;
        acc[4 * u + 1] += w * v[b][u].y;
        acc[4 * u + 2] += w * v[b][u].z;
        acc[4 * u + 3] += w * v[b][u].w;
      }
    }
    m = mb;
  }
}

}  // namespace tpa
