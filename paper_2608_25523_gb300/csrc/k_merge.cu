// Exact log-sum-exp merge of split partial results.
//
// Each (token, q head) has n_slots partial results (o_i normalised over a
// disjoint key subset, lse_i natural-log): the shared-prefix splits of the
// dense kernel and the suffix splits of the split-KV kernel.  With
// M = max_i lse_i and c_i = exp(lse_i - M):
//     o = sum_i c_i o_i / sum_i c_i,   lse = M + ln(sum_i c_i),
// which equals single-pass attention over the union of the subsets.  One
// warp per (token, head); lanes own contiguous head_dim slices.
#include "kernels.h"
#include "ptx.cuh"

namespace tpa {

namespace {

constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;

template <int D>
__global__ void __launch_bounds__(256)
    merge_kernel(const MergeTok* __restrict__ toks, int n_tok, const float* __restrict__ part_o,
                 const float* __restrict__ part_lse, __nv_bfloat16* __restrict__ out,
                 float* __restrict__ lse_out, int hq) {
  constexpr int VEC = D / 32;  // 4 (d=128) or 2 (d=64)
  const int lane = threadIdx.x & 31;
  const int64_t total = static_cast<int64_t>(n_tok) * hq;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  for (int64_t w = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5; w < total;
       w += nwarps) {
    const int t = static_cast<int>(w / hq);
    const int h = static_cast<int>(w % hq);
    const MergeTok m = toks[t];
    const int64_t base = m.slot_base + static_cast<int64_t>(h) * m.n_slots;
    float mx = -INFINITY;
    for (int s = lane; s < m.n_slots; s += 32) mx = fmaxf(mx, part_lse[base + s]);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    float acc[VEC];
#pragma unroll
    for (int i = 0; i < VEC; ++i) acc[i] = 0.f;
    float tot = 0.f;
    if (mx > -INFINITY) {
      for (int s = 0; s < m.n_slots; ++s) {
        const float c = exp2f((part_lse[base + s] - mx) * kLog2e);
        tot += c;
        const float* src = part_o + (base + s) * D + lane * VEC;
        if constexpr (VEC == 4) {
          const float4 v = *reinterpret_cast<const float4*>(src);
          acc[0] += c * v.x;
          acc[1] += c * v.y;
          acc[2] += c * v.z;
          acc[3] += c * v.w;
        } else {
          const float2 v = *reinterpret_cast<const float2*>(src);
          acc[0] += c * v.x;
          acc[1] += c * v.y;
        }
      }
    }
    const float inv = tot > 0.f ? 1.f / tot : 0.f;
    __nv_bfloat16* dst = out + (static_cast<int64_t>(m.q_row) * hq + h) * D + lane * VEC;
    if constexpr (VEC == 4) {
      uint2 pk;
      pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
      pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
      *reinterpret_cast<uint2*>(dst) = pk;
    } else {
      *reinterpret_cast<uint32_t*>(dst) = pack_bf16(acc[0] * inv, acc[1] * inv);
    }
    if (lane == 0)
      lse_out[static_cast<int64_t>(m.q_row) * hq + h] =
          tot > 0.f ? mx + log2f(tot) * kLn2 : -INFINITY;
  }
}

}  // namespace

cudaError_t launch_merge(const MergeTok* toks, int n_tok, const float* part_o,
                         const float* part_lse, __nv_bfloat16* out, float* lse, int hq, int d,
                         cudaStream_t stream) {
  if (n_tok <= 0) return cudaSuccess;
  const int64_t warps = static_cast<int64_t>(n_tok) * hq;
  int64_t blocks = (warps + 7) / 8;
  if (blocks > 4096) blocks = 4096;
  if (d == 128)
    merge_kernel<128><<<static_cast<int>(blocks), 256, 0, stream>>>(toks, n_tok, part_o,
                                                                   part_lse, out, lse, hq);
  else
    merge_kernel<64><<<static_cast<int>(blocks), 256, 0, stream>>>(toks, n_tok, part_o,
                                                                  part_lse, out, lse, hq);
  return cudaGetLastError();
}

}  // namespace tpa
