// Exact log-sum-exp merge of split partial results.
//
// Each (token, q head) has n_slots partial results (o_i normalised over a
// disjoint key subset, lse_i natural-log): the shared-prefix splits of the
// dense kernel and the suffix splits of the split-KV kernel.  With
// M = max_i lse_i and c_i = exp(lse_i - M):
//     o = sum_i c_i o_i / sum_i c_i,   lse = M + ln(sum_i c_i),
// which equals single-pass attention over the union of the subsets.  D/4
// lanes per (token, head), one float4 of o each; a lane loads 8 partials at
// once (merge.cuh), so a merge costs one memory latency per 8 partials.
// After a cascade decode it runs as a programmatic dependent of the main
// kernel: its CTAs are resident before that kernel ends and wait in
// griddepcontrol.wait for its partials.
#include "kernels.h"
#include "merge.cuh"
#include "ptx.cuh"

namespace tpa {

namespace {

constexpr float kLn2 = 0.6931471805599453f;
constexpr int kMergeThreads = 128;

template <int D>
__global__ void __launch_bounds__(kMergeThreads)
    merge_kernel(const MergeTok* __restrict__ toks, int n_tok, const float* __restrict__ part_o,
                 const float* __restrict__ part_lse, int64_t part_slots, uint32_t* status,
                 __nv_bfloat16* __restrict__ out, float* __restrict__ lse_out, int hq,
                 const unsigned long long* plan_flag, unsigned long long plan_seq) {
  pdl_trigger();  // the next step's main kernel may become resident now
  constexpr int LPI = D / 4;     // lanes per (token, head)
  constexpr int IPW = 32 / LPI;  // (token, head) pairs per warp and pass
  const int lane = threadIdx.x & 31;
  const int64_t total = static_cast<int64_t>(n_tok) * hq;
  const int64_t warp = (static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
  const int64_t w0 = warp * IPW + lane / LPI;
  // With the plan uploaded ahead (its flag given), the first token record
  // comes from the plan before waiting for the kernel that writes the
  // partials; the partials are read after that wait.
  MergeTok m0{0, 0, 0, 0};
  if (plan_flag) {
    const int got = threadIdx.x == 0 ? wait_flag64(plan_flag, plan_seq) : 1;
    if (!__syncthreads_and(got)) {
      if (threadIdx.x == 0) atomicOr(status, kStatusPlanTimeout);
      return;
    }
    if (w0 < total) m0 = toks[w0 / hq];
  }
  pdl_wait();     // no-op unless launched as a dependent
  for (int64_t w = w0; w < total; w += nwarps * IPW) {
    const int t = static_cast<int>(w / hq);
    const int h = static_cast<int>(w % hq);
    const MergeTok m = (plan_flag && w == w0) ? m0 : toks[t];
    const int64_t base = m.slot_base + static_cast<int64_t>(h) * m.n_slots;
    const int col = 4 * (lane % LPI);
    if (base < 0 || m.n_slots < 0 || base + m.n_slots > part_slots) {
      // partial slots outside the partial buffer: not read (status bit)
      if (lane % LPI == 0) atomicOr(status, kStatusBadSlot);
      continue;
    }
    float acc[4], mx, tot;
    merge_partials<1, 8>(part_lse + base, part_o + base * D + col, m.n_slots, D, acc, mx, tot);
    const float inv = tot > 0.f ? 1.f / tot : 0.f;
    uint2 pk;
    pk.x = pack_bf16(acc[0] * inv, acc[1] * inv);
    pk.y = pack_bf16(acc[2] * inv, acc[3] * inv);
    *reinterpret_cast<uint2*>(out + (static_cast<int64_t>(m.q_row) * hq + h) * D + col) = pk;
    if (lane % LPI == 0)
      lse_out[static_cast<int64_t>(m.q_row) * hq + h] =
          tot > 0.f ? mx + __log2f(tot) * kLn2 : -INFINITY;
  }
}

template <int D>
cudaError_t launch_merge_t(const MergeTok* toks, int n_tok, const float* part_o,
                           const float* part_lse, int64_t part_slots, uint32_t* status,
                           __nv_bfloat16* out, float* lse, int hq, int num_sms, bool dependent,
                           const unsigned long long* plan_flag, unsigned long long plan_seq,
                           cudaStream_t stream) {
  constexpr int IPB = (kMergeThreads / 32) * (32 / (D / 4));  // pairs per block and pass
  const int64_t pairs = static_cast<int64_t>(n_tok) * hq;
  int64_t blocks = (pairs + IPB - 1) / IPB;
  // At most one wave: as many blocks as can be resident at once (blocks
  // beyond that would start only as the first ones finish and double the
  // latency chain of the pairs they loop over).
  static int per_sm = 0;
  if (per_sm == 0) {
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, merge_kernel<D>, kMergeThreads, 0) !=
            cudaSuccess ||
        n < 1)
      n = 1;
    per_sm = n;
  }
  const int64_t cap = static_cast<int64_t>(num_sms > 0 ? num_sms : 1) * per_sm;
  if (blocks > cap) blocks = cap;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(blocks));
  cfg.blockDim = dim3(kMergeThreads);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, merge_kernel<D>, toks, n_tok, part_o, part_lse, part_slots, status,
                            out, lse, hq, plan_flag, plan_seq);
}

}  // namespace

cudaError_t launch_merge(const MergeTok* toks, int n_tok, const float* part_o,
                         const float* part_lse, int64_t part_slots, uint32_t* status,
                         __nv_bfloat16* out, float* lse, int hq, int d, int num_sms,
                         bool dependent, const unsigned long long* plan_flag,
                         unsigned long long plan_seq, cudaStream_t stream) {
  if (n_tok <= 0) return cudaSuccess;
  if (d == 128)
    return launch_merge_t<128>(toks, n_tok, part_o, part_lse, part_slots, status, out, lse, hq,
                               num_sms, dependent, plan_flag, plan_seq, stream);
  if (d == 64)
    return launch_merge_t<64>(toks, n_tok, part_o, part_lse, part_slots, status, out, lse, hq,
                              num_sms, dependent, plan_flag, plan_seq, stream);
  return cudaErrorInvalidValue;
}

}  // namespace tpa
