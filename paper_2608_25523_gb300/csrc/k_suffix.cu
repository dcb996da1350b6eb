// Standalone split-KV kernel (flat cross-check decode): 4 independent warps
// per CTA, each running split_warp_loop with its own TMA page ring.
#include "split_kv.cuh"

namespace tpa {

namespace {

template <int D>
struct SuffixCfg {
  static constexpr int kWarps = 4;
  static constexpr int kStages = D == 128 ? 3 : 6;
  using W = SplitCfg<D, kStages>;
  static constexpr int kBarOffset = kWarps * W::kWarpBytes;
  static constexpr int kSmem = 1024 + kBarOffset + kWarps * kStages * 8;
};

template <int D, int G>
__global__ void __launch_bounds__(128) suffix_kernel(const __grid_constant__ SuffixParams p) {
  pdl_trigger();  // the merge kernel after it may become resident now
  using C = SuffixCfg<D>;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  __shared__ int abort_flag;
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint8_t* ring = smem + warp * C::W::kWarpBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kBarOffset) + warp * S;
  if (threadIdx.x == 0) abort_flag = 0;
  if (lane == 0) {
    for (int s = 0; s < S; ++s) mbar_init(&bars[s], 1);
    fence_mbar_init();
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    prefetch_tmap(&p.tmap_k);
    prefetch_tmap(&p.tmap_v);
  }
  SplitArgs a{&p.tmap_k, &p.tmap_v, p.q, p.part_o, p.part_lse, p.items, p.n_items,
              nullptr, nullptr, nullptr, 0, 0, 0, p.pages, p.queue, p.status, p.num_pages,
              p.hq, p.hkv, p.scale_log2, p.k_new, p.v_new, p.k_pool, p.v_pool, p.part_slots, 0};
  split_warp_loop<D, G, S>(a, ring, bars, &abort_flag, lane, false);
}

template <int D, int G>
cudaError_t launch_suffix_t(const SuffixParams& p, int num_sms, cudaStream_t stream) {
  using C = SuffixCfg<D>;
  int per_sm = 1;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, suffix_kernel<D, G>,
                                                                128, C::kSmem);
  if (e != cudaSuccess) return e;
  if (per_sm < 1) per_sm = 1;
  int64_t grid = static_cast<int64_t>(num_sms) * per_sm;
  const int64_t need = (p.n_items + C::kWarps - 1) / C::kWarps;
  if (grid > need) grid = need;
  if (grid < 1) grid = 1;
  suffix_kernel<D, G><<<static_cast<int>(grid), 128, C::kSmem, stream>>>(p);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_suffix(const SuffixParams& p, int num_sms, int head_dim, int group,
                          cudaStream_t stream) {
  if (p.n_items <= 0) return cudaSuccess;
  if (head_dim == 128 && group == 4) return launch_suffix_t<128, 4>(p, num_sms, stream);
  if (head_dim == 128 && group == 8) return launch_suffix_t<128, 8>(p, num_sms, stream);
  if (head_dim == 64 && group == 4) return launch_suffix_t<64, 4>(p, num_sms, stream);
  if (head_dim == 64 && group == 8) return launch_suffix_t<64, 8>(p, num_sms, stream);
  return cudaErrorInvalidValue;
}

cudaError_t init_suffix_kernels() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(suffix_kernel<128, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SuffixCfg<128>::kSmem)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(suffix_kernel<128, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SuffixCfg<128>::kSmem)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(suffix_kernel<64, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                SuffixCfg<64>::kSmem)) != cudaSuccess)
    return e;
  return cudaFuncSetAttribute(suffix_kernel<64, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              SuffixCfg<64>::kSmem);
}

}  // namespace tpa
