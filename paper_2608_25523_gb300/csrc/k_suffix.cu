// Split-KV paged attention: the second level of the decode cascade.
//
// Every request adds a private dynamic suffix (plus its decode tokens) to
// the shared agent prefix (Sec. III, Eq. 2: d_r(t) on top of ell_a), so its
// suffix keys are read by that request alone.  One warp takes one work item
// -- the G = Hq/Hkv query rows of one token against one key range of one
// page run -- and produces a partial (o, lse) that the LSE merge combines
// with the prefix level.  The same kernel covers every key of a request in
// the flat cross-check mode.
//
// Design (memory-bound: ~4 flop per KV byte at G=4):
//  * each page of one kv head is one TMA box per operand (128-byte swizzle)
//    landing in a per-warp ring of kStages stages,
//    so loads run kStages pages ahead of the math;
//  * S^T tiles use mma.sync m16n8k16 with the G query rows on the M side
//    (padded to 16) and the 16 keys of the page on N; P*V reuses the S
//    accumulators as the A operand (no shared-memory round trip); V comes
//    through ldmatrix.trans;
//  * online softmax in base 2 with fp32 accumulators;
//  * persistent CTAs pull items from an atomic counter (items arrive sorted
//    longest first).
#include "kernels.h"
#include "ptx.cuh"

namespace tpa {

namespace {

constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

template <int D>
struct SuffixCfg {
  static constexpr int kWarps = 4;
  static constexpr int kStages = D == 128 ? 3 : 6;
  static constexpr int NCH = D / 64;                 // 64-dim chunks (128-byte rows)
  static constexpr int kPageBytes = NCH * 2048;      // one page of one kv head, K or V
  static constexpr int kStageBytes = 2 * kPageBytes;
  static constexpr int kWarpBytes = kStages * kStageBytes;
  static constexpr int kBarOffset = kWarps * kWarpBytes;
  static constexpr int kSmem = 1024 + kBarOffset + kWarps * kStages * 8;
};

template <int D, int G>
__global__ void __launch_bounds__(128) suffix_kernel(const __grid_constant__ SuffixParams p) {
  using C = SuffixCfg<D>;
  constexpr int S = C::kStages;
  extern __shared__ uint8_t smem_raw[];
  __shared__ int abort_flag;
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  uint8_t* ring = smem + warp * C::kWarpBytes;
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

  const int gq = lane >> 2;   // mma group: query row of this lane
  const int tig = lane & 3;   // thread in group
  uint32_t it = 0;            // pages consumed by this warp so far (ring position)
  bool failed = false;
  uint32_t issued = 0;        // pages issued by this warp so far

  while (!failed) {
    int idx = 0;
    if (lane == 0) idx = static_cast<int>(atomicAdd(p.queue, 1u));
    idx = __shfl_sync(0xffffffffu, idx, 0);
    if (idx >= p.n_items) break;
    const SuffixItem item = p.items[idx];
    const int npg = (item.n_keys + kPage - 1) / kPage;

    // Query fragments (A operand): rows >= G and the upper 8 rows are zero.
    uint32_t qa[D / 16][2];
    {
      const bool real = gq < G;
      const __nv_bfloat16* qrow =
          p.q + (static_cast<int64_t>(item.q_row) * p.hq + item.kv_head * G + (real ? gq : 0)) * D;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        qa[kk][0] = real ? *reinterpret_cast<const uint32_t*>(qrow + 16 * kk + 2 * tig) : 0u;
        qa[kk][1] = real ? *reinterpret_cast<const uint32_t*>(qrow + 16 * kk + 8 + 2 * tig) : 0u;
      }
    }

    auto issue = [&](int pg) {  // lane 0: TMA page `pg` of the item into ring slot issued % S
      const int st = static_cast<int>(issued % S);
      uint8_t* kst = ring + st * C::kStageBytes;
      uint8_t* vst = kst + C::kPageBytes;
      int64_t pid = p.pages[item.pages + pg];
      if (pid < 0 || pid >= p.num_pages) {
        atomicOr(p.status, kStatusBadPage);
        pid = 0;
      }
      const int z = static_cast<int>(pid * p.hkv + item.kv_head);
      fence_proxy_async();
      mbar_arrive_expect_tx(&bars[st], 2 * C::kPageBytes);
      tma_load_5d(kst, &p.tmap_k, &bars[st], 0, 0, 0, 0, z);
      tma_load_5d(vst, &p.tmap_v, &bars[st], 0, 0, 0, 0, z);
      ++issued;
    };

    if (lane == 0) {
      const int pre = npg < S ? npg : S;
      for (int i = 0; i < pre; ++i) issue(i);
    }
    issued = __shfl_sync(0xffffffffu, issued, 0);

    float o[D / 8][4];
#pragma unroll
    for (int nt = 0; nt < D / 8; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
    float m = -INFINITY, l = 0.f;

    for (int pg = 0; pg < npg; ++pg) {
      const uint32_t cnt = it + pg;
      const int st = static_cast<int>(cnt % S);
      if (!__all_sync(0xffffffffu, mbar_wait(&bars[st], (cnt / S) & 1u, &abort_flag))) {
        failed = true;
        break;
      }
      uint8_t* kst = ring + st * C::kStageBytes;
      uint8_t* vst = kst + C::kPageBytes;
      const int valid = item.n_keys - pg * kPage;
      if (valid < kPage) {
        // Slots past the end of the run hold stale pool data (possibly not
        // finite); zero their V rows so 0-weight keys contribute exactly 0.
        const int nunits = (kPage - valid) * C::NCH * 8;
        for (int u = lane; u < nunits; u += 32) {
          const int key = valid + u / (C::NCH * 8);
          const int cu = u % (C::NCH * 8);
          *reinterpret_cast<uint4*>(vst + kv_off<C::NCH>(key, cu)) = make_uint4(0, 0, 0, 0);
        }
        __syncwarp();
      }
      const uint32_t kbase = smem_u32(kst);
      const uint32_t vbase = smem_u32(vst);

      // S = Q K^T over the page's 16 keys: n-tile 0 = keys 0-7, n-tile 1 = keys 8-15.
      float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
      {
        const int key = ((lane >> 4) << 3) + (lane & 7);
        const int usel = (lane >> 3) & 1;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const int unit = 2 * kk + usel;
          uint32_t b0, b1, b2, b3;
          ldmatrix_x4(kbase + kv_off<C::NCH>(key, unit), b0, b1, b2, b3);
          mma_bf16_16816(s0, qa[kk][0], 0u, qa[kk][1], 0u, b0, b1);
          mma_bf16_16816(s1, qa[kk][0], 0u, qa[kk][1], 0u, b2, b3);
        }
      }
      const float sc = p.scale_log2;
      const int k0 = 2 * tig;
      const float x0 = k0 < valid ? s0[0] * sc : -INFINITY;
      const float x1 = k0 + 1 < valid ? s0[1] * sc : -INFINITY;
      const float x2 = k0 + 8 < valid ? s1[0] * sc : -INFINITY;
      const float x3 = k0 + 9 < valid ? s1[1] * sc : -INFINITY;
      float mx = fmaxf(fmaxf(x0, x1), fmaxf(x2, x3));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 1));
      mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, 2));
      const float m_new = fmaxf(m, mx);  // finite: key 0 of every page is valid
      const float alpha = fast_exp2(m - m_new);
      const float p0 = fast_exp2(x0 - m_new), p1 = fast_exp2(x1 - m_new);
      const float p2 = fast_exp2(x2 - m_new), p3 = fast_exp2(x3 - m_new);
      l = l * alpha + ((p0 + p1) + (p2 + p3));
      m = m_new;
#pragma unroll
      for (int nt = 0; nt < D / 8; ++nt) {
        o[nt][0] *= alpha;
        o[nt][1] *= alpha;
      }
      const uint32_t pa0 = pack_bf16(p0, p1);
      const uint32_t pa2 = pack_bf16(p2, p3);

      // O += P V: V rows are keys (k), dims are n; two n-tiles per ldmatrix.x4.trans.
      {
        const int mat = lane >> 3;
        const int key = ((mat & 1) << 3) + (lane & 7);
#pragma unroll
        for (int np = 0; np < D / 16; ++np) {
          const int unit = 2 * np + (mat >> 1);
          uint32_t b0, b1, b2, b3;
          ldmatrix_x4_trans(vbase + kv_off<C::NCH>(key, unit), b0, b1, b2, b3);
          mma_bf16_16816(o[2 * np], pa0, 0u, pa2, 0u, b0, b1);
          mma_bf16_16816(o[2 * np + 1], pa0, 0u, pa2, 0u, b2, b3);
        }
      }
      __syncwarp();
      if (lane == 0 && pg + S < npg) issue(pg + S);
      issued = __shfl_sync(0xffffffffu, issued, 0);
    }
    if (failed) break;
    it += npg;

    l += __shfl_xor_sync(0xffffffffu, l, 1);
    l += __shfl_xor_sync(0xffffffffu, l, 2);
    if (gq < G) {
      const int h = item.kv_head * G + gq;
      const int64_t slot = item.slot_base + static_cast<int64_t>(h) * item.n_slots + item.split;
      const float inv = 1.f / l;
      float* dst = p.part_o + slot * D;
#pragma unroll
      for (int nt = 0; nt < D / 8; ++nt)
        *reinterpret_cast<float2*>(dst + 8 * nt + 2 * tig) =
            make_float2(o[nt][0] * inv, o[nt][1] * inv);
      if (tig == 0) p.part_lse[slot] = (m + __log2f(l)) * kLn2;
    }
  }

  if (failed) {
    if (lane == 0) {
      atomicOr(p.status, kStatusSuffixTimeout);
      abort_flag = 1;
    }
  }
  // Every issued page must land before the CTA exits: wait (bounded) for
  // the outstanding ring slots.  On the normal path none are outstanding.
  if (lane == 0 && failed) {
    volatile int never = 0;
    for (uint32_t c = it; c < issued; ++c) {
      const int st = static_cast<int>(c % S);
      (void)mbar_wait(&bars[st], (c / S) & 1u, &never);
    }
  }
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
