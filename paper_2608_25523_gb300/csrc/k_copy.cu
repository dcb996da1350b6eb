// KV writes into the paged pool and page-run copies.
//
//  * append: the new tokens of a call (decode tokens, prefill chunks, plain
//    appends) go to (page, slot) positions chosen by the host planner.
//    Suffixes start on a fresh page, so shared prefix pages are never
//    written by a request (the prefix is paid once per agent, Eq. 2).
//  * page copy: a contiguous [len][Hkv][d] prefix <-> its page run, in
//    either direction.  The prefix movement between CPU and GPU memory
//    (Sec. IV-B, Eq. 7) uses it on the device side of a copy-engine
//    transfer: the reload scatters a staged prefix into free, possibly
//    fragmented pages, the offload gathers the pages into the staging area.
//    Prefix writes from device (or mapped pinned host) arrays use it
//    directly.
// Every copy moves 16-byte units; consecutive threads take consecutive
// units of one token row, so both sides are coalesced.
#include "kernels.h"

namespace tpa {

namespace {

constexpr int kCopyThreads = 256;

constexpr int kAppendUnroll = 4;

// Unit x of the call (32-bit: the host checks the count) is 16-byte unit
// x % upr of slot (x / upr) % 16 of run x / (16 upr), where a slot row is
// one token's K (or V) across the kv heads and slots past the run's n are
// idle; each thread loads kAppendUnroll units of K and of V before it
// stores any, so enough bytes are in flight to stream at HBM rate.
template <int CPR>
__global__ void __launch_bounds__(kCopyThreads)
    append_kernel(const AppendRow* __restrict__ rows, int n_runs, const uint4* __restrict__ k_src,
                  const uint4* __restrict__ v_src, uint4* __restrict__ k_pool,
                  uint4* __restrict__ v_pool, int64_t num_pages, int hkv, uint32_t* status) {
  const int upr = hkv * CPR;
  const int total = n_runs * kPage * upr;
  const int stride = gridDim.x * blockDim.x;
  for (int u = blockIdx.x * blockDim.x + threadIdx.x; u < total; u += kAppendUnroll * stride) {
    uint4 kx[kAppendUnroll], vx[kAppendUnroll];
    int64_t dst[kAppendUnroll];
#pragma unroll
    for (int i = 0; i < kAppendUnroll; ++i) {
      dst[i] = -1;
      const int x = u + i * stride;
      if (x >= total) continue;
      const int row = x / upr;  // run * 16 + token of the run
      const int rem = x - row * upr;
      const AppendRow r = rows[row / kPage];
      const int j = row % kPage;
      if (j >= r.n) continue;
      if (r.page < 0 || r.page >= num_pages || r.slot < 0 || r.slot + r.n > kPage) {
        atomicOr(status, kStatusBadPage);
        continue;
      }
      const int h = rem / CPR, c = rem % CPR;
      dst[i] = ((static_cast<int64_t>(r.page) * hkv + h) * kPage + r.slot + j) * CPR + c;
      const int64_t src = static_cast<int64_t>(r.src + j) * upr + rem;
      kx[i] = k_src[src];
      vx[i] = v_src[src];
    }
#pragma unroll
    for (int i = 0; i < kAppendUnroll; ++i) {
      if (dst[i] < 0) continue;
      k_pool[dst[i]] = kx[i];
      v_pool[dst[i]] = vx[i];
    }
  }
}

__global__ void __launch_bounds__(kCopyThreads)
    page_copy_kernel(const int32_t* __restrict__ pages, int len, int to_pages,
                     const uint4* __restrict__ k_lin, const uint4* __restrict__ v_lin,
                     uint4* __restrict__ k_lin_out, uint4* __restrict__ v_lin_out,
                     uint4* __restrict__ k_pool, uint4* __restrict__ v_pool, int64_t num_pages,
                     int hkv, int cpr, uint32_t* status) {
  const int64_t total = static_cast<int64_t>(len) * hkv * cpr;
  for (int64_t u = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; u < total;
       u += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int c = static_cast<int>(u % cpr);
    const int64_t t = u / cpr;
    const int h = static_cast<int>(t % hkv);
    const int tok = static_cast<int>(t / hkv);
    const int64_t page = pages[tok / kPage];
    if (page < 0 || page >= num_pages) {
      atomicOr(status, kStatusBadPage);
      continue;
    }
    const int64_t lin = (static_cast<int64_t>(tok) * hkv + h) * cpr + c;
    const int64_t pg = ((page * hkv + h) * kPage + tok % kPage) * cpr + c;
    if (to_pages) {
      k_pool[pg] = k_lin[lin];
      v_pool[pg] = v_lin[lin];
    } else {
      k_lin_out[lin] = k_pool[pg];
      v_lin_out[lin] = v_pool[pg];
    }
  }
}

int copy_grid(int64_t units) {
  int64_t blocks = (units + kCopyThreads - 1) / kCopyThreads;
  if (blocks > 4096) blocks = 4096;
  if (blocks < 1) blocks = 1;
  return static_cast<int>(blocks);
}

}  // namespace

cudaError_t launch_append(const AppendRow* rows, int n_runs, const void* k_src,
                          const void* v_src, const PoolGeom& pool, uint32_t* status,
                          cudaStream_t stream) {
  if (n_runs <= 0) return cudaSuccess;
  const int cpr = pool.d / 8;
  const int64_t units = static_cast<int64_t>(n_runs) * kPage * pool.hkv * cpr;
  if (units > INT32_MAX || (cpr != 8 && cpr != 16)) return cudaErrorInvalidValue;
  const int grid = copy_grid((units + kAppendUnroll - 1) / kAppendUnroll);
  auto* const ks = static_cast<const uint4*>(k_src);
  auto* const vs = static_cast<const uint4*>(v_src);
  auto* const kp = static_cast<uint4*>(pool.k);
  auto* const vp = static_cast<uint4*>(pool.v);
  if (cpr == 16)
    append_kernel<16><<<grid, kCopyThreads, 0, stream>>>(rows, n_runs, ks, vs, kp, vp,
                                                         pool.num_pages, pool.hkv, status);
  else
    append_kernel<8><<<grid, kCopyThreads, 0, stream>>>(rows, n_runs, ks, vs, kp, vp,
                                                        pool.num_pages, pool.hkv, status);
  return cudaGetLastError();
}

cudaError_t launch_page_copy(const int32_t* pages, int len, int to_pages, const void* k_lin,
                             const void* v_lin, void* k_lin_out, void* v_lin_out,
                             const PoolGeom& pool, uint32_t* status, cudaStream_t stream) {
  if (len <= 0) return cudaSuccess;
  const int cpr = pool.d / 8;
  const int64_t units = static_cast<int64_t>(len) * pool.hkv * cpr;
  page_copy_kernel<<<copy_grid(units), kCopyThreads, 0, stream>>>(
      pages, len, to_pages, static_cast<const uint4*>(k_lin), static_cast<const uint4*>(v_lin),
      static_cast<uint4*>(k_lin_out), static_cast<uint4*>(v_lin_out),
      static_cast<uint4*>(pool.k), static_cast<uint4*>(pool.v), pool.num_pages, pool.hkv, cpr,
      status);
  return cudaGetLastError();
}

}  // namespace tpa
