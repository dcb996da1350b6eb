// Fixed device scratch for tpa_decode_static_scratch: the split-KV partial
// results of one decode call live in a file-scope device array of this
// translation unit instead of the workspace the caller allocated.  Under
// lazy module loading (CUDA's default) only a context that runs this entry
// point loads the array; with CUDA_MODULE_LOADING=EAGER every context that
// loads the library holds it.  The address is cached per device: it is the
// primary context's, valid until that context is destroyed (cudaDeviceReset).
#include <cuda_runtime.h>

#include <mutex>

#include "kernels.h"

namespace tpa {

namespace {

constexpr size_t kStaticScratchBytes = size_t{16} << 20;  // 16 MiB per device
constexpr int kMaxDevices = 64;

__device__ __align__(256) unsigned char g_static_scratch[kStaticScratchBytes];

std::mutex g_mu;
void* g_addr[kMaxDevices] = {};

}  // namespace

size_t static_scratch_bytes() { return kStaticScratchBytes; }

cudaError_t static_scratch(int device, void** ptr) {
  if (device < 0 || device >= kMaxDevices) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> lock(g_mu);
  if (!g_addr[device]) {
    // resolved once per device, with that device current
    int prev = 0;
    cudaError_t e = cudaGetDevice(&prev);
    if (e != cudaSuccess) return e;
    if (prev != device && (e = cudaSetDevice(device)) != cudaSuccess) return e;
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_static_scratch);
    if (prev != device) {
      const cudaError_t r = cudaSetDevice(prev);
      if (e == cudaSuccess) e = r;
    }
    if (e != cudaSuccess) return e;
    g_addr[device] = p;
  }
  *ptr = g_addr[device];
  return cudaSuccess;
}

}  // namespace tpa
