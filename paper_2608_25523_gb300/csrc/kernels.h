// Host-side launchers of the library's kernels.
#pragma once
#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "plan.h"

namespace tpa {

// Paged pool geometry: bf16 [num_pages][hkv][16][d].
struct PoolGeom {
  void* k;
  void* v;
  int64_t num_pages;
  int hkv;
  int d;
};

// K/V writes: `n_runs` runs of consecutive tokens, each within one page.
// k_src/v_src are [tokens][hkv][d]; device or mapped pinned-host pointers.
cudaError_t launch_append(const AppendRow* rows, int n_runs, const void* k_src,
                          const void* v_src, const PoolGeom& pool, uint32_t* status,
                          cudaStream_t stream);

// Contiguous [len][hkv][d] <-> the pages of a page run.  to_pages = 1 copies
// src -> pages (prefix write, reload); 0 copies pages -> dst (gather, offload).
cudaError_t launch_page_copy(const int32_t* pages, int len, int to_pages, const void* k_lin,
                             const void* v_lin, void* k_lin_out, void* v_lin_out,
                             const PoolGeom& pool, uint32_t* status, cudaStream_t stream);

struct DenseParams {
  CUtensorMap tmap_k;  // 5-D view of the K pool: one box = one page of one kv head
  CUtensorMap tmap_v;
  // Device array of 2 * hkv 5-D views, K then V, one per kv head, whose
  // last dimension steps over whole pages: one box = 8 consecutive pages of
  // that kv head (a full tile whose pages are contiguous in the pool).
  const CUtensorMap* run_maps;
  const __nv_bfloat16* q;
  __nv_bfloat16* out;
  float* lse;
  float* part_o;
  float* part_lse;
  int64_t part_slots;  // entries of part_lse (part_o: part_slots x d); other slots are refused
  const DenseItem* items;
  const DenseTok* toks;
  const int32_t* pages;
  const __nv_bfloat16* k_new;  // rows appended by split items with app_src >= 0
  const __nv_bfloat16* v_new;
  __nv_bfloat16* k_pool;
  __nv_bfloat16* v_pool;
  uint32_t* status;
  int64_t num_pages;
  int n_items;       // dense items (128-row tiles)
  int n_dense_ctas;  // CTAs running dense items; the rest of the grid runs split-KV items
  // split-KV items, derived on the device from per-token records (SplitArgs)
  const SplitTok* stoks;
  const int32_t* full_prefix;
  const int32_t* tail_order;
  int n_stok, n_full, split_keys;
  int n_sitems;      // hkv * (n_full + tails)
  uint32_t* squeue;  // zeroed work counter of the split-KV items
  int hq, hkv;
  float scale_log2;  // log2(e) / sqrt(d)
  // Non-null: the plan was uploaded on another stream, followed by this
  // 8-byte flag; every CTA waits (bounded) until it reads plan_seq there.
  const unsigned long long* plan_flag;
  unsigned long long plan_seq;
};

// One persistent launch, one CTA per SM: the first n_dense_ctas CTAs run the
// dense tensor-core items (tcgen05 + TMEM + TMA), the others the split-KV
// items (warp MMA).  Grid = n_dense_ctas + n_split_ctas.  dependent = true
// launches it as a programmatic dependent of the kernel before it on the
// stream: its CTAs may start while that kernel finishes and wait for it in
// griddepcontrol.wait before touching any memory it could use.
cudaError_t launch_dense(const DenseParams& p, int n_split_ctas, int head_dim, int group,
                         bool dependent, cudaStream_t stream);

// Chunked causal prefill, one persistent launch of `grid` CTAs (one per
// SM) over items of two 128-row query tiles that share their key tiles
// (tcgen05 + TMEM + TMA).  Items must have n_tok <= 256 / group and at
// least one key tile; outputs go to p.out / p.lse (out_mode 1).  p.plan_flag
// must be null.
cudaError_t launch_prefill_pair(const DenseParams& p, int grid, int head_dim, int group,
                                cudaStream_t stream);

struct SuffixParams {
  CUtensorMap tmap_k;
  CUtensorMap tmap_v;
  const __nv_bfloat16* q;
  float* part_o;
  float* part_lse;
  int64_t part_slots;  // entries of part_lse (part_o: part_slots x d); other slots are refused
  const SuffixItem* items;
  const int32_t* pages;
  uint32_t* queue;     // zeroed work counter
  uint32_t* status;
  int64_t num_pages;
  int n_items;
  int hq, hkv;
  float scale_log2;
  // in-kernel append of the step's token (cascade decode); null otherwise
  const __nv_bfloat16* k_new;
  const __nv_bfloat16* v_new;
  __nv_bfloat16* k_pool;
  __nv_bfloat16* v_pool;
};

// Split-KV paged attention of G query rows per warp (warp-level MMA).
cudaError_t launch_suffix(const SuffixParams& p, int num_sms, int head_dim, int group,
                          cudaStream_t stream);

// Exact LSE merge of each token's partials into bf16 out and fp32 lse.
// dependent = true launches it as a programmatic dependent of the kernel
// before it on the stream (which triggers early): its CTAs become resident
// while that kernel still runs and start merging the moment it completes.
// plan_flag (non-null when the plan was uploaded ahead with that flag):
// the kernel reads its first token record before its programmatic wait.
cudaError_t launch_merge(const MergeTok* toks, int n_tok, const float* part_o,
                         const float* part_lse, int64_t part_slots, uint32_t* status,
                         __nv_bfloat16* out, float* lse, int hq, int d, int num_sms,
                         bool dependent, const unsigned long long* plan_flag,
                         unsigned long long plan_seq, cudaStream_t stream);

// Raise dynamic shared-memory limits of the kernels (once per device).
cudaError_t init_kernels();

// The 256-byte aligned static device array behind tpa_decode_static_scratch:
// its size, and its address on `device` (looked up once per device with that
// device current; no allocation).
size_t static_scratch_bytes();
cudaError_t static_scratch(int device, void** ptr);

}  // namespace tpa
