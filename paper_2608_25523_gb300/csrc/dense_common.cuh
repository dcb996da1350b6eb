// Pieces shared by the two tcgen05 attention kernels (k_dense.cu: 128-row
// tiles, decode level 1 and prefill; k_prefill.cu: pairs of 128-row tiles,
// chunked prefill): the key-tile walk of a work item, the item order of a
// persistent CTA and the TMA producer that streams K or V tiles of 8 pages
// through a shared-memory ring.
#pragma once
#include "kernels.h"
#include "ptx.cuh"

namespace tpa {
namespace dense_detail {

constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// A K or V tile of 128 keys (8 pages of one kv head) in shared memory:
// [page][8-key half][64-dim chunk][8 rows][128 B], 128B-swizzled, so that
// each 8 x 128 B block is one swizzle atom.
template <int D>
struct KVTile {
  static constexpr int NCH = D / 64;             // 64-dim chunks of a 128-byte row
  static constexpr int kChunk = 128 * 128;       // one chunk of a 128-row/128-key tile
  static constexpr int kBytes = NCH * kChunk;    // the whole tile
  static constexpr int kPageBytes = NCH * 2048;  // one page of one kv head
  static constexpr int kGroup = NCH * 1024;      // stride of 8-key groups
};

struct TileInfo {
  int key0;      // first key of the tile within its segment
  int nvalid;    // keys of the tile inside the range (1..128)
  int causal;
  int page_off;  // page-list index of the tile's first page
};

// Key tile j of an item: its first segment's tiles, then its second's.
__device__ __forceinline__ TileInfo tile_at(const DenseItem& it, int j) {
  const int t0 = it.seg_k1[0] > it.seg_k0[0] ? (it.seg_k1[0] - it.seg_k0[0] + 127) / 128 : 0;
  const int seg = j < t0 ? 0 : 1;
  const int jj = j < t0 ? j : j - t0;
  TileInfo t;
  t.key0 = it.seg_k0[seg] + 128 * jj;
  const int rest = it.seg_k1[seg] - t.key0;
  t.nvalid = rest < 128 ? rest : 128;
  t.causal = it.seg_causal[seg];
  t.page_off = it.seg_pages[seg] + t.key0 / kPage;
  return t;
}

// k-th item of this CTA among g persistent CTAs: snake order over a
// longest-first list.
__device__ __forceinline__ int item_of(int k, int g) {
  return k * g + ((k & 1) ? g - 1 - static_cast<int>(blockIdx.x) : static_cast<int>(blockIdx.x));
}

// One warp streaming the K (or V) tiles of this CTA's items, in item and
// tile order, through an S-stage ring (full/empty mbarrier pairs, phase
// g / S of the CTA's g-th tile).  Lane i (< 8) owns page i of every tile: it
// loads that page id three tiles ahead and issues the page's TMA box, so a
// tile's boxes go out from 8 lanes at once; a full tile on 8 consecutive
// pages goes as one box of the kv head's page-run view (run_map).  Lane 0
// posts the expected byte count first.  The next item's descriptor and
// first page ids are loaded while the current one streams, so item
// boundaries add no load latency.  Returns false on a timeout (after
// letting every issued copy land).
template <int D, int S>
__device__ __forceinline__ bool kv_producer(const DenseParams& p, const DenseItem* items,
                                            int n_items, int n_ctas, const CUtensorMap* tmap,
                                            const CUtensorMap* run_map_base, uint8_t* ring,
                                            uint64_t* full, uint64_t* empty, bool report_bad,
                                            volatile int* abort_flag, int lane) {
  using T = KVTile<D>;
  int ph_last[S];
#pragma unroll
  for (int s = 0; s < S; ++s) ph_last[s] = -1;
  bool pok = true;
  auto wait_all = [&](uint64_t* bar, uint32_t parity) {
    return __all_sync(0xffffffffu, mbar_wait(bar, parity, abort_flag)) != 0;
  };
  auto page_id = [&](const DenseItem& it, int j) -> int32_t {  // raw; validated when used
    if (j >= it.n_tiles) return 0;
    const TileInfo t = tile_at(it, j);
    return lane < (t.nvalid + kPage - 1) / kPage ? __ldg(p.pages + t.page_off + lane) : 0;
  };
  DenseItem item{};
  int32_t f0 = 0, f1 = 0, f2 = 0;
  if (item_of(0, n_ctas) < n_items) {
    item = items[item_of(0, n_ctas)];
    f0 = page_id(item, 0);
    f1 = page_id(item, 1);
    f2 = page_id(item, 2);
  }
  int gt = 0;  // tiles of this CTA so far (ring position)
  for (int k = 0; pok; ++k) {
    const int idx = item_of(k, n_ctas);
    if (idx >= n_items) break;
    const int ntiles = item.n_tiles;
    const int idx_n = item_of(k + 1, n_ctas);
    const bool has_next = idx_n < n_items;
    DenseItem nitem{};
    int32_t n0 = 0, n1 = 0, n2 = 0;
    bool next_ready = false;
    int32_t pid0 = f0, pid1 = f1, pid2 = f2;  // page ids three tiles ahead
    for (int j = 0; j < ntiles; ++j, ++gt) {
      const TileInfo t = tile_at(item, j);
      const int s = gt % S;
      const uint32_t ph = (gt / S) & 1;
      const int npg = (t.nvalid + kPage - 1) / kPage;
      const uint32_t bytes = static_cast<uint32_t>(npg * T::kPageBytes);
      const int32_t pid = pid0;
      pid0 = pid1;
      pid1 = pid2;
      pid2 = page_id(item, j + 3);
      const bool bad = lane < npg && (pid < 0 || pid >= p.num_pages);
      if (__any_sync(0xffffffffu, bad) && lane == 0 && report_bad) atomicOr(p.status, kStatusBadPage);
      const int z = (bad ? 0 : pid) * p.hkv + item.kv_head;
      const int32_t pid_0 = __shfl_sync(0xffffffffu, pid, 0);
      const bool run =
          npg == 8 && __all_sync(0xffffffffu, lane >= 8 || (!bad && pid == pid_0 + lane));
      if (!wait_all(&empty[s], ph ^ 1u)) { pok = false; break; }
      if (lane == 0) mbar_arrive_expect_tx(&full[s], bytes);
      __syncwarp();
      if (run) {
        if (lane == 0)
          tma_load_5d(ring + s * T::kBytes, run_map_base + item.kv_head, &full[s], 0, 0, 0, 0, pid_0);
      } else if (lane < npg) {
        tma_load_5d(ring + s * T::kBytes + lane * T::kPageBytes, tmap, &full[s], 0, 0, 0, 0, z);
      }
      ph_last[s] = static_cast<int>(ph);
      if (has_next && j == 0) nitem = items[idx_n];
      if (has_next && j == 1) {
        n0 = page_id(nitem, 0);
        n1 = page_id(nitem, 1);
        n2 = page_id(nitem, 2);
        next_ready = true;
      }
    }
    if (has_next && !next_ready) {
      if (ntiles == 0) nitem = items[idx_n];
      n0 = page_id(nitem, 0);
      n1 = page_id(nitem, 1);
      n2 = page_id(nitem, 2);
    }
    item = nitem;
    f0 = n0;
    f1 = n1;
    f2 = n2;
  }
  if (!pok && lane == 0) *abort_flag = 1;
  __syncwarp();
  if (*abort_flag && lane == 0) {
    // let every issued copy land before the CTA's shared memory goes away
    volatile int never = 0;
#pragma unroll
    for (int s = 0; s < S; ++s)
      if (ph_last[s] >= 0) (void)mbar_wait(&full[s], ph_last[s], &never);
  }
  __syncwarp();  // the warp reaches the teardown barrier converged
  return pok;
}

}  // namespace dense_detail
}  // namespace tpa
