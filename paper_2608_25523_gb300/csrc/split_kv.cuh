// Split-KV paged attention, one warp per work item: the second level of the
// decode cascade.
//
// Every request adds a private dynamic suffix (plus its decode tokens) to
// the shared agent prefix (Sec. III, Eq. 2: d_r(t) on top of ell_a), so its
// suffix keys are read by that request alone.  A work item is the G =
// Hq/Hkv query rows of one token against one key range of one page run (a
// request suffix, or in the flat cross-check mode also a prefix); it yields
// a partial (o, lse).  In the cascade decode the item holding a request's
// last key first appends the step's token to the pool.
//
// Design (memory-bound: ~4 flop per KV byte at G=4):
//  * each page of one kv head is one TMA box per operand (128-byte swizzle)
//    landing in a per-warp ring of S stages, so loads run S pages ahead;
//  * S^T tiles use mma.sync m16n8k16 with the G query rows on the M side
//    (padded to 16) and the 16 keys of the page on N; P*V reuses the S
//    accumulators as the A operand (no shared-memory round trip); V comes
//    through ldmatrix.trans;
//  * online softmax in base 2 with fp32 accumulators;
//  * warps pull items from an atomic counter (items sorted longest first);
//    2 S pages before the current item ends a warp claims and resolves its
//    next item, appends its token and loads its page ids, and keeps its ring
//    full across the item boundary, so items cost no extra load latency,
//    while the queue's tail stays unclaimed for warps that join it late.
#pragma once
#include "kernels.h"
#include "ptx.cuh"

namespace tpa {

struct SplitArgs {
  const CUtensorMap* tmap_k;  // kernel-parameter tensor maps of the pools
  const CUtensorMap* tmap_v;
  const __nv_bfloat16* q;
  float* part_o;
  float* part_lse;
  const SuffixItem* items;    // explicit items, or null: derived from toks (below)
  int n_items;
  // derived items (cascade decode): item idx -> unit idx / hkv, kv head idx % hkv;
  // units [0, n_full) are full ranges (token found in full_prefix), the rest
  // are tails in tail_order
  const SplitTok* toks;
  const int32_t* full_prefix;  // [n_tok + 1] cumulative full ranges per token
  const int32_t* tail_order;   // tokens with a tail, longest tail first
  int n_tok, n_full, split_keys;
  const int32_t* pages;
  uint32_t* queue;
  uint32_t* status;
  int64_t num_pages;
  int hq, hkv;
  float scale_log2;
  // cascade decode only (null otherwise): in-kernel append of the step's token
  const __nv_bfloat16* k_new;
  const __nv_bfloat16* v_new;
  __nv_bfloat16* k_pool;
  __nv_bfloat16* v_pool;
  int64_t part_slots;  // entries of part_lse; a slot outside [0, part_slots) is not written
  int read_once;       // 1: every page is read by this launch once (request suffixes): its loads
                       // are marked L2 evict-first, so the partials written meanwhile stay in L2
};

template <int D, int S>
struct SplitCfg {
  static constexpr int NCH = D / 64;
  static constexpr int kPageBytes = NCH * 2048;      // one page of one kv head, K or V
  static constexpr int kStageBytes = 2 * kPageBytes;
  static constexpr int kWarpBytes = S * kStageBytes;
};

namespace split_detail {

constexpr float kLn2 = 0.6931471805599453f;

__device__ __forceinline__ float fast_exp2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// Work item `idx` (explicit, or derived from the per-token records).  Called
// by the whole warp.
__device__ __forceinline__ SuffixItem fetch_item(const SplitArgs& a, int idx) {
  if (a.items) return a.items[idx];
  const int u = idx / a.hkv;
  int tok, s, k0, k1;
  if (u < a.n_full) {
    // the token is the number of i in [1, n_tok) with full_prefix[i] <= u
    // (full_prefix is non-decreasing): the lanes test 32 entries a round
    const int lane = threadIdx.x & 31;
    tok = 0;
    for (int i0 = 1; i0 < a.n_tok; i0 += 32) {
      const int i = i0 + lane;
      tok += __popc(__ballot_sync(0xffffffffu, i < a.n_tok && __ldg(a.full_prefix + i) <= u));
    }
    s = u - __ldg(a.full_prefix + tok);
    k0 = s * a.split_keys;
    k1 = k0 + a.split_keys;
  } else {
    tok = __ldg(a.tail_order + (u - a.n_full));
    const int keys = __ldg(&a.toks[tok].keys);
    s = keys / a.split_keys;
    k0 = s * a.split_keys;
    k1 = keys;
  }
  const SplitTok t = a.toks[tok];
  SuffixItem it;
  it.q_row = t.q_row;
  it.kv_head = idx % a.hkv;
  it.pages = t.pages + k0 / kPage;
  it.n_keys = k1 - k0;
  it.slot_base = t.slot_base;
  it.n_slots = t.n_slots;
  it.split = t.split0 + s;
  it.app_src = k1 == t.keys ? t.q_row : -1;
  it.app_dst = t.app_dst;
  return it;
}

}  // namespace split_detail

// Runs work items until the queue is empty.  `ring` is this warp's S stages,
// `bars` its S initialised mbarriers (count 1).  wait_prev: the launch is a
// programmatic dependent whose wait (griddepcontrol.wait) this loop makes
// once its first item is resolved from the plan, before touching anything
// earlier kernels wrote.  Returns false after a timeout (status bit set,
// in-flight copies drained).
template <int D, int G, int S>
__device__ bool split_warp_loop(const SplitArgs& a, uint8_t* ring, uint64_t* bars,
                                volatile int* abort_flag, int lane, bool wait_prev) {
  using namespace split_detail;
  using C = SplitCfg<D, S>;
  const int gq = lane >> 2;  // mma group: query row of this lane
  const int tig = lane & 3;  // thread in group
  uint32_t it = 0;           // pages consumed by this warp so far (ring position)
  uint32_t issued = 0;       // pages issued by this warp so far (lane 0's count, broadcast)
  bool failed = false;

  // An item with its page ids: lane i holds pages i and i + 32 of its run.
  struct Work {
    SuffixItem item;
    int npg;
    int32_t pid0, pid1;
  };
  // The item and its page ids (plan data only)
  auto resolve_work = [&](int idx, Work& w) {  // whole warp
    w.item = fetch_item(a, idx);
    w.npg = (w.item.n_keys + kPage - 1) / kPage;
    w.pid0 = lane < w.npg ? __ldg(a.pages + w.item.pages + lane) : 0;
    w.pid1 = lane + 32 < w.npg ? __ldg(a.pages + w.item.pages + lane + 32) : 0;
  };
  auto append_work = [&](const Work& w) {  // whole warp
    if (w.item.app_src >= 0 && a.k_new) {
      // append the step's token to the pool before its page is loaded (its
      // page belongs to this item alone: key ranges start on page boundaries)
      constexpr int U = D / 8;  // 16-byte units of one row
      const int64_t pg = w.item.app_dst / kPage;
      if (pg >= 0 && pg < a.num_pages) {
        const int64_t src = (static_cast<int64_t>(w.item.app_src) * a.hkv + w.item.kv_head) * D;
        const int64_t dst = ((pg * a.hkv + w.item.kv_head) * kPage + w.item.app_dst % kPage) * D;
        for (int u = lane; u < 2 * U; u += 32) {
          const bool isv = u >= U;
          const int uu = isv ? u - U : u;
          const uint4 v = reinterpret_cast<const uint4*>((isv ? a.v_new : a.k_new) + src)[uu];
          reinterpret_cast<uint4*>((isv ? a.v_pool : a.k_pool) + dst)[uu] = v;
        }
      } else if (lane == 0) {
        atomicOr(a.status, kStatusBadPage);
      }
      asm volatile("fence.proxy.async.global;" ::: "memory");
      __syncwarp();
    }
  };
  auto load_work = [&](int idx, Work& w) {
    resolve_work(idx, w);
    append_work(w);
  };
  // TMA page `pg` of `w` into ring slot issued % S (whole warp; lane 0 issues)
  auto issue = [&](const Work& w, int pg) {
    int64_t pid = pg < 32   ? __shfl_sync(0xffffffffu, w.pid0, pg)
                  : pg < 64 ? __shfl_sync(0xffffffffu, w.pid1, pg - 32)
                            : static_cast<int64_t>(__ldg(a.pages + w.item.pages + pg));
    if (lane == 0) {
      const int st = static_cast<int>(issued % S);
      uint8_t* kst = ring + st * C::kStageBytes;
      uint8_t* vst = kst + C::kPageBytes;
      if (pid < 0 || pid >= a.num_pages) {
        atomicOr(a.status, kStatusBadPage);
        pid = 0;
      }
      const int z = static_cast<int>(pid * a.hkv + w.item.kv_head);
      fence_proxy_async();
      mbar_arrive_expect_tx(&bars[st], 2 * C::kPageBytes);
      if (a.read_once) {
        const uint64_t pol = l2_policy_evict_first();
        tma_load_5d_hint(kst, a.tmap_k, &bars[st], 0, 0, 0, 0, z, pol);
        tma_load_5d_hint(vst, a.tmap_v, &bars[st], 0, 0, 0, 0, z, pol);
      } else {
        tma_load_5d(kst, a.tmap_k, &bars[st], 0, 0, 0, 0, z);
        tma_load_5d(vst, a.tmap_v, &bars[st], 0, 0, 0, 0, z);
      }
    }
    ++issued;
  };
  auto claim = [&]() -> uint32_t { return lane == 0 ? atomicAdd(a.queue, 1u) : 0u; };

  // The first item is claimed and resolved from the plan before waiting for
  // the previous kernel (wait_prev); its append and page loads come after.
  int idx = __shfl_sync(0xffffffffu, static_cast<int>(claim()), 0);
  Work cur{};
  int cur_iss = 0;  // pages of cur issued
  if (idx < a.n_items) resolve_work(idx, cur);
  if (wait_prev) pdl_wait();
  if (idx < a.n_items) {
    append_work(cur);
    while (cur_iss < cur.npg && cur_iss < S) issue(cur, cur_iss++);
  }

  while (idx < a.n_items) {
    // The next item is claimed 2 S pages before this one ends (at once for a
    // short item) and resolved right away, so its page loads follow this
    // item's last pages without a gap; claiming later than that leaves the
    // queue's tail to CTAs that join it late instead of piling it up behind
    // busy warps.
    const int claim_at = cur.npg > 2 * S ? cur.npg - 2 * S : 0;
    Work nxt{};
    int nxt_iss = 0;
    int idx_n = a.n_items;
    const SuffixItem& item = cur.item;

    // Query fragments (A operand): rows >= G and the upper 8 rows are zero.
    uint32_t qa[D / 16][2];
    {
      const bool real = gq < G;
      const __nv_bfloat16* qrow =
          a.q + (static_cast<int64_t>(item.q_row) * a.hq + item.kv_head * G + (real ? gq : 0)) * D;
#pragma unroll
      for (int kk = 0; kk < D / 16; ++kk) {
        qa[kk][0] = real ? *reinterpret_cast<const uint32_t*>(qrow + 16 * kk + 2 * tig) : 0u;
        qa[kk][1] = real ? *reinterpret_cast<const uint32_t*>(qrow + 16 * kk + 8 + 2 * tig) : 0u;
      }
    }

    float o[D / 8][4];
#pragma unroll
    for (int nt = 0; nt < D / 8; ++nt) o[nt][0] = o[nt][1] = o[nt][2] = o[nt][3] = 0.f;
    float m = -INFINITY, l = 0.f;

    for (int pg = 0; pg < cur.npg; ++pg) {
      const uint32_t cnt = it + pg;
      const int st = static_cast<int>(cnt % S);
      if (!__all_sync(0xffffffffu, mbar_wait(&bars[st], (cnt / S) & 1u, abort_flag))) {
        failed = true;
        it += pg;  // first page not consumed: pages it .. issued-1 are in flight
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
      const float sc = a.scale_log2;
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
      if (pg == claim_at) {
        idx_n = __shfl_sync(0xffffffffu, static_cast<int>(claim()), 0);
        if (idx_n < a.n_items) load_work(idx_n, nxt);
      }
      // refill the slot this page freed: this item's next page, else the next item's
      if (cur_iss < cur.npg) issue(cur, cur_iss++);
      else if (nxt_iss < nxt.npg) issue(nxt, nxt_iss++);
    }
    if (failed) break;
    it += cur.npg;

    l += __shfl_xor_sync(0xffffffffu, l, 1);
    l += __shfl_xor_sync(0xffffffffu, l, 2);
    const int64_t slot =
        item.slot_base + static_cast<int64_t>(item.kv_head * G + (gq < G ? gq : 0)) * item.n_slots +
        item.split;
    const bool slot_ok = slot >= 0 && slot < a.part_slots;
    if (!__all_sync(0xffffffffu, slot_ok || gq >= G) && lane == 0) atomicOr(a.status, kStatusBadSlot);
    if (gq < G && slot_ok) {
      const float inv = 1.f / l;
      float* dst = a.part_o + slot * D;
#pragma unroll
      for (int nt = 0; nt < D / 8; ++nt)
        *reinterpret_cast<float2*>(dst + 8 * nt + 2 * tig) =
            make_float2(o[nt][0] * inv, o[nt][1] * inv);
      if (tig == 0) a.part_lse[slot] = (m + __log2f(l)) * kLn2;
    }

    idx = idx_n;
    cur = nxt;
    cur_iss = nxt_iss;
    while (issued - it < static_cast<uint32_t>(S) && cur_iss < cur.npg) issue(cur, cur_iss++);
  }

  if (failed) {
    if (lane == 0) {
      atomicOr(a.status, kStatusSuffixTimeout);
      *abort_flag = 1;
      // every issued page must land before the CTA exits
      volatile int never = 0;
      for (uint32_t c = it; c < issued; ++c) {
        const int st = static_cast<int>(c % S);
        (void)mbar_wait(&bars[st], (c / S) & 1u, &never);
      }
    }
    __syncwarp();
  }
  return !failed;
}

}  // namespace tpa
