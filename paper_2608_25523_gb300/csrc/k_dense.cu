// Persistent dense tensor-core attention over paged KV (tcgen05 + TMEM + TMA).
//
// One launch runs a whole list of work items, each a 128-row query tile
// (128/G tokens x the G q heads of one kv head) against up to two key
// segments (runs of pages of one prefix or one suffix):
//
//  * decode, level 1: all requests of agent a share one resident prefix
//    (Sec. I: one static path of the prefix cache per agent; Sec. III,
//    Eq. 2: the prefix is paid once per agent), so the queries of all of a's
//    decode tokens are stacked and the prefix K/V streams through the tensor
//    cores once per tile instead of once per request;
//  * decode, level 2 runs in the same launch on the other CTAs (split_kv.cuh:
//    one warp per request suffix range, which also appends the step's token);
//    both levels write fp32 partials (o, lse) that the merge kernel, launched
//    as a programmatic dependent of this one, combines exactly;
//  * chunked causal prefill (Sec. VI cites chunked prefill): a tile of one
//    request's chunk attends to the whole prefix and causally to the
//    request's own suffix, writing final outputs directly.
//
// A CTA owns one SM (226 KB of shared memory).  The first n_dense_ctas CTAs
// walk their share of the dense items (longest first, snake order), holding
// 512 TMEM columns, and then join the split-KV work; the rest run split-KV
// warps from the start on the same shared memory.
//   warps 0, 10 TMA producers of K and V: tiles of 8 pages into a 3-stage
//               ring each, running ahead across item boundaries; lane i
//               loads page i's id three tiles ahead.  A full tile on 8
//               consecutive pages is one 128B-swizzled box of the kv head's
//               page-run view, otherwise each lane issues its page's box
//   warp 1      TMEM owner; one lane issues tcgen05.mma, whichever of QK /
//               PV is ready first (QK may run two tiles ahead of PV):
//                 S_j = Q K_j^T  (M=128, N=128 keys, K=d)   into TMEM S[j%2]
//                 O  += P_j V_j  (M=128, N=d, K=128 keys)   into TMEM O, with P_j
//                                read from TMEM P[j%2] and V_j from shared memory
//   warps 2..9  warp w owns TMEM lane quarter w % 4 (rows 32(w%4)..+31) and
//               key half (w-2)/4.  Per tile: read S, take the full-row max
//               (both warps of a pair, so their running max agrees without
//               synchronising; the load-with-maximum form of tcgen05.ld
//               gives it for a full tile), write P (bf16) for their key half into
//               TMEM, rescale O in
//               TMEM only when the max grew by more than 2^8 (otherwise the
//               stale max stays the reference, which is exact: it is only a
//               stabiliser); then the item's epilogue.  The next item's Q
//               rows are copied in (cp.async) as soon as the current item's
//               last QK has completed, so its first QKs overlap the epilogue.
// Every mbarrier wait is bounded.  On a timeout the CTA records a status bit
// and every role still walks the same item/tile sequence (skipping the work,
// never a named barrier), drains its copies and MMAs, frees TMEM and returns.
#include "kernels.h"
#include "ptx.cuh"
#include "dense_common.cuh"
#include "split_kv.cuh"

namespace tpa {

namespace {

using namespace dense_detail;


constexpr int kThreads = 352;               // K producer, MMA, 8 softmax warps, V producer
constexpr int kWarpV = 10;                  // the V producer warp
constexpr int kSoftmax = 256;

__device__ __forceinline__ void softmax_bar() { asm volatile("bar.sync 2, 256;" ::: "memory"); }

constexpr int kSplitWarps = 8;
constexpr int kSplitStages = 3;

template <int D>
struct DenseCfg {
  static constexpr int NCH = D / 64;               // 64-dim chunks of a 128-byte row
  static constexpr int kChunk = 128 * 128;         // one chunk of a 128-row/128-key tile
  static constexpr int kQBytes = NCH * kChunk;     // Q   [chunk][row][128 B]
  static constexpr int kKVBytes = NCH * kChunk;    // K,V 8 pages, see kv_off
  static constexpr int kPageBytes = NCH * 2048;    // one page of one kv head
  static constexpr int kGroup = NCH * 1024;        // stride of 8-key groups
  static constexpr int kStages = 3;   // K and V ring depth
  static constexpr int kOffQ = 0;
  static constexpr int kOffK = kOffQ + kQBytes;
  static constexpr int kOffV = kOffK + kStages * kKVBytes;
  static constexpr int kOffBar = kOffV + kStages * kKVBytes;
  static constexpr int kNumBars = 22;
  static constexpr int kOffL = kOffBar + kNumBars * 8;   // partial row sums [2][128]
  static constexpr int kOffMisc = kOffL + 2 * 128 * 4;
  // split-KV CTAs of the same launch lay out their page rings from the start
  static constexpr int kSplitSmem =
      kSplitWarps * (SplitCfg<D, kSplitStages>::kWarpBytes + kSplitStages * 8) + 16;
  static constexpr int kSmem = 1024 + (kOffMisc + 64 > kSplitSmem ? kOffMisc + 64 : kSplitSmem);
  static constexpr uint32_t kTmemCols = 512;
  // TMEM: S double buffer, O, then P double buffer (bf16, two per column)
  static constexpr uint32_t kColS0 = 0, kColS1 = 128, kColO = 256, kColP = 256 + D;
};

// barrier slots
enum { B_KFULL = 0, B_KEMPTY = 3, B_VFULL = 6, B_VEMPTY = 9, B_SFULL = 12, B_SFREE = 14,
       B_PFULL = 16, B_PVDONE = 18, B_QFULL = 20, B_DRAIN = 21 };

// Split-KV role of a CTA of the same launch: 8 independent warps, each with
// a 3-stage TMA page ring in the shared memory the dense role would use.

// first: the CTA starts here (its programmatic-dependency wait is still to
// come); otherwise it joins after its dense items, having waited already.
template <int D, int G>
__device__ __forceinline__ void split_role(const DenseParams& p, uint8_t* smem, bool first) {
  using W = SplitCfg<D, kSplitStages>;
  static_assert(kSplitWarps * (W::kWarpBytes + kSplitStages * 8) + 16 <= DenseCfg<D>::kSmem - 1024,
                "split-KV rings fit in the launch's shared memory");
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= kSplitWarps) return;
  uint8_t* ring = smem + warp * W::kWarpBytes;
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + kSplitWarps * W::kWarpBytes) + warp * kSplitStages;
  volatile int* abort_flag = reinterpret_cast<volatile int*>(
      smem + kSplitWarps * (W::kWarpBytes + kSplitStages * 8));
  if (threadIdx.x == 0) *abort_flag = 0;
  if (lane == 0) {
    for (int s = 0; s < kSplitStages; ++s) mbar_init(&bars[s], 1);
    fence_mbar_init();
  }
  asm volatile("bar.sync 3, 256;" ::: "memory");
  if (threadIdx.x == 0) {
    prefetch_tmap(&p.tmap_k);
    prefetch_tmap(&p.tmap_v);
  }
  // the wait for the kernel before this one comes inside the warp loop, once
  // the first item is resolved from the plan (which no earlier kernel writes)
  SplitArgs a{&p.tmap_k, &p.tmap_v, p.q, p.part_o, p.part_lse, nullptr, p.n_sitems,
              p.stoks, p.full_prefix, p.tail_order, p.n_stok, p.n_full, p.split_keys, p.pages,
              p.squeue, p.status, p.num_pages, p.hq, p.hkv, p.scale_log2, p.k_new, p.v_new,
              p.k_pool, p.v_pool, p.part_slots, 1};
  split_warp_loop<D, G, kSplitStages>(a, ring, bars, abort_flag, lane, first);
}

template <int D, int G>
__global__ void __launch_bounds__(kThreads, 1) dense_kernel(const __grid_constant__ DenseParams p) {
  using C = DenseCfg<D>;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kOffBar);
  float* lpart = reinterpret_cast<float*>(smem + C::kOffL);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);

  pdl_trigger();  // the merge kernel after a decode may become resident now
  if (p.plan_flag) {
    // the plan came on another stream: wait for its flag (bounded)
    const int got = threadIdx.x == 0 ? wait_flag64(p.plan_flag, p.plan_seq) : 1;
    if (!__syncthreads_and(got)) {
      if (threadIdx.x == 0) atomicOr(p.status, kStatusPlanTimeout);
      return;
    }
  }
  if (static_cast<int>(blockIdx.x) >= p.n_dense_ctas) {
    split_role<D, G>(p, smem, true);
    return;
  }
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_ctas = p.n_dense_ctas;

  // ---------------------------------------------------------------- setup
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < C::kStages; ++i) {
      mbar_init(&bars[B_KFULL + i], 1);
      mbar_init(&bars[B_KEMPTY + i], 1);
      mbar_init(&bars[B_VFULL + i], 1);
      mbar_init(&bars[B_VEMPTY + i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars[B_SFULL + i], 1);
      mbar_init(&bars[B_SFREE + i], kSoftmax);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&bars[B_PFULL + i], kSoftmax);
      mbar_init(&bars[B_PVDONE + i], 1);
    }
    mbar_init(&bars[B_QFULL], kSoftmax);
    mbar_init(&bars[B_DRAIN], 1);
    fence_mbar_init();
    prefetch_tmap(&p.tmap_k);
    prefetch_tmap(&p.tmap_v);
  }
  if (threadIdx.x >= 32 && threadIdx.x < 32 + 2 * p.hkv && p.run_maps)
    prefetch_tmap(p.run_maps + (threadIdx.x - 32));
  if (warp == 1) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;
  // The setup above touches only this CTA's shared and tensor memory; from
  // here on the kernel before this one (if this is its programmatic
  // dependent) must have completed.
  pdl_wait();

  if (warp == 0 || warp == kWarpV) {
    // ------------------------------------------------------------ producers
    // Warp 0 streams K, warp kWarpV streams V, each through its own 3-stage
    // ring, so K runs ahead of the PV pipeline.
    const bool is_v = warp == kWarpV;
    const bool pok = kv_producer<D, C::kStages>(
        p, p.items, p.n_items, n_ctas, is_v ? &p.tmap_v : &p.tmap_k, p.run_maps + (is_v ? p.hkv : 0),
        smem + (is_v ? C::kOffV : C::kOffK), bars + (is_v ? B_VFULL : B_KFULL),
        bars + (is_v ? B_VEMPTY : B_KEMPTY), !is_v, abort_flag, lane);
    if (!pok && lane == 0) atomicOr(p.status, kStatusDenseTimeout);
  } else if (warp == 1) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = umma_idesc_bf16(128, 128, false, false);
      constexpr uint32_t idesc_pv = umma_idesc_bf16(128, D, false, true);
      const uint32_t qbase = smem_u32(smem + C::kOffQ);
      const uint32_t kbase0 = smem_u32(smem + C::kOffK);
      const uint32_t vbase0 = smem_u32(smem + C::kOffV);
      auto issue_qk = [&](int g) {
        const int s = g & 1;            // S buffer
        const int ks = g % C::kStages;  // K stage
        tc_fence_after();
        const uint32_t kb = kbase0 + ks * C::kKVBytes;
        const uint32_t scol = s ? C::kColS1 : C::kColS0;
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk) {
          const uint64_t a = umma_sdesc(qbase + (kk >> 2) * C::kChunk + (kk & 3) * 32, 16, 1024);
          const uint64_t b = umma_sdesc(kb + (kk >> 2) * 1024 + (kk & 3) * 32, 16, C::kGroup);
          umma_bf16_ss(tmem + scol, a, b, idesc_qk, kk > 0 ? 1u : 0u);
        }
        umma_commit(&bars[B_SFULL + s]);
        umma_commit(&bars[B_KEMPTY + ks]);
      };
      auto issue_pv = [&](int g, bool first) {
        const int ks = g % C::kStages;  // V stage
        tc_fence_after();
        const uint32_t vb = vbase0 + ks * C::kKVBytes;
        const uint32_t pcol = tmem + C::kColP + (g & 1) * 64;  // P from TMEM, 8 columns per 16 keys
#pragma unroll
        for (int kk = 0; kk < 8; ++kk) {
          const uint64_t b = umma_sdesc(vb + kk * C::kPageBytes, 1024, C::kGroup);
          umma_bf16_ts(tmem + C::kColO, pcol + kk * 8, b, idesc_pv, (!first || kk > 0) ? 1u : 0u);
        }
        umma_commit(&bars[B_PVDONE + (g & 1)]);
        umma_commit(&bars[B_VEMPTY + ks]);
      };
      bool ok = true;
      int gt = 0;
      for (int k = 0; ok; ++k) {
        const int idx = item_of(k, n_ctas);
        if (idx >= p.n_items) break;
        const int ntiles = p.items[idx].n_tiles;
        // Q of this item is copied in by the softmax warps once the previous
        // item's last QK has completed; O is overwritten only by this item's
        // first PV, whose P comes after they have read the previous O out
        if (!mbar_wait(&bars[B_QFULL], k & 1, abort_flag)) { ok = false; break; }
        // Issue whichever is ready first: QK of the next tile (K landed, its S
        // buffer released by the softmax two tiles back) or PV of the oldest
        // tile whose P is written (and V landed).  PVs stay in tile order.
        int nq = 0, np = 0;
        unsigned long long t_last = global_ns();
        while (ok && np < ntiles) {
          bool progressed = false;
          if (nq < ntiles && nq <= np + 2) {
            const int g = gt + nq;
            if (mbar_test(&bars[B_KFULL + g % C::kStages], (g / C::kStages) & 1) &&
                mbar_test(&bars[B_SFREE + (g & 1)], ((g >> 1) & 1) ^ 1u)) {
              issue_qk(g);
              ++nq;
              progressed = true;
            }
          }
          if (np < nq) {
            const int g = gt + np;
            if (mbar_test(&bars[B_PFULL + (g & 1)], (g >> 1) & 1) &&
                mbar_test(&bars[B_VFULL + g % C::kStages], (g / C::kStages) & 1)) {
              issue_pv(g, np == 0);
              ++np;
              progressed = true;
            }
          }
          if (progressed) {
            t_last = global_ns();
          } else if (*abort_flag || global_ns() - t_last > kWaitLimitNs) {
            ok = false;
          }
        }
        gt += ntiles;
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(p.status, kStatusDenseTimeout);
      }
      // all MMAs issued by this thread complete before TMEM is released
      umma_commit(&bars[B_DRAIN]);
      volatile int never = 0;
      (void)mbar_wait(&bars[B_DRAIN], 0, &never);
    }
    // lanes 1..31 wait here for the issuing lane: an aligned CTA barrier
    // must see the warp converged, or it may release before every TMEM
    // reader is done
    __syncwarp();
  } else {
    // ------------------------------------------------------------ softmax
    // Every softmax thread walks the same items and tiles even after a
    // failure (ok == false skips the work): the named barriers below must be
    // reached the same number of times by all 256 threads.
    const int sw = warp - 2;                 // softmax warp index 0..7
    const int half = sw >> 2;                // key half (and O column half)
    const int row = 32 * (warp & 3) + lane;  // TMEM lane quarter = warp % 4
    const int tok = row / G;
    const uint32_t lane_base = static_cast<uint32_t>(32 * (warp & 3)) << 16;
    const int own = half * 64;   // first S column of this thread's key half
    const int other = 64 - own;
    const float sc = p.scale_log2;
    bool ok = true;
    // warp-uniform outcome, so .sync.aligned tcgen05 ops never see a split warp
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      if (!ok) return false;
      if (__all_sync(0xffffffffu, mbar_wait(bar, parity, abort_flag))) return true;
      *abort_flag = 1;  // let the other roles stop waiting too
      return false;
    };
    // This thread's half of its Q row for an item (zero for padding rows),
    // copied straight into the swizzled Q tile.  The next item's copy starts
    // as soon as this item's last QK has completed, and Q_FULL is signalled
    // before this item's epilogue, so the next item's first QKs overlap it.
    auto load_q = [&](const DenseTok& t, int kv_head, bool valid) {
      constexpr int U = D / 16;
      const int head = kv_head * G + row % G;
      const __nv_bfloat16* src =
          p.q + (valid ? (static_cast<int64_t>(t.q_row) * p.hq + head) * D + half * (D / 2) : 0);
      uint8_t* qs = smem + C::kOffQ;
#pragma unroll
      for (int u = 0; u < U; ++u) {
        const int gu = half * U + u;
        cp_async_16(qs + (gu >> 3) * C::kChunk + swz128(row, gu & 7), src + 8 * u, valid ? 16u : 0u);
      }
      cp_async_commit();
    };
    auto q_ready = [&]() {
      cp_async_wait_all();
      fence_proxy_async();
      mbar_arrive(&bars[B_QFULL]);
    };
    constexpr DenseTok kNoTok = {0, 0x7fffffff, 0, 0};
    // descriptors of the item after the current one, loaded an item ahead
    DenseTok dt_next = kNoTok;
    int kv_next = 0;
    bool valid_next = false;
    {
      const int idx0 = item_of(0, n_ctas);
      if (idx0 < p.n_items) {
        kv_next = p.items[idx0].kv_head;
        valid_next = tok < p.items[idx0].n_tok;
        if (valid_next) dt_next = p.toks[p.items[idx0].tok_base + tok];
        load_q(dt_next, kv_next, valid_next);
        q_ready();
      }
    }
    int gt = 0;
    for (int k = 0;; ++k) {
      const int idx = item_of(k, n_ctas);
      if (idx >= p.n_items) break;
      const DenseItem item = p.items[idx];
      const int ntiles = item.n_tiles;
      const bool row_valid = valid_next;
      const DenseTok dt = dt_next;
      const int head = item.kv_head * G + row % G;
      const int idx_n = item_of(k + 1, n_ctas);
      const bool has_next = idx_n < p.n_items;
      dt_next = kNoTok;
      valid_next = false;
      if (has_next) {
        kv_next = p.items[idx_n].kv_head;
        valid_next = tok < p.items[idx_n].n_tok;
        if (valid_next) dt_next = p.toks[p.items[idx_n].tok_base + tok];
      }
      bool q_issued = false;
      float m_run = -INFINITY, l_run = 0.f;
      for (int j = 0; j < ntiles && ok; ++j) {
        const TileInfo t = tile_at(item, j);
        const int g = gt + j;
        const int s = g & 1;
        if (!wait_all(&bars[B_SFULL + s], (g >> 1) & 1)) { ok = false; break; }
        if (j == ntiles - 1 && has_next) {
          // the item's last QK has completed: its Q tile is free
          load_q(dt_next, kv_next, valid_next);
          q_issued = true;
        }
        tc_fence_after();
        const uint32_t scol = tmem + lane_base + (s ? C::kColS1 : C::kColS0);
        // both key halves of the row, each 32 columns with its maximum taken
        // by the TMEM load itself
        float x[64], y[64], cmax[4];
        tmem_ld32_max(scol + own, x, cmax[0]);
        tmem_ld32_max(scol + own + 32, x + 32, cmax[1]);
        tmem_ld32_max(scol + other, y, cmax[2]);
        tmem_ld32_max(scol + other + 32, y + 32, cmax[3]);
        tmem_wait_ld();
        tc_fence_before();
        mbar_arrive(&bars[B_SFREE + s]);

        int lim = t.nvalid;
        if (t.causal && dt.causal_pos < t.key0 + lim) {
          const int c = dt.causal_pos - t.key0 + 1;
          lim = c > 0 ? c : 0;
        }
        float mraw = fmaxf(fmax3f(cmax[0], cmax[1], cmax[2]), cmax[3]);
        if (lim < 128) {
          // keys past the range or the causal limit: masked, and the full-row
          // max taken again over the keys that remain (8 chains of 3-input max)
#pragma unroll
          for (int n = 0; n < 64; ++n) {
            x[n] = own + n < lim ? x[n] : -INFINITY;
            y[n] = other + n < lim ? y[n] : -INFINITY;
          }
          float acc[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) acc[i] = fmax3f(x[i], x[i + 8], y[i]);
#pragma unroll
          for (int kk = 16; kk < 64; kk += 8)
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = fmax3f(acc[i], x[kk + i], y[kk + i - 8]);
#pragma unroll
          for (int i = 0; i < 8; ++i) acc[i] = fmaxf(acc[i], y[56 + i]);
          mraw = fmax3f(fmax3f(acc[0], acc[1], acc[2]), fmax3f(acc[3], acc[4], acc[5]),
                        fmaxf(acc[6], acc[7]));
        }
        const float mx = mraw * sc;  // sc > 0: max of the scaled scores
        const float m_new = fmaxf(m_run, mx);
        const bool grow = m_new > m_run + kRescaleThreshold;
        const float m_use = grow ? m_new : m_run;
        const float alpha = grow ? fast_exp2(m_run - m_use) : 1.f;
        const float nref = m_use == -INFINITY ? 0.f : -m_use;
        // p = 2^(s * sc - m) over this thread's half: packed FMAs, MUFU ex2,
        // 8 independent partial sums
        float sacc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int n = 0; n < 64; n += 2) {
          ffma2(x[n], x[n + 1], x[n], x[n + 1], sc, sc, nref, nref);
          x[n] = fast_exp2(x[n]);
          x[n + 1] = fast_exp2(x[n + 1]);
        }
#pragma unroll
        for (int n = 0; n < 64; n += 16)
#pragma unroll
          for (int i = 0; i < 8; i += 2) {
            fadd2(sacc[i], sacc[i + 1], sacc[i], sacc[i + 1], x[n + 2 * i], x[n + 2 * i + 1]);
            fadd2(sacc[i], sacc[i + 1], sacc[i], sacc[i + 1], x[n + 2 * i + 2], x[n + 2 * i + 3]);
          }
        const float rsum = ((sacc[0] + sacc[1]) + (sacc[2] + sacc[3])) +
                           ((sacc[4] + sacc[5]) + (sacc[6] + sacc[7]));
        // P buffer g % 2 was last read by PV(g - 2)
        if (g >= 2 && !wait_all(&bars[B_PVDONE + (g & 1)], ((g >> 1) & 1) ^ 1u)) { ok = false; break; }
        // rescale this half of the O row when the reference max moved (with real
        // content), after PV(g - 1) has finished accumulating into it
        if (j > 0 && __any_sync(0xffffffffu, grow && m_run > -INFINITY)) {
          if (!wait_all(&bars[B_PVDONE + ((g - 1) & 1)], ((g - 1) >> 1) & 1)) { ok = false; break; }
          tc_fence_after();
          {
#pragma unroll 1
            for (int c = 0; c < D / 64; ++c) {
              float o[32];
              const uint32_t oc = tmem + lane_base + C::kColO + half * (D / 2) + 32 * c;
              tmem_ld32(oc, o);
              tmem_wait_ld();
#pragma unroll
              for (int i = 0; i < 32; ++i) o[i] *= alpha;
              tmem_st32(oc, o);
            }
            tmem_wait_st();
          }
        }
        l_run = l_run * alpha + rsum;
        m_run = m_use;
        if (t.nvalid < 128) {
          // keys past the range: zero their V rows (stale data may not be finite);
          // each half zeroes its own 64-dim chunk (or its half of the only chunk)
          if (!wait_all(&bars[B_VFULL + g % C::kStages], (g / C::kStages) & 1)) { ok = false; break; }
          if (row >= t.nvalid) {
            uint8_t* vst = smem + C::kOffV + (g % C::kStages) * C::kKVBytes;
            if (C::NCH == 2) {
#pragma unroll
              for (int u = 0; u < 8; ++u)
                *reinterpret_cast<uint4*>(vst + kv_off<C::NCH>(row, 8 * half + u)) =
                    make_uint4(0, 0, 0, 0);
            } else {
#pragma unroll
              for (int u = 0; u < 4; ++u)
                *reinterpret_cast<uint4*>(vst + kv_off<C::NCH>(row, 4 * half + u)) =
                    make_uint4(0, 0, 0, 0);
            }
          }
        }
        // this half of the P row (keys own .. own+63) into TMEM P buffer g % 2:
        // 32 columns of two bf16 each, in key order
        {
          float pk[32];
#pragma unroll
          for (int u = 0; u < 32; ++u) pk[u] = __uint_as_float(pack_bf16(x[2 * u], x[2 * u + 1]));
          tmem_st32(tmem + lane_base + C::kColP + (g & 1) * 64 + half * 32, pk);
          tmem_wait_st();
        }
        if (t.nvalid < 128) fence_proxy_async();  // the zeroed V rows, before the PV reads them
        tc_fence_before();
        mbar_arrive(&bars[B_PFULL + (g & 1)]);
      }

      if (has_next) {
        if (!q_issued) load_q(dt_next, kv_next, valid_next);
        q_ready();
      }

      // ---------------------------------------------------------- epilogue
      lpart[half * 128 + row] = l_run;
      softmax_bar();
      const float l_tot = lpart[row] + lpart[128 + row];
      if (ntiles > 0) {
        const int gl = gt + ntiles - 1;  // the item's last PV
        if (!wait_all(&bars[B_PVDONE + (gl & 1)], (gl >> 1) & 1)) ok = false;
      }
      const float inv = l_tot > 0.f ? 1.f / l_tot : 0.f;
      const float lse = l_tot > 0.f ? (m_run + __log2f(l_tot)) * kLn2 : -INFINITY;
      const int64_t slot = dt.slot_base + static_cast<int64_t>(head) * dt.n_slots + item.split;
      // a partial slot outside the partial buffer is not written (status bit)
      const bool slot_ok = item.out_mode != 0 || (slot >= 0 && slot < p.part_slots);
      if (ok && row_valid && !slot_ok) atomicOr(p.status, kStatusBadSlot);
      if (ok) {
        tc_fence_after();
#pragma unroll 1
        for (int c = 0; c < D / 64; ++c) {
          float o[32];
          const int col = half * (D / 2) + 32 * c;
          tmem_ld32(tmem + lane_base + C::kColO + col, o);
          tmem_wait_ld();
          if (row_valid && slot_ok) {
            if (item.out_mode == 0) {
              float4* dst = reinterpret_cast<float4*>(p.part_o + slot * D + col);
#pragma unroll
              for (int i = 0; i < 8; ++i)
                dst[i] = make_float4(o[4 * i] * inv, o[4 * i + 1] * inv, o[4 * i + 2] * inv,
                                     o[4 * i + 3] * inv);
            } else {
              uint4* dst = reinterpret_cast<uint4*>(
                  p.out + (static_cast<int64_t>(dt.q_row) * p.hq + head) * D + col);
#pragma unroll
              for (int i = 0; i < 4; ++i) {
                uint4 v;
                v.x = pack_bf16(o[8 * i + 0] * inv, o[8 * i + 1] * inv);
                v.y = pack_bf16(o[8 * i + 2] * inv, o[8 * i + 3] * inv);
                v.z = pack_bf16(o[8 * i + 4] * inv, o[8 * i + 5] * inv);
                v.w = pack_bf16(o[8 * i + 6] * inv, o[8 * i + 7] * inv);
                dst[i] = v;
              }
            }
          }
        }
        tc_fence_before();
        if (row_valid && slot_ok && half == 0) {
          if (item.out_mode == 0) p.part_lse[slot] = lse;
          else p.lse[static_cast<int64_t>(dt.q_row) * p.hq + head] = lse;
        }
      }
      gt += ntiles;
    }
    cp_async_wait_all();
    if (!ok) {
      *abort_flag = 1;
      atomicOr(p.status, kStatusDenseTimeout);
    }
    tc_fence_before();
  }

  // ---------------------------------------------------------------- teardown
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
  // Decode: this CTA's dense items are done (every copy it issued has been
  // consumed), so its warps join the split-KV work on the same shared memory.
  if (p.n_sitems > 0) {
    __syncthreads();
    if (!*abort_flag) split_role<D, G>(p, smem, false);
  }
}

template <int D, int G>
cudaError_t launch_dense_t(const DenseParams& p, int n_split_ctas, bool dependent,
                           cudaStream_t stream) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(static_cast<unsigned>(p.n_dense_ctas + n_split_ctas));
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = DenseCfg<D>::kSmem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = dependent ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, dense_kernel<D, G>, p);
}

}  // namespace

cudaError_t launch_dense(const DenseParams& p, int n_split_ctas, int head_dim, int group,
                         bool dependent, cudaStream_t stream) {
  if (p.n_dense_ctas + n_split_ctas <= 0) return cudaSuccess;
  if (head_dim == 128 && group == 4) return launch_dense_t<128, 4>(p, n_split_ctas, dependent, stream);
  if (head_dim == 128 && group == 8) return launch_dense_t<128, 8>(p, n_split_ctas, dependent, stream);
  if (head_dim == 64 && group == 4) return launch_dense_t<64, 4>(p, n_split_ctas, dependent, stream);
  if (head_dim == 64 && group == 8) return launch_dense_t<64, 8>(p, n_split_ctas, dependent, stream);
  return cudaErrorInvalidValue;
}

cudaError_t init_dense_kernels() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(dense_kernel<128, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                DenseCfg<128>::kSmem)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(dense_kernel<128, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                DenseCfg<128>::kSmem)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(dense_kernel<64, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                DenseCfg<64>::kSmem)) != cudaSuccess)
    return e;
  return cudaFuncSetAttribute(dense_kernel<64, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              DenseCfg<64>::kSmem);
}

}  // namespace tpa
