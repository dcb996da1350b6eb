// Chunked causal prefill on the tensor cores, two query tiles per CTA
// (tcgen05 + TMEM + TMA).
//
// A chunk's new tokens attend to their agent's whole resident prefix and,
// causally, to their own request's suffix (its earlier chunks and the chunk
// itself, appended to the pool just before).  A work item is a pair of
// 128-row query tiles -- 256/G consecutive tokens of one chunk x the G q heads
// of one kv head, tile A the first 128/G tokens and tile B the next -- that
// share every K/V tile of the item's key range (prefix pages, then suffix
// pages up to the item's last token).  Sharing halves the K/V traffic of
// shared memory and L2 per query row, and the two tiles give the tensor
// pipe independent work: while the softmax of one tile runs, the other
// tile's PV and next QK execute, so the chain QK -> softmax -> PV of a
// single tile no longer leaves the pipe idle.
//
// A CTA owns one SM and walks its share of the items (longest first, snake
// order):
//   warps 0..3  softmax of tile A, warps 4..7 of tile B (below)
//   warps 8, 10 TMA producers of K (3-stage ring) and V (2-stage ring), as in
//               the single-tile kernel (dense_common.cuh); warp 11 idles
//   warp 9      TMEM owner; one lane issues, in this fixed order per key
//               tile j (after S_A(0), S_B(0) of the item):
//                 O_A += P_A(j) V_j,  S_A(j+1) = Q_A K_{j+1}^T,
//                 O_B += P_B(j) V_j,  S_B(j+1) = Q_B K_{j+1}^T
//               (M = 128 rows; QK: N = 128 keys, K = d; PV: N = d, K = 128
//               keys with P read from TMEM).  The tensor pipe runs a CTA's
//               MMAs in issue order, so S_X(j+1) overwrites P_X(j) only after
//               PV_X(j) has read it.
//   softmax     warp w owns TMEM lane quarter w % 4 and each thread one
//               query row of its tile (a whole warpgroup per tile), all 128
//               keys of a tile: read S (the load-with-maximum form of
//               tcgen05.ld gives the row max of a full tile; a ragged or
//               causal tile takes it again after masking), P = 2^(s - m) as bf16 into
//               the first 64 columns of its S buffer, row sum; O is rescaled
//               in TMEM only when the max grew by more than 2^8 (the stale max
//               stays the reference otherwise, which is exact: it is only a
//               stabiliser); then the item's epilogue (bf16 out, fp32 lse).
//               The next item's Q rows are copied in (cp.async) as soon as
//               the tile's last QK has completed.
// TMEM (512 columns): S_A [0,128), S_B [128,256), O_A [256,256+d),
// O_B [256+d,256+2d).
// Registers: the launch gives every thread kLaunchRegs; the producer/MMA
// warpgroup then drops to kLowRegs and the two softmax warpgroups rise to
// kHighRegs (a whole S row, 128 floats, stays in registers), the same total.
// Every mbarrier wait is bounded; on a timeout the CTA records a status bit,
// every role stops, drains its copies and MMAs, frees TMEM and returns.
#include "dense_common.cuh"

namespace tpa {

namespace {

using namespace dense_detail;

constexpr int kThreads = 384;  // softmax warpgroups A and B, then K producer, MMA, V producer, idle
constexpr int kWarpK = 8, kWarpMma = 9, kWarpV = 10;
constexpr int kTileThreads = 128;  // softmax threads of one query tile
constexpr int kLaunchRegs = 168;   // what ptxas assigns under __launch_bounds__(384, 1)
constexpr int kLowRegs = 104, kHighRegs = 200;
static_assert(2 * 128 * kHighRegs + 128 * kLowRegs == kThreads * kLaunchRegs,
              "the register split redistributes exactly the launch allocation");

template <int D>
struct PairCfg {
  using T = KVTile<D>;
  static constexpr int kStagesK = 3;
  static constexpr int kStagesV = D == 128 ? 2 : 3;
  static constexpr int kQBytes = T::NCH * T::kChunk;  // one 128-row Q tile [chunk][row][128 B]
  static constexpr int kOffQ = 0;                     // Q_A, then Q_B
  static constexpr int kOffK = 2 * kQBytes;
  static constexpr int kOffV = kOffK + kStagesK * T::kBytes;
  static constexpr int kOffBar = kOffV + kStagesV * T::kBytes;
  // barriers: K full/empty, V full/empty, then per tile X: S full, P full,
  // PV done, Q full; then the drain barrier
  static constexpr int B_KFULL = 0;
  static constexpr int B_KEMPTY = B_KFULL + kStagesK;
  static constexpr int B_VFULL = B_KEMPTY + kStagesK;
  static constexpr int B_VEMPTY = B_VFULL + kStagesV;
  static constexpr int B_SFULL = B_VEMPTY + kStagesV;  // + X
  static constexpr int B_PFULL = B_SFULL + 2;
  static constexpr int B_PVDONE = B_PFULL + 2;
  static constexpr int B_QFULL = B_PVDONE + 2;
  static constexpr int B_DRAIN = B_QFULL + 2;
  static constexpr int kNumBars = B_DRAIN + 1;
  static constexpr int kOffMisc = kOffBar + kNumBars * 8;
  static constexpr int kSmem = 1024 + kOffMisc + 64;
  static constexpr uint32_t kTmemCols = 512;
  static constexpr uint32_t kColO = 256;  // O_X at kColO + X * D
};

template <int D, int G>
__global__ void __launch_bounds__(kThreads, 1) prefill_pair_kernel(const __grid_constant__ DenseParams p) {
  using C = PairCfg<D>;
  using T = KVTile<D>;
  static_assert(C::kSmem <= 232448, "shared memory of one CTA");
  static_assert(2 * 128 + 2 * D <= C::kTmemCols, "TMEM columns");
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>(
      (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + C::kOffBar);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(smem + C::kOffMisc);
  volatile int* abort_flag = reinterpret_cast<volatile int*>(smem + C::kOffMisc + 4);
  const int warp = threadIdx.x >> 5;
  const int lane = threadIdx.x & 31;
  const int n_ctas = static_cast<int>(gridDim.x);

  // ---------------------------------------------------------------- setup
  if (threadIdx.x == 0) {
    *abort_flag = 0;
    for (int i = 0; i < C::kStagesK; ++i) {
      mbar_init(&bars[C::B_KFULL + i], 1);
      mbar_init(&bars[C::B_KEMPTY + i], 1);
    }
    for (int i = 0; i < C::kStagesV; ++i) {
      mbar_init(&bars[C::B_VFULL + i], 1);
      mbar_init(&bars[C::B_VEMPTY + i], 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init(&bars[C::B_SFULL + x], 1);
      mbar_init(&bars[C::B_PFULL + x], kTileThreads);
      mbar_init(&bars[C::B_PVDONE + x], 1);
      mbar_init(&bars[C::B_QFULL + x], kTileThreads);
    }
    mbar_init(&bars[C::B_DRAIN], 1);
    fence_mbar_init();
    prefetch_tmap(&p.tmap_k);
    prefetch_tmap(&p.tmap_v);
  }
  if (threadIdx.x >= 32 && threadIdx.x < 32 + 2 * p.hkv && p.run_maps)
    prefetch_tmap(p.run_maps + (threadIdx.x - 32));
  if (warp == kWarpMma) tmem_alloc(tmem_slot, C::kTmemCols);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = *tmem_slot;

  // Each role's code sits inside the branch of its register change, so the
  // compiler allocates it under that warpgroup's limit.
  if (warp >= 8) {
  setmaxnreg_dec<kLowRegs>();
  if (warp == kWarpK || warp == kWarpV) {
    // ------------------------------------------------------------ producers
    const bool is_v = warp == kWarpV;
    bool pok;
    if (is_v)
      pok = kv_producer<D, C::kStagesV>(p, p.items, p.n_items, n_ctas, &p.tmap_v, p.run_maps + p.hkv,
                                        smem + C::kOffV, bars + C::B_VFULL, bars + C::B_VEMPTY,
                                        false, abort_flag, lane);
    else
      pok = kv_producer<D, C::kStagesK>(p, p.items, p.n_items, n_ctas, &p.tmap_k, p.run_maps,
                                        smem + C::kOffK, bars + C::B_KFULL, bars + C::B_KEMPTY,
                                        true, abort_flag, lane);
    if (!pok && lane == 0) atomicOr(p.status, kStatusDenseTimeout);
  } else if (warp == kWarpMma) {
    // ------------------------------------------------------------ MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc_qk = umma_idesc_bf16(128, 128, false, false);
      constexpr uint32_t idesc_pv = umma_idesc_bf16(128, D, false, true);
      const uint32_t qbase = smem_u32(smem + C::kOffQ);
      const uint32_t kbase = smem_u32(smem + C::kOffK);
      const uint32_t vbase = smem_u32(smem + C::kOffV);
      volatile int* const ab = abort_flag;
      bool ok = true;
      auto wait = [&](int b, uint32_t parity) {
        if (ok && !mbar_wait(&bars[b], parity, ab)) ok = false;
        return ok;
      };
      // The issuing thread stays lean: the tensor pipe accepts a new MMA only
      // as an earlier one retires, so any work between MMAs (descriptor
      // arithmetic, a barrier wait inside a group) leaves it idle.  The
      // descriptors of kk = 0 are built once; a kk step or a ring stage adds
      // its byte offset / 16 to the start-address field (bits 0-13, no carry:
      // shared addresses stay below 256 KB).  K and V tiles are consumed in
      // order through running stage / phase counters.
      const uint64_t dq0 = umma_sdesc(qbase, 16, 1024);
      const uint64_t dk0 = umma_sdesc(kbase, 16, T::kGroup);
      const uint64_t dv0 = umma_sdesc(vbase, 1024, T::kGroup);
      int ks = 0, vs = 0;          // ring stage of the next K tile / the current V tile
      uint32_t kph = 0, vph = 0;   // their full-barrier phases
      // S_X = Q_X K^T with K from stage ks; the tile's second QK (X = 1)
      // releases the stage
      auto issue_qk = [&](int x) {
        tc_fence_after();
        const uint64_t a0 = dq0 + static_cast<uint64_t>((x * C::kQBytes) >> 4);
        const uint64_t b0 = dk0 + static_cast<uint64_t>((ks * T::kBytes) >> 4);
#pragma unroll
        for (int kk = 0; kk < D / 16; ++kk)
          umma_bf16_ss(tmem + x * 128, a0 + (((kk >> 2) * T::kChunk + (kk & 3) * 32) >> 4),
                       b0 + (((kk >> 2) * 1024 + (kk & 3) * 32) >> 4), idesc_qk, kk > 0 ? 1u : 0u);
        umma_commit(&bars[C::B_SFULL + x]);
        if (x == 1) {
          umma_commit(&bars[C::B_KEMPTY + ks]);
          if (++ks == C::kStagesK) { ks = 0; kph ^= 1u; }
        }
      };
      // O_X (+)= P_X V with P_X from the first 64 columns of S_X and V from
      // stage vs; the tile's second PV (X = 1) releases the stage
      auto issue_pv = [&](int x, bool first) {
        tc_fence_after();
        const uint64_t b0 = dv0 + static_cast<uint64_t>((vs * T::kBytes) >> 4);
        const uint32_t pcol = tmem + x * 128;
#pragma unroll
        for (int kk = 0; kk < 8; ++kk)
          umma_bf16_ts(tmem + C::kColO + x * D, pcol + kk * 8, b0 + ((kk * T::kPageBytes) >> 4),
                       idesc_pv, (!first || kk > 0) ? 1u : 0u);
        umma_commit(&bars[C::B_PVDONE + x]);
        if (x == 1) {
          umma_commit(&bars[C::B_VEMPTY + vs]);
          if (++vs == C::kStagesV) { vs = 0; vph ^= 1u; }
        }
      };
      // The CTA's tiles in order, g counting across items; the first tile of
      // item k waits for both Q tiles of the item (phase k).  All waits of a
      // group come before its MMAs.
      int g = 0;
      for (int k = 0; ok; ++k) {
        const int idx = item_of(k, n_ctas);
        if (idx >= p.n_items) break;
        const int ntiles = p.items[idx].n_tiles;
        if (ntiles == 0) {  // no keys: only the item's Q phases to pass
          if (!wait(C::B_QFULL + 0, k & 1) || !wait(C::B_QFULL + 1, k & 1)) break;
          continue;
        }
        for (int j = 0; j < ntiles && ok; ++j, ++g) {
          if (j == 0) {
            // this item's S_A(0), S_B(0); the previous item's last PVs were
            // issued before them
            if (!wait(C::B_KFULL + ks, kph) || !wait(C::B_QFULL + 0, k & 1)) break;
            issue_qk(0);
            if (!wait(C::B_QFULL + 1, k & 1)) break;
            issue_qk(1);
          }
          const bool more = j + 1 < ntiles;
          if (!wait(C::B_PFULL + 0, g & 1) || !wait(C::B_VFULL + vs, vph)) break;
          if (more && !wait(C::B_KFULL + ks, kph)) break;
          issue_pv(0, j == 0);
          if (more) issue_qk(0);
          if (!wait(C::B_PFULL + 1, g & 1)) break;
          issue_pv(1, j == 0);
          if (more) issue_qk(1);
        }
      }
      if (!ok) {
        *abort_flag = 1;
        atomicOr(p.status, kStatusDenseTimeout);
      }
      // all MMAs issued by this thread complete before TMEM is released
      umma_commit(&bars[C::B_DRAIN]);
      volatile int never = 0;
      (void)mbar_wait(&bars[C::B_DRAIN], 0, &never);
    }
    __syncwarp();
  }
  } else {
    setmaxnreg_inc<kHighRegs>();
    // ------------------------------------------------------------ softmax
    const int x = warp >> 2;                 // query tile: 0 = A, 1 = B
    const int row = 32 * (warp & 3) + lane;  // row of the tile = TMEM lane
    const int tok_in = x * (128 / G) + row / G;  // token of the item
    const uint32_t lane_base = static_cast<uint32_t>(32 * (warp & 3)) << 16;
    const uint32_t scol = tmem + lane_base + x * 128;
    const uint32_t ocol = tmem + lane_base + C::kColO + x * D;
    uint64_t* const sfull = &bars[C::B_SFULL + x];
    uint64_t* const pfull = &bars[C::B_PFULL + x];
    uint64_t* const pvdone = &bars[C::B_PVDONE + x];
    uint64_t* const qfull = &bars[C::B_QFULL + x];
    uint8_t* const qs = smem + C::kOffQ + x * C::kQBytes;
    const float sc = p.scale_log2;
    bool ok = true;
    // warp-uniform outcome, so .sync.aligned tcgen05 ops never see a split warp
    auto wait_all = [&](uint64_t* bar, uint32_t parity) {
      if (!ok) return false;
      if (__all_sync(0xffffffffu, mbar_wait(bar, parity, abort_flag))) return true;
      *abort_flag = 1;
      ok = false;
      return false;
    };
    constexpr DenseTok kNoTok = {0, 0x7fffffff, 0, 0};
    // token i of an item: its DenseTok record, or derived from the item
    // (consecutive rows of one chunk)
    auto tok_of = [&](const DenseItem& it, int i) {
      return it.tok_base >= 0 ? p.toks[it.tok_base + i] : DenseTok{it.row0 + i, it.pos0 + i, 0, 0};
    };
    // this thread's Q row of an item (zero for rows past the item's tokens),
    // into the swizzled Q tile
    auto load_q = [&](const DenseItem& it) {
      const bool valid = tok_in < it.n_tok;
      const int head = it.kv_head * G + row % G;
      const DenseTok t = valid ? tok_of(it, tok_in) : kNoTok;
      const __nv_bfloat16* src =
          p.q + (valid ? (static_cast<int64_t>(t.q_row) * p.hq + head) * D : 0);
#pragma unroll
      for (int u = 0; u < D / 8; ++u)
        cp_async_16(qs + (u >> 3) * T::kChunk + swz128(row, u & 7), src + 8 * u, valid ? 16u : 0u);
      cp_async_commit();
    };
    auto q_ready = [&]() {
      cp_async_wait_all();
      fence_proxy_async();  // generic-proxy writes, read by the tensor cores
      mbar_arrive(qfull);
    };
    if (item_of(0, n_ctas) < p.n_items) {
      load_q(p.items[item_of(0, n_ctas)]);
      q_ready();
    }
    int gt = 0;
    for (int k = 0; ok; ++k) {
      const int idx = item_of(k, n_ctas);
      if (idx >= p.n_items) break;
      const DenseItem& item = p.items[idx];  // read per tile, not held in registers
      const int ntiles = item.n_tiles;
      const int idx_n = item_of(k + 1, n_ctas);
      const bool has_next = idx_n < p.n_items;
      const bool row_valid = tok_in < item.n_tok;
      const DenseTok dt = row_valid ? tok_of(item, tok_in) : kNoTok;
      const int head = item.kv_head * G + row % G;
      float m_run = -INFINITY, l_run = 0.f;
      bool q_issued = false;
      for (int j = 0; j < ntiles; ++j) {
        const TileInfo t = tile_at(item, j);
        const int g = gt + j;
        if (!wait_all(sfull, g & 1)) break;
        tc_fence_after();
        // S with the maximum of each 32 columns, taken by the TMEM load itself
        float s[128], cmax[4];
#pragma unroll
        for (int c = 0; c < 4; ++c) tmem_ld32_max(scol + 32 * c, s + 32 * c, cmax[c]);
        tmem_wait_ld();

        int lim = t.nvalid;
        if (t.causal && dt.causal_pos < t.key0 + lim) {
          const int c = dt.causal_pos - t.key0 + 1;
          lim = c > 0 ? c : 0;
        }
        float mraw = fmaxf(fmax3f(cmax[0], cmax[1], cmax[2]), cmax[3]);
        if (lim < 128) {
          // keys past the range or the causal limit: masked, and the row max
          // taken again over the keys that remain (8 chains of 3-input max)
#pragma unroll
          for (int n = 0; n < 128; ++n) s[n] = n < lim ? s[n] : -INFINITY;
          float acc[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) acc[i] = s[i];
#pragma unroll
          for (int kk = 8; kk < 128; kk += 16)
#pragma unroll
            for (int i = 0; i < 8; ++i) acc[i] = fmax3f(acc[i], s[kk + i], s[kk + 8 + i]);
          mraw = fmax3f(fmax3f(acc[0], acc[1], acc[2]), fmax3f(acc[3], acc[4], acc[5]),
                        fmaxf(acc[6], acc[7]));
        }
        const float mx = mraw * sc;  // sc > 0: max of the scaled scores
        const float m_new = fmaxf(m_run, mx);
        const bool grow = m_new > m_run + kRescaleThreshold;
        const float m_use = grow ? m_new : m_run;
        const float alpha = grow ? fast_exp2(m_run - m_use) : 1.f;
        const float nref = m_use == -INFINITY ? 0.f : -m_use;
        // p = 2^(s * sc - m): packed FMAs, MUFU ex2, 8 independent partial sums
        float sacc[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int n = 0; n < 128; n += 2) {
          ffma2(s[n], s[n + 1], s[n], s[n + 1], sc, sc, nref, nref);
          s[n] = fast_exp2(s[n]);
          s[n + 1] = fast_exp2(s[n + 1]);
        }
#pragma unroll
        for (int n = 0; n < 128; n += 16)
#pragma unroll
          for (int i = 0; i < 8; i += 2) {
            fadd2(sacc[i], sacc[i + 1], sacc[i], sacc[i + 1], s[n + 2 * i], s[n + 2 * i + 1]);
            fadd2(sacc[i], sacc[i + 1], sacc[i], sacc[i + 1], s[n + 2 * i + 2], s[n + 2 * i + 3]);
          }
        const float rsum = ((sacc[0] + sacc[1]) + (sacc[2] + sacc[3])) +
                           ((sacc[4] + sacc[5]) + (sacc[6] + sacc[7]));
        // P (bf16, two keys per column, in key order) over S's first 64
        // columns: only this thread reads this row of S, and it is done
#pragma unroll
        for (int h = 0; h < 2; ++h) {
          // packed in place: entry u <= 2u is overwritten after it was read
#pragma unroll
          for (int u = 0; u < 32; ++u)
            s[64 * h + u] = __uint_as_float(pack_bf16(s[64 * h + 2 * u], s[64 * h + 2 * u + 1]));
          tmem_st32(scol + 32 * h, s + 64 * h);
        }
        // the item's last QK of this tile has completed: Q_X is free
        if (j == ntiles - 1 && has_next) {
          load_q(p.items[idx_n]);
          q_issued = true;
        }
        // rescale the O row when the reference max moved (with real
        // content), after PV(g - 1) has finished accumulating into it
        if (j > 0 && __any_sync(0xffffffffu, grow && m_run > -INFINITY)) {
          if (!wait_all(pvdone, (g - 1) & 1)) break;
          tc_fence_after();
#pragma unroll 1
          for (int c = 0; c < D / 32; ++c) {
            float o[32];
            tmem_ld32(ocol + 32 * c, o);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] *= alpha;
            tmem_st32(ocol + 32 * c, o);
          }
        }
        tmem_wait_st();
        l_run = l_run * alpha + rsum;
        m_run = m_use;
        if (x == 0 && t.nvalid < 128) {
          // keys past the range: zero their V rows (stale data may not be
          // finite) before PV_A, which runs before PV_B
          if (!wait_all(&bars[C::B_VFULL + g % C::kStagesV], (g / C::kStagesV) & 1)) break;
          if (row >= t.nvalid) {
            uint8_t* vst = smem + C::kOffV + (g % C::kStagesV) * T::kBytes;
#pragma unroll
            for (int u = 0; u < D / 8; ++u)
              *reinterpret_cast<uint4*>(vst + kv_off<T::NCH>(row, u)) = make_uint4(0, 0, 0, 0);
          }
          fence_proxy_async();
        }
        tc_fence_before();
        mbar_arrive(pfull);
      }
      if (!ok) break;
      if (has_next) {
        if (!q_issued) load_q(p.items[idx_n]);  // an item without keys read no Q
        q_ready();
      }

      // ---------------------------------------------------------- epilogue
      if (ntiles > 0 && !wait_all(pvdone, (gt + ntiles - 1) & 1)) break;
      const float inv = l_run > 0.f ? 1.f / l_run : 0.f;
      const float lse = l_run > 0.f ? (m_run + __log2f(l_run)) * kLn2 : -INFINITY;
      tc_fence_after();
#pragma unroll 1
      for (int c = 0; c < D / 32; ++c) {
        float o[32];
        tmem_ld32(ocol + 32 * c, o);
        tmem_wait_ld();
        if (row_valid) {
          uint4* dst = reinterpret_cast<uint4*>(
              p.out + (static_cast<int64_t>(dt.q_row) * p.hq + head) * D + 32 * c);
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
      if (row_valid) p.lse[static_cast<int64_t>(dt.q_row) * p.hq + head] = lse;
      tc_fence_before();
      gt += ntiles;
    }
    cp_async_wait_all();
    tmem_wait_st();  // a failure may leave a P store unwaited
    if (!ok) atomicOr(p.status, kStatusDenseTimeout);
    tc_fence_before();
  }

  // ---------------------------------------------------------------- teardown
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, C::kTmemCols);
  }
}

template <int D, int G>
cudaError_t launch_prefill_pair_t(const DenseParams& p, int grid, cudaStream_t stream) {
  using C = PairCfg<D>;
  prefill_pair_kernel<D, G><<<grid, kThreads, C::kSmem, stream>>>(p);
  return cudaGetLastError();
}

// Set once by init_prefill_pair: every instantiation was given kLaunchRegs
// registers per thread, the allocation the warpgroup split redistributes.
// With any other count an increase could wait forever, so the kernel is
// not launched at all then.
bool g_regs_checked = false;

template <int D, int G>
cudaError_t check_regs() {
  cudaFuncAttributes a{};
  cudaError_t e = cudaFuncGetAttributes(&a, prefill_pair_kernel<D, G>);
  if (e != cudaSuccess) return e;
  return a.numRegs == kLaunchRegs ? cudaSuccess : cudaErrorInvalidDeviceFunction;
}

}  // namespace

cudaError_t launch_prefill_pair(const DenseParams& p, int grid, int head_dim, int group,
                                cudaStream_t stream) {
  if (p.n_items <= 0 || grid <= 0) return cudaSuccess;
  if (p.plan_flag) return cudaErrorInvalidValue;  // the plan goes up on the launch stream
  if (!g_regs_checked) return cudaErrorInvalidDeviceFunction;
  if (head_dim == 128 && group == 4) return launch_prefill_pair_t<128, 4>(p, grid, stream);
  if (head_dim == 128 && group == 8) return launch_prefill_pair_t<128, 8>(p, grid, stream);
  if (head_dim == 64 && group == 4) return launch_prefill_pair_t<64, 4>(p, grid, stream);
  if (head_dim == 64 && group == 8) return launch_prefill_pair_t<64, 8>(p, grid, stream);
  return cudaErrorInvalidValue;
}

cudaError_t init_prefill_pair() {
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(prefill_pair_kernel<128, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                PairCfg<128>::kSmem)))
    return e;
  if ((e = cudaFuncSetAttribute(prefill_pair_kernel<128, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                PairCfg<128>::kSmem)))
    return e;
  if ((e = cudaFuncSetAttribute(prefill_pair_kernel<64, 4>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                PairCfg<64>::kSmem)))
    return e;
  if ((e = cudaFuncSetAttribute(prefill_pair_kernel<64, 8>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                PairCfg<64>::kSmem)))
    return e;
  // a wrong register count leaves the kernel unlaunchable (launches fail
  // with cudaErrorInvalidDeviceFunction) without failing initialisation
  g_regs_checked = check_regs<128, 4>() == cudaSuccess && check_regs<128, 8>() == cudaSuccess &&
                   check_regs<64, 4>() == cudaSuccess && check_regs<64, 8>() == cudaSuccess;
  return cudaSuccess;
}

}  // namespace tpa
