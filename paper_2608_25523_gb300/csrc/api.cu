// C ABI: context, paged pool tables, per-call planning and launches.
//
// Host-side model of the paper's GPU state S_t = (R_t, Q_t) (Sec. III):
//   * agents  -> registered prefixes of length ell_a; resident ones hold a
//     run of pool pages (the prefix is paid once per agent, Eq. 2);
//   * requests -> open requests of an agent with a private suffix page run;
//   * the free-page list is the remaining budget B_t; a call that needs
//     more pages than are free fails with TPA_ERR_NO_SPACE.
// Every device-facing call builds one plan blob (page lists and work items)
// in a pinned staging slot, uploads it with one copy and launches the
// kernels.  Pages freed while queued work may still read them carry the
// sequence number of that work; whoever reuses them first waits for it.
#include <cudaTypedefs.h>

#include <algorithm>
#include <cmath>
#include <cstddef>
#include <cstdlib>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <string>
#include <unordered_map>
#include <vector>

#include "../../include/topas_attn.h"
#include "kernels.h"

namespace tpa {
cudaError_t init_dense_kernels();
cudaError_t init_suffix_kernels();
cudaError_t init_prefill_pair();
}  // namespace tpa

using namespace tpa;

namespace {

thread_local std::string g_err;

int fail(int code, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(buf, sizeof(buf), fmt, ap);
  va_end(ap);
  g_err = buf;
  return code;
}

#define CUDA_TRY(expr)                                                              \
  do {                                                                              \
    cudaError_t e_ = (expr);                                                        \
    if (e_ != cudaSuccess)                                                          \
      return fail(TPA_ERR_CUDA, "%s: %s (%s:%d)", #expr, cudaGetErrorString(e_),    \
                  __FILE__, __LINE__);                                              \
  } while (0)

constexpr int kRingSlots = 4;
constexpr int kSplitWarpsPerCta = 8;  // split-KV warps of a CTA in the fused decode launch
constexpr int kKernelKinds = 6;  // append, dense, split-KV, merge, page copy, paired prefill
enum { K_APPEND = 0, K_DENSE = 1, K_SUFFIX = 2, K_MERGE = 3, K_COPY = 4, K_PREFILL_PAIR = 5 };
constexpr size_t kAlign = 256;

size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }
int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }

struct Agent {
  int32_t len = -1;       // -1: not registered
  bool resident = false;
  std::vector<int32_t> pages;
  uint64_t ready_seq = 0; // reload/offload call the next reader must wait for
  uint64_t last_use = 0;  // last call that read or wrote the pages
};

struct Request {
  bool open = false;
  int32_t agent = -1;
  int32_t len = 0;
  std::vector<int32_t> pages;
  uint64_t last_use = 0;
};

struct Slot {
  uint8_t* host = nullptr;   // pinned staging
  uint8_t* dev = nullptr;    // device copy (workspace)
  cudaEvent_t done = nullptr;
  cudaStream_t stream = nullptr;  // stream `done` was recorded on
  uint64_t seq = 0;          // call that used the slot last (0: never)
};

// Sizes of one plan: number of records per section.
struct PlanSizes {
  int64_t pages = 0, append = 0, dense_tok = 0, dense = 0, suffix = 0, merge = 0, stok = 0,
          sint = 0;
};

struct PlanLayout {
  size_t off_pages, off_append, off_dense_tok, off_dense, off_suffix, off_merge, off_stok,
      off_sint, total;
};

PlanLayout layout_of(const PlanSizes& s) {
  PlanLayout l;
  size_t o = align_up(sizeof(PlanHeader), 64);
  l.off_pages = o;
  o = align_up(o + s.pages * 4, 64);
  l.off_append = o;
  o = align_up(o + s.append * sizeof(AppendRow), 64);
  l.off_dense_tok = o;
  o = align_up(o + s.dense_tok * sizeof(DenseTok), 64);
  l.off_dense = o;
  o = align_up(o + s.dense * sizeof(DenseItem), 64);
  l.off_suffix = o;
  o = align_up(o + s.suffix * sizeof(SuffixItem), 64);
  l.off_merge = o;
  o = align_up(o + s.merge * sizeof(MergeTok), 64);
  l.off_stok = o;
  o = align_up(o + s.stok * sizeof(SplitTok), 64);
  l.off_sint = o;
  o = align_up(o + s.sint * 4, 64);
  l.total = o;
  return l;
}

}  // namespace

struct tpa_ctx {
  tpa_config cfg{};
  int hq = 0, hkv = 0, d = 0, group = 0;
  bool plan_only = false;
  int64_t max_pages_per_seq = 0;
  int max_splits = 32;

  std::vector<int32_t> free_pages;   // used as a queue: next page at free_head
  size_t free_head = 0;
  std::vector<uint64_t> page_tag;    // call seq that may still read the page
  std::vector<Agent> agents;
  std::vector<Request> reqs;

  // device side
  int device = 0;
  int num_sms = 148;
  CUtensorMap tmap_k{}, tmap_v{};
  CUtensorMap* run_maps = nullptr;  // device copy (workspace) of the per-kv-head page-run views
  PoolGeom pool{};
  uint32_t* status = nullptr;
  float* part_o = nullptr;
  float* part_lse = nullptr;
  // staging area of the prefix movement: a whole prefix's K and V
  // ([max_seq_len][Hkv][d] bf16 each); the host link transfer is a copy-engine
  // copy into it, and the page scatter / gather an on-device kernel
  uint8_t* stage_k = nullptr;
  uint8_t* stage_v = nullptr;
  uint64_t stage_seq = 0;  // the last movement call that used it
  int64_t part_slots = 0;
  size_t plan_cap = 0;               // bytes of a plan slot; its upload flag follows it
  Slot ring[kRingSlots];
  cudaStream_t copy_stream = nullptr;  // decode plans are uploaded here, ahead of the kernels
  int ring_pos = 0;
  uint64_t seq = 0;
  uint64_t chain_seq = 0;            // last chain (ordered) call
  cudaStream_t chain_stream = nullptr;

  // options and statistics
  int decode_mode = 0;
  int prefill_rows = 256;
  bool staged_movement = true;  // TPA_OPT_MOVEMENT_STAGED  // query rows per prefill work item: 256 (tile pairs) or 128
  int test_plan_wait = 0;  // test hook: the next cascade decode waits for a flag never written
  int test_bad_page = 0;   // test hook: the next decode's first prefix page id is out of the pool
  int test_bad_slot = 0;   // test hook: the next decode's first token's partial slots are out of range
  int prefix_splits = 0;
  int suffix_split_keys = 0;
  int64_t last_dense = 0, last_suffix = 0, last_launches = 0;

  // per-kernel event timing (TPA_OPT_KERNEL_TIMING)
  int timing = 0;
  struct Pending {
    int kind;
    cudaEvent_t a, b;
  };
  std::vector<cudaEvent_t> ev_free;
  std::vector<Pending> pending;
  double k_ms[kKernelKinds] = {};
  int64_t k_n[kKernelKinds] = {};

  // per-call stamps and scratch reused across calls (no heap traffic in steady state)
  uint64_t stamp = 0;
  std::vector<uint64_t> req_stamp;    // request id -> stamp of the call that saw it
  std::vector<uint64_t> agent_stamp;  // agent id -> stamp
  std::vector<int32_t> agent_group;   // agent id -> group index in the current call
  std::vector<int32_t> order;         // scratch: token order
};

namespace {

// ------------------------------------------------------------------ helpers

bool valid_shape(const tpa_config* c) {
  if (!c) return false;
  if (c->page_size != kPage) return false;
  if (c->head_dim != 64 && c->head_dim != 128) return false;
  if (c->num_kv_heads <= 0 || c->num_q_heads <= 0) return false;
  if (c->num_q_heads % c->num_kv_heads) return false;
  const int g = c->num_q_heads / c->num_kv_heads;
  if (g != 4 && g != 8) return false;
  return true;
}

int64_t max_pages_of(const tpa_config* c) { return cdiv(c->max_seq_len + 1, kPage) + 1; }

int splits_of(const tpa_config* c) { return c->max_splits > 0 ? c->max_splits : 32; }

// Decode batches are at most min(max_tokens, max_requests) requests (ids are
// distinct); prefill chunks hold at most max_tokens rows.
int64_t max_batch_requests(const tpa_config* c) {
  return std::min<int64_t>(c->max_tokens, c->max_requests);
}

PlanSizes plan_capacity(const tpa_config* c) {
  const int64_t g = c->num_q_heads / c->num_kv_heads;
  const int64_t tpt = kTileRows / g;
  const int64_t T = c->max_tokens;
  const int64_t R = max_batch_requests(c);
  const int64_t A = std::min<int64_t>(c->max_agents, R);
  const int64_t S = splits_of(c);
  const int64_t H = c->num_kv_heads;
  PlanSizes s;
  s.pages = (R + A) * max_pages_of(c);
  s.append = T;
  s.dense_tok = T + R;
  // decode: stacked prefix tiles + per-token suffix items; prefill: chunk tiles
  s.dense = H * std::max((cdiv(R, tpt) + A) * S + R * S, cdiv(T, tpt) + R);
  s.suffix = R * H * S;
  s.merge = R;
  s.stok = R;
  s.sint = 2 * R + 1;
  return s;
}

// Wait on the device (stream `s`) for call `seq` if it may still be running.
void wait_for_seq(tpa_ctx* ctx, uint64_t seq, cudaStream_t s) {
  if (seq == 0 || ctx->plan_only) return;
  for (auto& sl : ctx->ring) {
    if (sl.seq == seq) {
      // work already queued on `s` is ordered before what follows on `s`; an
      // event wait would only stall the queue until that call has drained
      if (sl.stream == s) return;
      if (cudaEventQuery(sl.done) == cudaErrorNotReady) cudaStreamWaitEvent(s, sl.done, 0);
      else (void)cudaGetLastError();
      return;
    }
  }
  // not in the ring any more: its slot was recycled after a host-side wait
}

// Whether work on `s` would still have to wait for call `seq` (another
// stream's call that has not completed).
bool seq_pending(tpa_ctx* ctx, uint64_t seq, cudaStream_t s) {
  if (seq == 0 || ctx->plan_only) return false;
  for (auto& sl : ctx->ring) {
    if (sl.seq != seq) continue;
    if (sl.stream == s) return false;
    if (cudaEventQuery(sl.done) == cudaErrorNotReady) return true;
    (void)cudaGetLastError();
    return false;
  }
  return false;
}

// Take `n` pages from the free list; returns the highest reuse tag.
uint64_t take_pages(tpa_ctx* ctx, int64_t n, std::vector<int32_t>& out) {
  uint64_t tag = 0;
  for (int64_t i = 0; i < n; ++i) {
    const int32_t pg = ctx->free_pages[ctx->free_head++];
    tag = std::max(tag, ctx->page_tag[pg]);
    out.push_back(pg);
  }
  return tag;
}

void give_pages(tpa_ctx* ctx, std::vector<int32_t>& pages, uint64_t tag) {
  // compact the consumed head before appending
  if (ctx->free_head > 0 && ctx->free_head * 2 > ctx->free_pages.size()) {
    ctx->free_pages.erase(ctx->free_pages.begin(), ctx->free_pages.begin() + ctx->free_head);
    ctx->free_head = 0;
  }
  for (int32_t pg : pages) {
    ctx->page_tag[pg] = std::max(ctx->page_tag[pg], tag);
    ctx->free_pages.push_back(pg);
  }
  pages.clear();
}

int64_t free_count(const tpa_ctx* ctx) {
  return static_cast<int64_t>(ctx->free_pages.size() - ctx->free_head);
}

// Kernel timing: bracket a launch with events on its stream when enabled.
cudaEvent_t timing_event(tpa_ctx* ctx) {
  if (!ctx->ev_free.empty()) {
    cudaEvent_t e = ctx->ev_free.back();
    ctx->ev_free.pop_back();
    return e;
  }
  cudaEvent_t e = nullptr;
  if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
  return e;
}

int resolve_timing(tpa_ctx* ctx) {
  for (auto& p : ctx->pending) {
    float ms = 0.f;
    CUDA_TRY(cudaEventSynchronize(p.b));
    CUDA_TRY(cudaEventElapsedTime(&ms, p.a, p.b));
    ctx->k_ms[p.kind] += ms;
    ctx->k_n[p.kind] += 1;
    ctx->ev_free.push_back(p.a);
    ctx->ev_free.push_back(p.b);
  }
  ctx->pending.clear();
  return TPA_OK;
}

struct KernelTimer {
  tpa_ctx* ctx;
  int kind;
  cudaStream_t s;
  cudaEvent_t a = nullptr;
  KernelTimer(tpa_ctx* c, int k, cudaStream_t st) : ctx(c), kind(k), s(st) {
    if (ctx->timing && !ctx->plan_only) {
      if (ctx->pending.size() > 8192) resolve_timing(ctx);
      a = timing_event(ctx);
      if (a) cudaEventRecord(a, s);
    }
  }
  ~KernelTimer() {
    if (!a) return;
    cudaEvent_t b = timing_event(ctx);
    if (!b) return;
    cudaEventRecord(b, s);
    ctx->pending.push_back({kind, a, b});
  }
};

// Acquire the next plan slot (host-blocking only if kRingSlots calls are in flight).
Slot* acquire_slot(tpa_ctx* ctx) {
  Slot* s = &ctx->ring[ctx->ring_pos];
  ctx->ring_pos = (ctx->ring_pos + 1) % kRingSlots;
  if (!ctx->plan_only && s->seq != 0) cudaEventSynchronize(s->done);
  return s;
}

// Plan blob writer over a slot's host buffer.
struct PlanWriter {
  uint8_t* base;
  PlanLayout lay;
  PlanHeader* hdr;
  int32_t* pages;
  AppendRow* append;
  DenseTok* dtok;
  DenseItem* dense;
  SuffixItem* suffix;
  MergeTok* merge;
  SplitTok* stok;
  int32_t* sint;
  PlanWriter(uint8_t* b, const PlanLayout& l) : base(b), lay(l) {
    hdr = reinterpret_cast<PlanHeader*>(b);
    std::memset(hdr, 0, sizeof(PlanHeader));
    pages = reinterpret_cast<int32_t*>(b + l.off_pages);
    append = reinterpret_cast<AppendRow*>(b + l.off_append);
    dtok = reinterpret_cast<DenseTok*>(b + l.off_dense_tok);
    dense = reinterpret_cast<DenseItem*>(b + l.off_dense);
    suffix = reinterpret_cast<SuffixItem*>(b + l.off_suffix);
    merge = reinterpret_cast<MergeTok*>(b + l.off_merge);
    stok = reinterpret_cast<SplitTok*>(b + l.off_stok);
    sint = reinterpret_cast<int32_t*>(b + l.off_sint);
  }
};

template <class T>
const T* dev_ptr(const Slot* s, size_t off) {
  return reinterpret_cast<const T*>(s->dev + off);
}

int check_batch(tpa_ctx* ctx, int32_t n, const int32_t* reqs, bool need_resident) {
  if (n <= 0 || !reqs) return fail(TPA_ERR_INVALID_ARG, "empty batch");
  if (n > ctx->cfg.max_tokens) return fail(TPA_ERR_CAPACITY, "batch of %d > max_tokens", n);
  for (int i = 0; i < n; ++i) {
    const int32_t r = reqs[i];
    if (r < 0 || r >= ctx->cfg.max_requests) return fail(TPA_ERR_INVALID_ARG, "request id %d", r);
    if (!ctx->reqs[r].open) return fail(TPA_ERR_STATE, "request %d is not open", r);
    if (need_resident && !ctx->agents[ctx->reqs[r].agent].resident)
      return fail(TPA_ERR_NOT_RESIDENT, "prefix of agent %d (request %d) is not resident",
                  ctx->reqs[r].agent, r);
  }
  const uint64_t st = ++ctx->stamp;
  for (int i = 0; i < n; ++i) {
    if (ctx->req_stamp[reqs[i]] == st) return fail(TPA_ERR_INVALID_ARG, "request %d twice", reqs[i]);
    ctx->req_stamp[reqs[i]] = st;
  }
  return TPA_OK;
}

// Begin a chain call on `s`: order after the previous chain call.
void chain_begin(tpa_ctx* ctx, cudaStream_t s) {
  if (ctx->plan_only) return;
  if (ctx->chain_seq && ctx->chain_stream != s) wait_for_seq(ctx, ctx->chain_seq, s);
}

int upload(tpa_ctx* ctx, Slot* sl, size_t bytes, cudaStream_t s) {
  if (ctx->plan_only) return TPA_OK;
  CUDA_TRY(cudaMemcpyAsync(sl->dev, sl->host, bytes, cudaMemcpyHostToDevice, s));
  return TPA_OK;
}

// Upload a plan on the context's copy stream, followed by the call's
// sequence number into the slot's flag word: the kernel reading the plan
// waits (bounded) for that flag, so the call's own stream carries only
// kernels and the next step's kernel can be a programmatic dependent of the
// previous one.  The slot is reused only after its call's done event, which
// follows a kernel that saw the flag, so the copies have completed by then.
int upload_ahead(tpa_ctx* ctx, Slot* sl, size_t bytes, const unsigned long long** flag) {
  *flag = nullptr;
  if (ctx->plan_only) return TPA_OK;
  uint64_t* fh = reinterpret_cast<uint64_t*>(sl->host + ctx->plan_cap);
  *fh = ctx->seq;
  CUDA_TRY(cudaMemcpyAsync(sl->dev, sl->host, bytes, cudaMemcpyHostToDevice, ctx->copy_stream));
  CUDA_TRY(cudaMemcpyAsync(sl->dev + ctx->plan_cap, fh, sizeof(uint64_t), cudaMemcpyHostToDevice,
                           ctx->copy_stream));
  *flag = reinterpret_cast<const unsigned long long*>(sl->dev + ctx->plan_cap);
  return TPA_OK;
}

int finish_call(tpa_ctx* ctx, Slot* sl, cudaStream_t s, bool chain) {
  sl->seq = ctx->seq;
  if (chain) {
    ctx->chain_seq = ctx->seq;
    ctx->chain_stream = s;
  }
  if (ctx->plan_only) return TPA_OK;
  CUDA_TRY(cudaEventRecord(sl->done, s));
  sl->stream = s;
  return TPA_OK;
}

}  // namespace

// ====================================================================== ABI

extern "C" {

const char* tpa_last_error(void) { return g_err.c_str(); }

// One operand (K or V) of the longest prefix, [max_seq_len][Hkv][d] bf16.
static size_t stage_bytes(const tpa_config* cfg) {
  return static_cast<size_t>(cfg->max_seq_len) * cfg->num_kv_heads * cfg->head_dim * 2;
}

size_t tpa_workspace_size(const tpa_config* cfg) {
  if (!valid_shape(cfg) || cfg->max_tokens <= 0 || cfg->max_seq_len <= 0) return 0;
  const PlanLayout lay = layout_of(plan_capacity(cfg));
  const int64_t slots = max_batch_requests(cfg) * cfg->num_q_heads * splits_of(cfg);
  size_t total = kAlign;                                     // status word
  total += align_up(2 * static_cast<size_t>(cfg->num_kv_heads) * sizeof(CUtensorMap), kAlign);
  total += kRingSlots * (align_up(lay.total, kAlign) + kAlign);  // plan ring (+ upload flags)
  total += align_up(slots * cfg->head_dim * sizeof(float), kAlign);
  total += align_up(slots * sizeof(float), kAlign);
  total += 2 * align_up(stage_bytes(cfg), kAlign);           // prefix movement staging
  return total;
}

int tpa_create(const tpa_config* cfg, tpa_ctx** out) {
  if (!cfg || !out) return fail(TPA_ERR_INVALID_ARG, "null argument");
  *out = nullptr;
  if (!valid_shape(cfg))
    return fail(TPA_ERR_UNSUPPORTED, "supported: page 16, head_dim 64/128, group 4/8");
  if (cfg->num_pages <= 0 || cfg->max_agents <= 0 || cfg->max_requests <= 0 ||
      cfg->max_tokens <= 0 || cfg->max_seq_len <= 0 || cfg->max_splits < 0)
    return fail(TPA_ERR_INVALID_ARG, "sizes must be positive");
  if (cfg->num_pages * cfg->num_kv_heads >= (1ll << 31))
    return fail(TPA_ERR_UNSUPPORTED, "num_pages * num_kv_heads must be < 2^31");
  const bool plan_only = (cfg->flags & TPA_FLAG_PLAN_ONLY) != 0;
  if (!plan_only) {
    if (!cfg->k_pool || !cfg->v_pool || !cfg->workspace)
      return fail(TPA_ERR_INVALID_ARG, "pools and workspace are required");
    if ((reinterpret_cast<uintptr_t>(cfg->k_pool) | reinterpret_cast<uintptr_t>(cfg->v_pool)) & 15)
      return fail(TPA_ERR_INVALID_ARG, "pools must be 16-byte aligned");
    if (reinterpret_cast<uintptr_t>(cfg->workspace) & (kAlign - 1))
      return fail(TPA_ERR_INVALID_ARG, "workspace must be 256-byte aligned");
    if (cfg->workspace_bytes < tpa_workspace_size(cfg))
      return fail(TPA_ERR_INVALID_ARG, "workspace of %zu bytes < %zu needed", cfg->workspace_bytes,
                  tpa_workspace_size(cfg));
  }

  tpa_ctx* ctx = new tpa_ctx();
  ctx->cfg = *cfg;
  ctx->hq = cfg->num_q_heads;
  ctx->hkv = cfg->num_kv_heads;
  ctx->d = cfg->head_dim;
  ctx->group = ctx->hq / ctx->hkv;
  ctx->plan_only = plan_only;
  ctx->max_pages_per_seq = max_pages_of(cfg);
  ctx->max_splits = splits_of(cfg);
  ctx->agents.resize(cfg->max_agents);
  ctx->reqs.resize(cfg->max_requests);
  ctx->req_stamp.assign(cfg->max_requests, 0);
  ctx->agent_stamp.assign(cfg->max_agents, 0);
  ctx->agent_group.assign(cfg->max_agents, 0);
  ctx->page_tag.assign(cfg->num_pages, 0);
  ctx->free_pages.resize(cfg->num_pages);
  for (int64_t i = 0; i < cfg->num_pages; ++i) ctx->free_pages[i] = static_cast<int32_t>(i);
  if (cfg->page_order_seed) {
    // seeded Fisher-Yates with splitmix64: a fragmented pool, same on every host
    uint64_t x = cfg->page_order_seed;
    auto next = [&x]() {
      uint64_t z = (x += 0x9E3779B97F4A7C15ull);
      z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
      z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
      return z ^ (z >> 31);
    };
    for (int64_t i = cfg->num_pages - 1; i > 0; --i) {
      const int64_t j = static_cast<int64_t>(next() % static_cast<uint64_t>(i + 1));
      std::swap(ctx->free_pages[i], ctx->free_pages[j]);
    }
  }

  const PlanLayout lay = layout_of(plan_capacity(cfg));
  ctx->plan_cap = align_up(lay.total, kAlign);
  ctx->part_slots = max_batch_requests(cfg) * ctx->hq * ctx->max_splits;

  if (plan_only) {
    for (auto& s : ctx->ring) s.host = static_cast<uint8_t*>(std::malloc(ctx->plan_cap));
    *out = ctx;
    return TPA_OK;
  }

  auto cleanup = [ctx](int code) {
    tpa_destroy(ctx);
    return code;
  };
  int rc;
  cudaError_t e;
  if ((e = cudaGetDevice(&ctx->device)) != cudaSuccess)
    return cleanup(fail(TPA_ERR_CUDA, "cudaGetDevice: %s", cudaGetErrorString(e)));
  if ((e = cudaDeviceGetAttribute(&ctx->num_sms, cudaDevAttrMultiProcessorCount, ctx->device)) !=
      cudaSuccess)
    return cleanup(fail(TPA_ERR_CUDA, "SM count: %s", cudaGetErrorString(e)));
  if ((e = tpa::init_kernels()) != cudaSuccess)
    return cleanup(fail(TPA_ERR_CUDA, "kernel attributes: %s", cudaGetErrorString(e)));

  // TMA descriptors: a 5-D view of each pool in which one box is one page of
  // one kv head, (64 dims, 8 slots, d/64 chunks, 2 slot halves, page*hkv), so
  // it lands as [slot half][chunk][8 slots][128 B] with 128-byte swizzle
  void* fn = nullptr;
  cudaDriverEntryPointQueryResult q;
  if ((e = cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault,
                                            &q)) != cudaSuccess ||
      q != cudaDriverEntryPointSuccess || !fn)
    return cleanup(fail(TPA_ERR_CUDA, "cuTensorMapEncodeTiled entry point unavailable"));
  auto encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
  const cuuint64_t row = static_cast<cuuint64_t>(ctx->d) * 2;  // bytes of one slot's d-row
  const cuuint64_t nch = static_cast<cuuint64_t>(ctx->d / 64);
  const cuuint64_t dims[5] = {64, 8, nch, 2, static_cast<cuuint64_t>(cfg->num_pages * ctx->hkv)};
  const cuuint64_t strides[4] = {row, 128, 8 * row, static_cast<cuuint64_t>(kPage) * row};
  const cuuint32_t box[5] = {64, 8, static_cast<cuuint32_t>(nch), 2, 1};
  const cuuint32_t estr[5] = {1, 1, 1, 1, 1};
  for (int w = 0; w < 2; ++w) {
    CUresult r = encode(w ? &ctx->tmap_v : &ctx->tmap_k, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5,
                        w ? cfg->v_pool : cfg->k_pool, dims, strides, box, estr,
                        CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (r != CUDA_SUCCESS) return cleanup(fail(TPA_ERR_CUDA, "cuTensorMapEncodeTiled: %d", (int)r));
  }
  // per-kv-head views for runs of consecutive pages: the kv head is in the
  // base address and the last dimension steps over pages
  std::vector<CUtensorMap> runs(2 * static_cast<size_t>(ctx->hkv));
  {
    const cuuint64_t rdims[5] = {64, 8, nch, 2, static_cast<cuuint64_t>(cfg->num_pages)};
    const cuuint64_t rstrides[4] = {row, 128, 8 * row,
                                    static_cast<cuuint64_t>(ctx->hkv) * kPage * row};
    const cuuint32_t rbox[5] = {64, 8, static_cast<cuuint32_t>(nch), 2, 8};
    for (int w = 0; w < 2; ++w)
      for (int h = 0; h < ctx->hkv; ++h) {
        void* base = static_cast<uint8_t*>(w ? cfg->v_pool : cfg->k_pool) +
                     static_cast<size_t>(h) * kPage * row;
        CUresult r = encode(&runs[w * ctx->hkv + h], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 5, base,
                            rdims, rstrides, rbox, estr, CU_TENSOR_MAP_INTERLEAVE_NONE,
                            CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                            CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
        if (r != CUDA_SUCCESS)
          return cleanup(fail(TPA_ERR_CUDA, "cuTensorMapEncodeTiled (runs): %d", (int)r));
      }
  }
  ctx->pool = PoolGeom{cfg->k_pool, cfg->v_pool, cfg->num_pages, ctx->hkv, ctx->d};

  // workspace carve-up
  uint8_t* ws = static_cast<uint8_t*>(cfg->workspace);
  ctx->status = reinterpret_cast<uint32_t*>(ws);
  size_t off = kAlign;
  ctx->run_maps = reinterpret_cast<CUtensorMap*>(ws + off);
  off += align_up(runs.size() * sizeof(CUtensorMap), kAlign);
  for (auto& s : ctx->ring) {
    s.dev = ws + off;
    off += ctx->plan_cap + kAlign;
  }
  ctx->part_o = reinterpret_cast<float*>(ws + off);
  off += align_up(ctx->part_slots * ctx->d * sizeof(float), kAlign);
  ctx->part_lse = reinterpret_cast<float*>(ws + off);
  off += align_up(ctx->part_slots * sizeof(float), kAlign);
  ctx->stage_k = ws + off;
  off += align_up(stage_bytes(cfg), kAlign);
  ctx->stage_v = ws + off;

  for (auto& s : ctx->ring) {
    if ((e = cudaHostAlloc(reinterpret_cast<void**>(&s.host), ctx->plan_cap + kAlign,
                           cudaHostAllocDefault)) != cudaSuccess)
      return cleanup(fail(TPA_ERR_CUDA, "pinned staging: %s", cudaGetErrorString(e)));
    if ((e = cudaEventCreateWithFlags(&s.done, cudaEventDisableTiming)) != cudaSuccess)
      return cleanup(fail(TPA_ERR_CUDA, "event: %s", cudaGetErrorString(e)));
  }
  if ((e = cudaMemcpy(ctx->run_maps, runs.data(), runs.size() * sizeof(CUtensorMap),
                      cudaMemcpyHostToDevice)) != cudaSuccess)
    return cleanup(fail(TPA_ERR_CUDA, "tensor maps: %s", cudaGetErrorString(e)));
  if ((e = cudaStreamCreateWithFlags(&ctx->copy_stream, cudaStreamNonBlocking)) != cudaSuccess)
    return cleanup(fail(TPA_ERR_CUDA, "copy stream: %s", cudaGetErrorString(e)));
  if ((e = cudaMemsetAsync(ctx->status, 0, sizeof(uint32_t), 0)) != cudaSuccess)
    return cleanup(fail(TPA_ERR_CUDA, "status init: %s", cudaGetErrorString(e)));
  for (auto& s : ctx->ring)
    if ((e = cudaMemsetAsync(s.dev + ctx->plan_cap, 0, sizeof(uint64_t), 0)) != cudaSuccess)
      return cleanup(fail(TPA_ERR_CUDA, "flag init: %s", cudaGetErrorString(e)));
  if ((e = cudaStreamSynchronize(0)) != cudaSuccess)
    return cleanup(fail(TPA_ERR_CUDA, "status init: %s", cudaGetErrorString(e)));
  (void)rc;
  *out = ctx;
  return TPA_OK;
}

int tpa_destroy(tpa_ctx* ctx) {
  if (!ctx) return TPA_OK;
  if (ctx->plan_only) {
    for (auto& s : ctx->ring) std::free(s.host);
  } else {
    for (auto& s : ctx->ring) {
      if (s.done) {
        if (s.seq) cudaEventSynchronize(s.done);
        cudaEventDestroy(s.done);
      }
      if (s.host) cudaFreeHost(s.host);
    }
    resolve_timing(ctx);
    for (cudaEvent_t e : ctx->ev_free) cudaEventDestroy(e);
    if (ctx->copy_stream) {
      cudaStreamSynchronize(ctx->copy_stream);
      cudaStreamDestroy(ctx->copy_stream);
    }
  }
  delete ctx;
  return TPA_OK;
}

// ---------------------------------------------------------------- prefixes

int tpa_prefix_register(tpa_ctx* ctx, int32_t agent, int32_t len) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  if (agent < 0 || agent >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", agent);
  if (len < 0 || len > ctx->cfg.max_seq_len) return fail(TPA_ERR_INVALID_ARG, "prefix length %d", len);
  Agent& a = ctx->agents[agent];
  if (a.len >= 0) return fail(TPA_ERR_STATE, "agent %d is already registered", agent);
  const int64_t need = cdiv(len, kPage);
  if (need > free_count(ctx))
    return fail(TPA_ERR_NO_SPACE, "prefix needs %lld pages, %lld free", (long long)need,
                (long long)free_count(ctx));
  a.pages.clear();
  const uint64_t tag = take_pages(ctx, need, a.pages);
  a.len = len;
  a.resident = true;
  a.ready_seq = 0;
  a.last_use = tag;  // a later writer must wait for the pages' previous readers
  return TPA_OK;
}

// Copy `len` tokens between a contiguous [len][Hkv][d] pair of arrays and a
// page run.  `staged`: the contiguous side is host memory, moved by the copy
// engine through the workspace's staging area while the page scatter (to
// pages) or gather (from pages) is a short on-device kernel, so the link
// transfer holds no SM while compute runs beside it; otherwise the kernel
// reads or writes the contiguous side itself.
static int page_copy_call(tpa_ctx* ctx, const std::vector<int32_t>& pages, int len, int to_pages,
                          const void* k_in, const void* v_in, void* k_out, void* v_out,
                          cudaStream_t s, bool chain, uint64_t wait_seq, Slot** used,
                          bool staged = false) {
  const size_t bytes = static_cast<size_t>(len) * ctx->hkv * ctx->d * 2;
  if (staged && len > ctx->cfg.max_seq_len) return fail(TPA_ERR_CAPACITY, "%d tokens > max_seq_len", len);
  Slot* sl = acquire_slot(ctx);
  ++ctx->seq;
  PlanSizes sz;
  sz.pages = static_cast<int64_t>(pages.size());
  const PlanLayout lay = layout_of(sz);
  if (lay.total > ctx->plan_cap) return fail(TPA_ERR_CAPACITY, "page list too long");
  PlanWriter w(sl->host, lay);
  w.hdr->n_pages = static_cast<int32_t>(pages.size());
  std::memcpy(w.pages, pages.data(), pages.size() * 4);
  if (chain) chain_begin(ctx, s);
  wait_for_seq(ctx, wait_seq, s);
  if (staged) wait_for_seq(ctx, ctx->stage_seq, s);  // the staging area's previous user
  int rc = upload(ctx, sl, lay.total, s);
  if (rc) return rc;
  if (!ctx->plan_only) {
    const bool in = staged && to_pages && len > 0, out = staged && !to_pages && len > 0;
    if (in) {
      CUDA_TRY(cudaMemcpyAsync(ctx->stage_k, k_in, bytes, cudaMemcpyDefault, s));
      CUDA_TRY(cudaMemcpyAsync(ctx->stage_v, v_in, bytes, cudaMemcpyDefault, s));
      k_in = ctx->stage_k;
      v_in = ctx->stage_v;
    }
    {
      KernelTimer kt(ctx, K_COPY, s);
      CUDA_TRY(launch_page_copy(dev_ptr<int32_t>(sl, lay.off_pages), len, to_pages, k_in, v_in,
                                out ? ctx->stage_k : k_out, out ? ctx->stage_v : v_out, ctx->pool,
                                ctx->status, s));
    }
    if (out) {
      CUDA_TRY(cudaMemcpyAsync(k_out, ctx->stage_k, bytes, cudaMemcpyDefault, s));
      CUDA_TRY(cudaMemcpyAsync(v_out, ctx->stage_v, bytes, cudaMemcpyDefault, s));
    }
  }
  if (staged) ctx->stage_seq = ctx->seq;
  ctx->last_launches = 1;
  if (used) *used = sl;
  return finish_call(ctx, sl, s, chain);
}

static int resolve_host_ptr(const void* p, const void** dev) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    (void)cudaGetLastError();
    return fail(TPA_ERR_INVALID_ARG, "host pointer %p is not known to CUDA", p);
  }
  if (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged) {
    *dev = p;
    return TPA_OK;
  }
  if (at.type != cudaMemoryTypeHost)
    return fail(TPA_ERR_INVALID_ARG, "host memory %p is not pinned", p);
  void* d = nullptr;
  if (cudaHostGetDevicePointer(&d, const_cast<void*>(p), 0) != cudaSuccess || !d) {
    (void)cudaGetLastError();
    return fail(TPA_ERR_INVALID_ARG, "pinned host memory %p is not mapped", p);
  }
  *dev = d;
  return TPA_OK;
}

int tpa_prefix_write(tpa_ctx* ctx, int32_t agent, const void* k, const void* v, void* stream) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  if (agent < 0 || agent >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", agent);
  Agent& a = ctx->agents[agent];
  if (a.len < 0) return fail(TPA_ERR_STATE, "agent %d is not registered", agent);
  if (!a.resident) return fail(TPA_ERR_NOT_RESIDENT, "agent %d is not resident", agent);
  if (a.len == 0) return TPA_OK;
  if (!k || !v) return fail(TPA_ERR_INVALID_ARG, "null source");
  const void* kd = k;
  const void* vd = v;
  if (!ctx->plan_only) {
    int rc;
    if ((rc = resolve_host_ptr(k, &kd)) || (rc = resolve_host_ptr(v, &vd))) return rc;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  wait_for_seq(ctx, a.ready_seq, s);
  const int rc = page_copy_call(ctx, a.pages, a.len, 1, kd, vd, nullptr, nullptr, s, true,
                                a.last_use, nullptr);
  if (rc) return rc;
  a.last_use = ctx->seq;
  a.ready_seq = 0;
  return TPA_OK;
}

int tpa_prefix_evict(tpa_ctx* ctx, int32_t agent) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  if (agent < 0 || agent >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", agent);
  Agent& a = ctx->agents[agent];
  if (a.len < 0) return fail(TPA_ERR_STATE, "agent %d is not registered", agent);
  if (!a.resident) return fail(TPA_ERR_NOT_RESIDENT, "agent %d is already evicted", agent);
  give_pages(ctx, a.pages, std::max(a.last_use, a.ready_seq));
  a.resident = false;
  return TPA_OK;
}

int tpa_prefix_reload(tpa_ctx* ctx, int32_t agent, const void* host_k, const void* host_v,
                      void* side_stream, void* done_event) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  if (agent < 0 || agent >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", agent);
  Agent& a = ctx->agents[agent];
  if (a.len < 0) return fail(TPA_ERR_STATE, "agent %d is not registered", agent);
  if (a.resident) return fail(TPA_ERR_STATE, "agent %d is already resident", agent);
  if (a.len > 0 && (!host_k || !host_v)) return fail(TPA_ERR_INVALID_ARG, "null source");
  // pinned host (or device) memory only; the direct mode's kernel reads it
  // through its mapped device address
  const void* kd = host_k;
  const void* vd = host_v;
  if (!ctx->plan_only && a.len > 0) {
    int rc;
    if ((rc = resolve_host_ptr(host_k, &kd)) || (rc = resolve_host_ptr(host_v, &vd))) return rc;
  }
  const bool staged = ctx->staged_movement;
  const int64_t need = cdiv(a.len, kPage);
  if (need > free_count(ctx))
    return fail(TPA_ERR_NO_SPACE, "reload needs %lld pages, %lld free", (long long)need,
                (long long)free_count(ctx));
  std::vector<int32_t> pages;
  const uint64_t tag = take_pages(ctx, need, pages);
  cudaStream_t s = static_cast<cudaStream_t>(side_stream);
  const int rc = page_copy_call(ctx, pages, a.len, 1, staged ? host_k : kd, staged ? host_v : vd,
                                nullptr, nullptr, s, false, std::max(tag, a.last_use), nullptr,
                                staged);
  if (rc) {
    // give the pages back untouched (nothing was queued that writes them)
    for (auto it = pages.rbegin(); it != pages.rend(); ++it) ctx->free_pages[--ctx->free_head] = *it;
    return rc;
  }
  a.pages = std::move(pages);
  a.resident = true;
  a.ready_seq = ctx->seq;
  a.last_use = ctx->seq;
  if (done_event && !ctx->plan_only) CUDA_TRY(cudaEventRecord(static_cast<cudaEvent_t>(done_event), s));
  return TPA_OK;
}

int tpa_prefix_offload(tpa_ctx* ctx, int32_t agent, void* host_k, void* host_v, void* side_stream,
                       void* done_event) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  if (agent < 0 || agent >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", agent);
  Agent& a = ctx->agents[agent];
  if (a.len < 0) return fail(TPA_ERR_STATE, "agent %d is not registered", agent);
  if (!a.resident) return fail(TPA_ERR_NOT_RESIDENT, "agent %d is not resident", agent);
  if (a.len > 0 && (!host_k || !host_v)) return fail(TPA_ERR_INVALID_ARG, "null destination");
  // pinned host (or device) memory only; the direct mode's kernel writes it
  // through its mapped device address
  const void* kd = host_k;
  const void* vd = host_v;
  if (!ctx->plan_only && a.len > 0) {
    int rc;
    if ((rc = resolve_host_ptr(host_k, &kd)) || (rc = resolve_host_ptr(host_v, &vd))) return rc;
  }
  const bool staged = ctx->staged_movement;
  cudaStream_t s = static_cast<cudaStream_t>(side_stream);
  // the pages' last writer/readers must finish before the copy reads them
  wait_for_seq(ctx, ctx->chain_seq, s);
  const int rc = page_copy_call(ctx, a.pages, a.len, 0, nullptr, nullptr,
                                staged ? host_k : const_cast<void*>(kd),
                                staged ? host_v : const_cast<void*>(vd), s, false,
                                std::max(a.ready_seq, a.last_use), nullptr, staged);
  if (rc) return rc;
  a.last_use = ctx->seq;
  give_pages(ctx, a.pages, ctx->seq);
  a.resident = false;
  a.ready_seq = 0;
  if (done_event && !ctx->plan_only) CUDA_TRY(cudaEventRecord(static_cast<cudaEvent_t>(done_event), s));
  return TPA_OK;
}

// ---------------------------------------------------------------- requests

int tpa_request_open(tpa_ctx* ctx, int32_t req, int32_t agent) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  if (req < 0 || req >= ctx->cfg.max_requests) return fail(TPA_ERR_INVALID_ARG, "request id %d", req);
  if (agent < 0 || agent >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", agent);
  if (ctx->reqs[req].open) return fail(TPA_ERR_STATE, "request %d is already open", req);
  if (ctx->agents[agent].len < 0) return fail(TPA_ERR_STATE, "agent %d is not registered", agent);
  Request& r = ctx->reqs[req];
  r = Request();
  r.open = true;
  r.agent = agent;
  return TPA_OK;
}

int tpa_request_close(tpa_ctx* ctx, int32_t req) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  if (req < 0 || req >= ctx->cfg.max_requests) return fail(TPA_ERR_INVALID_ARG, "request id %d", req);
  Request& r = ctx->reqs[req];
  if (!r.open) return fail(TPA_ERR_STATE, "request %d is not open", req);
  give_pages(ctx, r.pages, r.last_use);
  r = Request();
  return TPA_OK;
}

int tpa_request_truncate(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* lens) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  int rc = check_batch(ctx, n, reqs, false);
  if (rc) return rc;
  if (!lens) return fail(TPA_ERR_INVALID_ARG, "null lengths");
  for (int i = 0; i < n; ++i)
    if (lens[i] < 0 || lens[i] > ctx->reqs[reqs[i]].len)
      return fail(TPA_ERR_INVALID_ARG, "truncate request %d to %d of %d tokens", reqs[i], lens[i],
                  ctx->reqs[reqs[i]].len);
  for (int i = 0; i < n; ++i) {
    Request& r = ctx->reqs[reqs[i]];
    const size_t keep = static_cast<size_t>(cdiv(lens[i], kPage));
    if (r.pages.size() > keep) {
      std::vector<int32_t> tail(r.pages.begin() + keep, r.pages.end());
      r.pages.resize(keep);
      give_pages(ctx, tail, r.last_use);
    }
    r.len = lens[i];
  }
  return TPA_OK;
}

// Reserve pages for appending ntok[i] tokens to request reqs[i]; all or nothing.
static int reserve_append(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* ntok,
                          uint64_t* tag) {
  int64_t need = 0;
  for (int i = 0; i < n; ++i) {
    const Request& r = ctx->reqs[reqs[i]];
    if (ntok[i] < 0) return fail(TPA_ERR_INVALID_ARG, "negative token count");
    if (static_cast<int64_t>(r.len) + ntok[i] > ctx->cfg.max_seq_len)
      return fail(TPA_ERR_CAPACITY, "suffix of request %d would exceed max_seq_len", reqs[i]);
    need += cdiv(r.len + ntok[i], kPage) - static_cast<int64_t>(r.pages.size());
  }
  if (need > free_count(ctx))
    return fail(TPA_ERR_NO_SPACE, "append needs %lld pages, %lld free", (long long)need,
                (long long)free_count(ctx));
  uint64_t t = 0;
  for (int i = 0; i < n; ++i) {
    Request& r = ctx->reqs[reqs[i]];
    const int64_t add = cdiv(r.len + ntok[i], kPage) - static_cast<int64_t>(r.pages.size());
    t = std::max(t, take_pages(ctx, add, r.pages));
  }
  *tag = t;
  return TPA_OK;
}

// Runs (one per page touched) of appending ntok[i] tokens after each
// request's current length: the count, and the records themselves (source
// rows follow the requests' order).
static int64_t append_runs(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* ntok) {
  int64_t runs = 0;
  for (int i = 0; i < n; ++i)
    if (ntok[i] > 0) runs += cdiv(ctx->reqs[reqs[i]].len % kPage + ntok[i], kPage);
  return runs;
}

static void write_append_rows(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* ntok,
                              AppendRow* rows) {
  int64_t run = 0;
  int32_t src = 0;
  for (int i = 0; i < n; ++i) {
    const Request& r = ctx->reqs[reqs[i]];
    for (int t = 0; t < ntok[i];) {
      const int pos = r.len + t;
      const int slot = pos % kPage;
      const int cnt = std::min(kPage - slot, ntok[i] - t);
      rows[run++] = AppendRow{src, r.pages[pos / kPage], slot, cnt};
      src += cnt;
      t += cnt;
    }
  }
}

int tpa_kv_append(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* ntok,
                  const void* k_new, const void* v_new, void* stream) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  int rc = check_batch(ctx, n, reqs, false);
  if (rc) return rc;
  if (!ntok) return fail(TPA_ERR_INVALID_ARG, "null token counts");
  int64_t total = 0;
  for (int i = 0; i < n; ++i) total += ntok[i] > 0 ? ntok[i] : 0;
  if (total > ctx->cfg.max_tokens) return fail(TPA_ERR_CAPACITY, "%lld tokens > max_tokens", (long long)total);
  if (total > 0 && (!k_new || !v_new)) return fail(TPA_ERR_INVALID_ARG, "null K/V");
  uint64_t tag = 0;
  if ((rc = reserve_append(ctx, n, reqs, ntok, &tag))) return rc;
  Slot* sl = acquire_slot(ctx);
  ++ctx->seq;
  PlanSizes sz;
  const int64_t runs = append_runs(ctx, n, reqs, ntok);
  sz.append = runs;
  const PlanLayout lay = layout_of(sz);
  PlanWriter w(sl->host, lay);
  w.hdr->n_append = static_cast<int32_t>(runs);
  write_append_rows(ctx, n, reqs, ntok, w.append);
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  chain_begin(ctx, s);
  wait_for_seq(ctx, tag, s);
  if ((rc = upload(ctx, sl, lay.total, s))) return rc;
  if (!ctx->plan_only) {
    KernelTimer kt(ctx, K_APPEND, s);
    CUDA_TRY(launch_append(dev_ptr<AppendRow>(sl, lay.off_append), static_cast<int>(runs), k_new,
                           v_new, ctx->pool, ctx->status, s));
  }
  for (int i = 0; i < n; ++i) {
    Request& r = ctx->reqs[reqs[i]];
    r.len += ntok[i];
    r.last_use = ctx->seq;
  }
  ctx->last_launches = 1;
  ctx->last_dense = ctx->last_suffix = 0;
  return finish_call(ctx, sl, s, true);
}

// ------------------------------------------------------------- attention

namespace {

struct AgentGroup {
  int32_t agent;
  std::vector<int32_t> toks;  // positions in the batch
  int32_t page_off = 0;       // prefix pages in the plan's page list
  int32_t n_split = 0;        // key splits of the prefix level
  int32_t tiles_per_split = 0;
};

}  // namespace

// Fill the DenseParams common to every dense launch.
static DenseParams dense_params(tpa_ctx* ctx, const Slot* sl, const PlanLayout& lay, int n_items,
                                const void* q, void* out, float* lse) {
  DenseParams dp{};
  dp.tmap_k = ctx->tmap_k;
  dp.tmap_v = ctx->tmap_v;
  dp.run_maps = ctx->run_maps;
  dp.q = static_cast<const __nv_bfloat16*>(q);
  dp.out = static_cast<__nv_bfloat16*>(out);
  dp.lse = lse;
  dp.part_o = ctx->part_o;
  dp.part_lse = ctx->part_lse;
  dp.part_slots = ctx->part_slots;
  dp.items = dev_ptr<DenseItem>(sl, lay.off_dense);
  dp.toks = dev_ptr<DenseTok>(sl, lay.off_dense_tok);
  dp.pages = dev_ptr<int32_t>(sl, lay.off_pages);
  dp.k_pool = static_cast<__nv_bfloat16*>(ctx->cfg.k_pool);
  dp.v_pool = static_cast<__nv_bfloat16*>(ctx->cfg.v_pool);
  dp.status = ctx->status;
  dp.num_pages = ctx->cfg.num_pages;
  dp.n_items = n_items;
  dp.hq = ctx->hq;
  dp.hkv = ctx->hkv;
  dp.scale_log2 = 1.4426950408889634f / std::sqrt(static_cast<float>(ctx->d));
  return dp;
}

// Build and launch a decode step.
//  cascade (default): one persistent tcgen05 launch.  Work items are the
//    stacked shared-prefix tiles of each agent (level 1) and, per token and
//    kv head, its suffix (level 2, which also appends the step's token);
//    then the LSE merge, launched as its programmatic dependent.
//  flat (cross-check): KV append, the split-KV kernel over every key of
//    each request (prefix included), and a separate LSE merge.
int tpa_decode(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const void* q, const void* k_new,
               const void* v_new, void* out, float* lse, void* stream) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  int rc = check_batch(ctx, n, reqs, true);
  if (rc) return rc;
  if (!ctx->plan_only && (!q || !k_new || !v_new || !out || !lse))
    return fail(TPA_ERR_INVALID_ARG, "null tensor");
  const int G = ctx->group, hkv = ctx->hkv, hq = ctx->hq;
  const int tpt = kTileRows / G;
  const bool flat = ctx->decode_mode == 1;

  // group tokens by agent (first appearance order)
  std::vector<AgentGroup> groups;
  std::vector<int32_t> group_of(n);
  {
    const uint64_t st = ++ctx->stamp;
    for (int i = 0; i < n; ++i) {
      const int32_t a = ctx->reqs[reqs[i]].agent;
      if (ctx->agent_stamp[a] != st) {
        ctx->agent_stamp[a] = st;
        ctx->agent_group[a] = static_cast<int32_t>(groups.size());
        groups.push_back(AgentGroup{a, {}});
        groups.back().toks.reserve(n);
      }
      group_of[i] = ctx->agent_group[a];
      groups[group_of[i]].toks.push_back(i);
    }
  }
  auto keys_of = [&](int i) -> int64_t { return ctx->reqs[reqs[i]].len + 1; };  // with the new token
  auto lp_of = [&](int i) -> int64_t { return ctx->agents[ctx->reqs[reqs[i]].agent].len; };

  // ---- work decomposition -------------------------------------------------
  int64_t split_keys = 0;  // suffix (and, flat, prefix) key range per item
  int dense_ctas = 0;      // cascade: CTAs running the stacked prefix tiles
  if (flat) {
    int64_t sum_keys = 0;
    for (int i = 0; i < n; ++i) sum_keys += keys_of(i) + lp_of(i);
    split_keys = ctx->suffix_split_keys;
    if (split_keys <= 0) {
      // about two items per resident warp of the split-KV kernel
      const int64_t warps = static_cast<int64_t>(ctx->num_sms) * 8;
      split_keys = std::min<int64_t>(std::max<int64_t>(cdiv(sum_keys * hkv, 2 * warps), 64), 1024);
    }
    split_keys = cdiv(split_keys, kPage) * kPage;
    for (;;) {
      int64_t worst = 0;
      for (int i = 0; i < n; ++i)
        worst = std::max(worst, cdiv(keys_of(i), split_keys) + cdiv(lp_of(i), split_keys));
      if (worst <= ctx->max_splits) break;
      split_keys *= 2;
    }
  } else {
    // Level 1 (dense CTAs): stacked prefix tiles, each split into `sp` key
    // ranges; level 2 (split-KV CTAs): the suffixes.  The split count and the
    // number of dense CTAs are chosen together so that every dense CTA gets
    // the same whole number m of (near-equal) items while the split-KV CTAs
    // finish at about the same time: the dense level is tensor-heavy and the
    // split level HBM-heavy, so the two run side by side (a dense CTA that is
    // done early still joins the split-KV work).  Rates measured on GB300
    // with both roles streaming: a dense 128x128 tile ~2 us, plus ~2 us per
    // item (the next item's Q is loaded once the previous item's last QK is
    // done); split-KV ~50 GB/s of KV per SM.  Ties go to fewer splits.
    constexpr double kTileUs = 2.0, kItemUs = 2.0, kSplitBytesPerUs = 50e3;
    double split_bytes = 0;
    for (int i = 0; i < n; ++i) split_bytes += static_cast<double>(keys_of(i)) * hkv * 4.0 * ctx->d;
    const double w_split = split_bytes / kSplitBytesPerUs;  // SM-microseconds
    int64_t ptiles_max = 0;
    for (auto& g : groups) ptiles_max = std::max<int64_t>(ptiles_max, cdiv(ctx->agents[g.agent].len, kTileKeys));
    int best_sp = 1, best_d = 0;
    double best_t = 1e300;
    if (ptiles_max > 0) {
      const int sp_lo = ctx->prefix_splits > 0 ? ctx->prefix_splits : 1;
      const int sp_hi = ctx->prefix_splits > 0 ? ctx->prefix_splits
                                               : static_cast<int>(std::min<int64_t>(16, ptiles_max));
      for (int sp = sp_lo; sp <= sp_hi; ++sp) {
        int64_t items = 0, kmax = 0;
        for (auto& g : groups) {
          const int64_t pt = cdiv(ctx->agents[g.agent].len, kTileKeys);
          if (pt == 0) continue;
          const int64_t k = cdiv(pt, std::min<int64_t>(sp, pt));
          items += static_cast<int64_t>(hkv) * cdiv(g.toks.size(), tpt) * cdiv(pt, k);
          kmax = std::max(kmax, k);
        }
        for (int m = 1; m <= 8; ++m) {
          int d = static_cast<int>(cdiv(items, m));
          if (d > ctx->num_sms - (w_split > 0 ? 1 : 0)) continue;
          const double t_dense = (kTileUs * kmax + kItemUs) * m;
          const double t_split = w_split > 0 ? w_split / (ctx->num_sms - d) : 0.0;
          const double t = std::max(t_dense, t_split);
          if (t < best_t) {
            best_t = t;
            best_sp = sp;
            best_d = d;
          }
        }
      }
      if (best_d == 0) {  // more items than SMs at m <= 8: all but one SM dense
        best_sp = sp_lo;
        best_d = ctx->num_sms - (w_split > 0 ? 1 : 0);
      }
    }
    dense_ctas = best_d;
    for (auto& g : groups) {
      const int64_t ptiles = cdiv(ctx->agents[g.agent].len, kTileKeys);
      if (ptiles == 0) continue;
      const int64_t ns = std::min<int64_t>(best_sp, ptiles);
      g.tiles_per_split = static_cast<int32_t>(cdiv(ptiles, ns));
      g.n_split = static_cast<int32_t>(cdiv(ptiles, g.tiles_per_split));
      if (g.n_split >= ctx->max_splits)
        return fail(TPA_ERR_CAPACITY, "prefix splits exceed max_splits");
    }
    // Level 2 (split-KV role): about two items per split-KV warp, rounded up
    // to a power of two keys, 64..1024.  (Measured on GB300: with late item
    // claims the step times of the suffix-key sweep dip at 256 and 512 keys
    // and are flat near 1024, so rounding up costs nothing where it does not
    // help.)
    int64_t sum_keys = 0;
    for (int i = 0; i < n; ++i) sum_keys += keys_of(i);
    split_keys = ctx->suffix_split_keys;
    if (split_keys <= 0) {
      const int64_t warps = static_cast<int64_t>(ctx->num_sms) * 6;
      const int64_t target = std::min<int64_t>(std::max<int64_t>(cdiv(sum_keys * hkv, 2 * warps), 64), 1024);
      split_keys = 64;
      while (split_keys < target) split_keys *= 2;
    }
    split_keys = cdiv(split_keys, kPage) * kPage;
    for (;;) {
      int64_t worst = 0;
      for (int i = 0; i < n; ++i)
        worst = std::max<int64_t>(worst, groups[group_of[i]].n_split + cdiv(keys_of(i), split_keys));
      if (worst <= ctx->max_splits) break;
      split_keys *= 2;
    }
  }

  // partial slots per token
  std::vector<int32_t> slot_base(n), n_slots(n);
  int64_t slots = 0;
  for (int i = 0; i < n; ++i) {
    const int64_t ns = flat ? cdiv(lp_of(i), split_keys) + cdiv(keys_of(i), split_keys)
                            : groups[group_of[i]].n_split + cdiv(keys_of(i), split_keys);
    n_slots[i] = static_cast<int32_t>(ns);
    slot_base[i] = static_cast<int32_t>(slots);
    slots += static_cast<int64_t>(hq) * ns;
  }
  if (slots > ctx->part_slots) return fail(TPA_ERR_CAPACITY, "partial slots exhausted");
  if (ctx->test_bad_slot && n > 0) {
    // every kernel checks partial slots against the buffer: nothing of this
    // token's partials is written or read
    slot_base[0] = static_cast<int32_t>(std::min<int64_t>(ctx->part_slots, INT32_MAX));
    ctx->test_bad_slot = 0;
  }

  // plan sizes (suffix page counts after this step's append)
  PlanSizes sz;
  for (auto& g : groups) sz.pages += ctx->agents[g.agent].pages.size();
  for (int i = 0; i < n; ++i) sz.pages += cdiv(keys_of(i), kPage);
  if (flat) {
    sz.append = n;
    sz.merge = n;
    for (int i = 0; i < n; ++i)
      sz.suffix += hkv * (cdiv(keys_of(i), split_keys) + cdiv(lp_of(i), split_keys));
  } else {
    sz.dense_tok = n;
    sz.merge = n;
    for (auto& g : groups) sz.dense += static_cast<int64_t>(hkv) * cdiv(g.toks.size(), tpt) * g.n_split;
    sz.stok = n;
    sz.sint = 2 * static_cast<int64_t>(n) + 1;
  }
  const PlanLayout lay = layout_of(sz);
  if (lay.total > ctx->plan_cap)
    return fail(TPA_ERR_CAPACITY, "plan of %zu bytes > %zu", lay.total, ctx->plan_cap);

  // pages for the new tokens (all checks are done: from here on only CUDA errors can fail)
  std::vector<int32_t> ones(n, 1);
  uint64_t tag = 0;
  if ((rc = reserve_append(ctx, n, reqs, ones.data(), &tag))) return rc;

  Slot* sl = acquire_slot(ctx);
  ++ctx->seq;
  PlanWriter w(sl->host, lay);

  // page list: prefixes, then each token's suffix (after the append)
  int32_t np = 0;
  for (auto& g : groups) {
    const Agent& a = ctx->agents[g.agent];
    g.page_off = np;
    std::memcpy(w.pages + np, a.pages.data(), a.pages.size() * 4);
    np += static_cast<int32_t>(a.pages.size());
  }
  if (ctx->test_bad_page && !groups.empty() && !ctx->agents[groups[0].agent].pages.empty()) {
    // a read-only prefix page: every kernel read of it is bounds-checked
    w.pages[0] = static_cast<int32_t>(ctx->cfg.num_pages);
    ctx->test_bad_page = 0;
  }
  std::vector<int32_t> suf_off(n);
  for (int i = 0; i < n; ++i) {
    const Request& r = ctx->reqs[reqs[i]];
    suf_off[i] = np;
    std::memcpy(w.pages + np, r.pages.data(), r.pages.size() * 4);
    np += static_cast<int32_t>(r.pages.size());
  }

  int32_t nd = 0, ns = 0, nt = 0, n_full = 0;
  if (flat) {
    write_append_rows(ctx, n, reqs, ones.data(), w.append);
    for (int i = 0; i < n; ++i) w.merge[i] = MergeTok{i, slot_base[i], n_slots[i], 0};
    for (int i = 0; i < n; ++i) {
      int split = 0;
      for (int pass = 0; pass < 2; ++pass) {
        const int64_t len = pass == 0 ? lp_of(i) : keys_of(i);
        const int32_t base = pass == 0 ? groups[group_of[i]].page_off : suf_off[i];
        for (int64_t k0 = 0; k0 < len; k0 += split_keys, ++split)
          for (int h = 0; h < hkv; ++h)
            w.suffix[ns++] = SuffixItem{i, h, static_cast<int32_t>(base + k0 / kPage),
                                        static_cast<int32_t>(std::min<int64_t>(split_keys, len - k0)),
                                        slot_base[i], n_slots[i], split, -1, 0, {0, 0, 0}};
      }
    }
    std::stable_sort(w.suffix, w.suffix + ns,
                     [](const SuffixItem& a, const SuffixItem& b) { return a.n_keys > b.n_keys; });
  } else {
    for (int i = 0; i < n; ++i) w.merge[i] = MergeTok{i, slot_base[i], n_slots[i], 0};
    // level 1: stacked prefix tiles of each agent
    for (auto& g : groups) {
      if (g.n_split == 0) continue;
      const int64_t lp = ctx->agents[g.agent].len;
      const int nqt = static_cast<int>(cdiv(g.toks.size(), tpt));
      for (int qt = 0; qt < nqt; ++qt) {
        const int t0 = qt * tpt;
        const int t1 = std::min<int>(static_cast<int>(g.toks.size()), t0 + tpt);
        const int32_t tok_base = nt;
        for (int t = t0; t < t1; ++t) {
          const int i = g.toks[t];
          w.dtok[nt++] = DenseTok{i, 0x7fffffff, slot_base[i], n_slots[i]};
        }
        for (int h = 0; h < hkv; ++h)
          for (int sp = 0; sp < g.n_split; ++sp) {
            DenseItem it{};
            it.tok_base = tok_base;
            it.n_tok = t1 - t0;
            it.kv_head = h;
            it.split = sp;
            it.out_mode = 0;
            it.seg_pages[0] = g.page_off;
            it.seg_k0[0] = static_cast<int32_t>(static_cast<int64_t>(sp) * g.tiles_per_split * kTileKeys);
            it.seg_k1[0] = static_cast<int32_t>(
                std::min<int64_t>(lp, static_cast<int64_t>(sp + 1) * g.tiles_per_split * kTileKeys));
            it.n_tiles = static_cast<int32_t>(cdiv(it.seg_k1[0] - it.seg_k0[0], kTileKeys));
            w.dense[nd++] = it;
          }
      }
    }
    // level 2: one record per token; the split-KV warps derive the items
    // (full key ranges first, then the tails by decreasing length) and the
    // item holding a request's last key appends the step's token first
    int32_t* full_prefix = w.sint;
    int32_t* tail_order = w.sint + n + 1;
    full_prefix[0] = 0;
    std::vector<int32_t>& ord = ctx->order;
    ord.clear();
    for (int i = 0; i < n; ++i) {
      const Request& r = ctx->reqs[reqs[i]];
      const int64_t keys = keys_of(i);
      const int pos = r.len;  // slot of the new token
      w.stok[i] = SplitTok{i, suf_off[i], static_cast<int32_t>(keys), slot_base[i], n_slots[i],
                           groups[group_of[i]].n_split, r.pages[pos / kPage] * kPage + pos % kPage, 0};
      full_prefix[i + 1] = full_prefix[i] + static_cast<int32_t>(keys / split_keys);
      if (keys % split_keys) ord.push_back(i);
    }
    std::sort(ord.begin(), ord.end(), [&](int32_t x, int32_t y) {
      const int64_t rx = keys_of(x) % split_keys, ry = keys_of(y) % split_keys;
      return rx != ry ? rx > ry : x < y;
    });
    for (size_t t = 0; t < ord.size(); ++t) tail_order[t] = ord[t];
    n_full = full_prefix[n];
    ns = hkv * (n_full + static_cast<int32_t>(ord.size()));
    std::stable_sort(w.dense, w.dense + nd,
                     [](const DenseItem& a, const DenseItem& b) { return a.n_tiles > b.n_tiles; });
  }

  PlanHeader* hd = w.hdr;
  hd->n_pages = np;
  hd->n_append = flat ? n : 0;
  hd->n_dense_tok = nt;
  hd->n_dense = nd;
  hd->n_suffix = ns;
  hd->n_merge = n;

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  chain_begin(ctx, s);
  wait_for_seq(ctx, tag, s);
  for (auto& g : groups) wait_for_seq(ctx, ctx->agents[g.agent].ready_seq, s);
  const unsigned long long* plan_flag = nullptr;
  if ((rc = flat ? upload(ctx, sl, lay.total, s) : upload_ahead(ctx, sl, lay.total, &plan_flag)))
    return rc;

  int launches = 0;
  if (!ctx->plan_only) {
    const float scale_log2 = 1.4426950408889634f / std::sqrt(static_cast<float>(ctx->d));
    if (flat) {
      {
        KernelTimer kt(ctx, K_APPEND, s);
        CUDA_TRY(launch_append(dev_ptr<AppendRow>(sl, lay.off_append), n, k_new, v_new, ctx->pool,
                               ctx->status, s));
      }
      SuffixParams sp{};
      sp.tmap_k = ctx->tmap_k;
      sp.tmap_v = ctx->tmap_v;
      sp.q = static_cast<const __nv_bfloat16*>(q);
      sp.part_o = ctx->part_o;
      sp.part_lse = ctx->part_lse;
      sp.part_slots = ctx->part_slots;
      sp.items = dev_ptr<SuffixItem>(sl, lay.off_suffix);
      sp.pages = dev_ptr<int32_t>(sl, lay.off_pages);
      sp.queue = reinterpret_cast<uint32_t*>(sl->dev + offsetof(PlanHeader, queue));
      sp.status = ctx->status;
      sp.num_pages = ctx->cfg.num_pages;
      sp.n_items = ns;
      sp.hq = hq;
      sp.hkv = hkv;
      sp.scale_log2 = scale_log2;
      {
        KernelTimer kt(ctx, K_SUFFIX, s);
        CUDA_TRY(launch_suffix(sp, ctx->num_sms, ctx->d, G, s));
      }
      {
        KernelTimer kt(ctx, K_MERGE, s);
        CUDA_TRY(launch_merge(dev_ptr<MergeTok>(sl, lay.off_merge), n, ctx->part_o, ctx->part_lse,
                              ctx->part_slots, ctx->status,
                              static_cast<__nv_bfloat16*>(out), lse, hq, ctx->d, ctx->num_sms,
                              true, nullptr, 0, s));
      }
      launches = 3;
    } else {
      // one launch, one CTA per SM: dense CTAs for level 1, the rest split-KV
      const int n_dense = std::min(dense_ctas, nd);
      const int n_split = ns > 0 ? std::min<int>(ctx->num_sms - n_dense,
                                                 static_cast<int>(cdiv(ns, kSplitWarpsPerCta)))
                                 : 0;
      DenseParams dp = dense_params(ctx, sl, lay, nd, q, out, lse);
      dp.n_dense_ctas = n_dense;
      dp.stoks = dev_ptr<SplitTok>(sl, lay.off_stok);
      dp.full_prefix = dev_ptr<int32_t>(sl, lay.off_sint);
      dp.tail_order = dev_ptr<int32_t>(sl, lay.off_sint) + n + 1;
      dp.n_stok = n;
      dp.n_full = n_full;
      dp.split_keys = static_cast<int32_t>(split_keys);
      dp.n_sitems = ns;
      dp.squeue = reinterpret_cast<uint32_t*>(sl->dev + offsetof(PlanHeader, queue));
      dp.k_new = static_cast<const __nv_bfloat16*>(k_new);
      dp.v_new = static_cast<const __nv_bfloat16*>(v_new);
      {
          KernelTimer kt(ctx, K_DENSE, s);
        dp.plan_flag = plan_flag;
        dp.plan_seq = ctx->seq;
        if (ctx->test_plan_wait) {  // a value the flag word never takes
          dp.plan_seq = ctx->seq | (1ull << 63);
          ctx->test_plan_wait = 0;
        }
        // a programmatic dependent of the previous step's merge on this stream
        CUDA_TRY(launch_dense(dp, n_split, ctx->d, G, true, s));
      }
      {
        // a programmatic dependent: resident before the main kernel ends
        KernelTimer kt(ctx, K_MERGE, s);
        CUDA_TRY(launch_merge(dev_ptr<MergeTok>(sl, lay.off_merge), n, ctx->part_o, ctx->part_lse,
                              ctx->part_slots, ctx->status,
                              static_cast<__nv_bfloat16*>(out), lse, hq, ctx->d, ctx->num_sms,
                              true, dp.plan_flag, dp.plan_seq, s));
      }
      launches = 2;
    }
  }
  for (int i = 0; i < n; ++i) {
    Request& r = ctx->reqs[reqs[i]];
    r.len += 1;
    r.last_use = ctx->seq;
  }
  for (auto& g : groups) ctx->agents[g.agent].last_use = ctx->seq;
  ctx->last_dense = nd;
  ctx->last_suffix = ns;
  ctx->last_launches = launches;
  return finish_call(ctx, sl, s, true);
}

int tpa_prefill_chunk(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* chunk_len,
                      const void* q, const void* k_new, const void* v_new, void* out, float* lse,
                      void* stream) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  int rc = check_batch(ctx, n, reqs, true);
  if (rc) return rc;
  if (!chunk_len) return fail(TPA_ERR_INVALID_ARG, "null chunk lengths");
  int64_t total = 0;
  for (int i = 0; i < n; ++i) {
    if (chunk_len[i] <= 0) return fail(TPA_ERR_INVALID_ARG, "chunk length %d", chunk_len[i]);
    total += chunk_len[i];
  }
  if (total > ctx->cfg.max_tokens) return fail(TPA_ERR_CAPACITY, "%lld tokens > max_tokens", (long long)total);
  if (!ctx->plan_only && (!q || !k_new || !v_new || !out || !lse))
    return fail(TPA_ERR_INVALID_ARG, "null tensor");
  const int G = ctx->group, hkv = ctx->hkv;
  const bool pairs = ctx->prefill_rows == 2 * kTileRows;
  const int tpt = (pairs ? 2 * kTileRows : kTileRows) / G;  // tokens per work item

  cudaStream_t s = static_cast<cudaStream_t>(stream);
  std::vector<int32_t> offset(n);
  for (int i = 0; i < n; ++i) offset[i] = ctx->reqs[reqs[i]].len;
  // Chunks of an agent whose prefix reload (on another stream) is still in
  // flight run in a second launch after the stream waits for that reload;
  // the other chunks' items run meanwhile.  Only the requests that need an
  // incoming prefix wait for its movement (Sec. IV-B, Eq. 7).
  std::vector<uint8_t> late(n, 0);
  {
    bool any_early = false, any_late = false;
    for (int i = 0; i < n; ++i) {
      late[i] = seq_pending(ctx, ctx->agents[ctx->reqs[reqs[i]].agent].ready_seq, s) ? 1 : 0;
      (late[i] ? any_late : any_early) = true;
    }
    if (!any_early || !any_late) std::fill(late.begin(), late.end(), 0);
  }

  std::vector<int32_t> agents_seen;
  PlanSizes sz;
  const int64_t runs = append_runs(ctx, n, reqs, chunk_len);
  sz.append = runs;
  sz.dense_tok = pairs ? 0 : total;  // paired items derive their tokens from row0 / pos0
  std::unordered_map<int32_t, int32_t> agent_off;
  for (int i = 0; i < n; ++i) {
    const int32_t a = ctx->reqs[reqs[i]].agent;
    if (!agent_off.count(a)) {
      agent_off[a] = 0;
      agents_seen.push_back(a);
      sz.pages += ctx->agents[a].pages.size();
    }
    sz.pages += cdiv(offset[i] + chunk_len[i], kPage);
    sz.dense += static_cast<int64_t>(hkv) * cdiv(chunk_len[i], tpt);
  }
  const PlanLayout lay = layout_of(sz);
  if (lay.total > ctx->plan_cap) return fail(TPA_ERR_CAPACITY, "plan of %zu bytes > %zu", lay.total, ctx->plan_cap);
  uint64_t tag = 0;
  if ((rc = reserve_append(ctx, n, reqs, chunk_len, &tag))) return rc;

  Slot* sl = acquire_slot(ctx);
  ++ctx->seq;
  PlanWriter w(sl->host, lay);
  int32_t np = 0;
  for (int32_t a : agents_seen) {
    agent_off[a] = np;
    const Agent& ag = ctx->agents[a];
    std::memcpy(w.pages + np, ag.pages.data(), ag.pages.size() * 4);
    np += static_cast<int32_t>(ag.pages.size());
  }
  write_append_rows(ctx, n, reqs, chunk_len, w.append);  // positions before this call
  // Items go straight to their place, the early chunks' items first, each
  // group in longest-first order (a stable counting sort on the key-tile
  // count): first count the items of each length, then write them.
  auto tiles_of = [&](int i, int t1) {
    const int64_t lp = ctx->agents[ctx->reqs[reqs[i]].agent].len;
    return static_cast<int32_t>(cdiv(lp, kTileKeys) + cdiv(offset[i] + t1, kTileKeys));
  };
  int32_t max_tiles = 0;  // a request's last tile has the most keys
  for (int i = 0; i < n; ++i) max_tiles = std::max(max_tiles, tiles_of(i, chunk_len[i]));
  const size_t n_len = static_cast<size_t>(max_tiles) + 1;
  std::vector<int32_t> at(2 * n_len, 0);  // [group][key tiles]
  for (int i = 0; i < n; ++i)
    for (int t0 = 0; t0 < chunk_len[i]; t0 += tpt)
      at[late[i] * n_len + tiles_of(i, std::min(chunk_len[i], t0 + tpt))] += hkv;
  int32_t n_early = 0;
  for (int g = 0, acc = 0; g < 2; ++g) {  // exclusive prefix, longest first
    for (size_t k = n_len; k-- > 0;) {
      const int32_t c = at[g * n_len + k];
      at[g * n_len + k] = acc;
      acc += c;
    }
    if (g == 0) n_early = acc;
  }
  int32_t nt = 0, nd = 0;
  int64_t row0 = 0;
  for (int i = 0; i < n; ++i) {
    const Request& r = ctx->reqs[reqs[i]];
    const int64_t lp = ctx->agents[r.agent].len;
    const int32_t suf = np;
    std::memcpy(w.pages + np, r.pages.data(), r.pages.size() * 4);
    np += static_cast<int32_t>(r.pages.size());
    const int c = chunk_len[i];
    for (int t0 = 0; t0 < c; t0 += tpt) {
      const int t1 = std::min(c, t0 + tpt);
      DenseItem it{};
      if (pairs) {
        it.tok_base = -1;
        it.row0 = static_cast<int32_t>(row0 + t0);
        it.pos0 = offset[i] + t0;
      } else {
        it.tok_base = nt;
        for (int t = t0; t < t1; ++t)
          w.dtok[nt++] = DenseTok{static_cast<int32_t>(row0 + t), offset[i] + t, 0, 0};
      }
      it.n_tok = t1 - t0;
      it.out_mode = 1;
      it.seg_pages[0] = agent_off[r.agent];
      it.seg_k0[0] = 0;
      it.seg_k1[0] = static_cast<int32_t>(lp);
      it.seg_pages[1] = suf;
      it.seg_k0[1] = 0;
      it.seg_k1[1] = offset[i] + t1;  // keys up to the tile's last position
      it.seg_causal[1] = 1;
      it.n_tiles = tiles_of(i, t1);
      int32_t& pos = at[late[i] * n_len + it.n_tiles];
      DenseItem* dst = w.dense + pos;
      pos += hkv;
      for (int h = 0; h < hkv; ++h) {
        it.kv_head = h;
        dst[h] = it;
      }
      nd += hkv;
    }
    row0 += c;
  }
  PlanHeader* hd = w.hdr;
  hd->n_pages = np;
  hd->n_append = static_cast<int32_t>(runs);
  hd->n_dense_tok = nt;
  hd->n_dense = nd;

  chain_begin(ctx, s);
  wait_for_seq(ctx, tag, s);
  if ((rc = upload(ctx, sl, lay.total, s))) return rc;
  if (!ctx->plan_only) {
    {
      KernelTimer kt(ctx, K_APPEND, s);
      CUDA_TRY(launch_append(dev_ptr<AppendRow>(sl, lay.off_append), static_cast<int>(runs), k_new,
                             v_new, ctx->pool, ctx->status, s));
    }
    // items [0, n_early) after the reloads of their agents (if any is
    // still pending, no chunk is late), then the late ones after theirs
    for (int g = 0; g < 2; ++g) {
      const int32_t i0 = g == 0 ? 0 : n_early, i1 = g == 0 ? n_early : nd;
      for (int i = 0; i < n; ++i)
        if (late[i] == g) wait_for_seq(ctx, ctx->agents[ctx->reqs[reqs[i]].agent].ready_seq, s);
      if (i1 == i0) continue;
      DenseParams dp = dense_params(ctx, sl, lay, i1 - i0, q, out, lse);
      dp.items += i0;
      dp.n_dense_ctas = std::min(i1 - i0, ctx->num_sms);
      KernelTimer kt(ctx, pairs ? K_PREFILL_PAIR : K_DENSE, s);
      if (pairs)
        CUDA_TRY(launch_prefill_pair(dp, dp.n_dense_ctas, ctx->d, G, s));
      else
        CUDA_TRY(launch_dense(dp, 0, ctx->d, G, false, s));
    }
  }
  for (int i = 0; i < n; ++i) {
    Request& r = ctx->reqs[reqs[i]];
    r.len += chunk_len[i];
    r.last_use = ctx->seq;
  }
  for (int32_t a : agents_seen) ctx->agents[a].last_use = ctx->seq;
  ctx->last_dense = nd;
  ctx->last_suffix = 0;
  ctx->last_launches = 2;
  return finish_call(ctx, sl, s, true);
}

int tpa_decode_static_scratch(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const void* q,
                              const void* k_new, const void* v_new, void* out, float* lse,
                              void* stream) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  // [slots][d] fp32 partial outputs, then [slots] fp32 partial LSEs
  const size_t bytes = static_scratch_bytes();
  const int64_t slots = static_cast<int64_t>((bytes - kAlign) / ((ctx->d + 1) * sizeof(float)));
  void* base = nullptr;
  if (!ctx->plan_only) {
    const cudaError_t e = static_scratch(ctx->device, &base);
    if (e != cudaSuccess)
      return fail(TPA_ERR_CUDA, "static scratch address: %s", cudaGetErrorString(e));
  }
  float* const saved_o = ctx->part_o;
  float* const saved_lse = ctx->part_lse;
  const int64_t saved_slots = ctx->part_slots;
  ctx->part_o = static_cast<float*>(base);
  ctx->part_lse = base ? reinterpret_cast<float*>(static_cast<uint8_t*>(base) +
                                                  align_up(slots * ctx->d * sizeof(float), kAlign))
                       : nullptr;
  ctx->part_slots = slots;
  int rc = tpa_decode(ctx, n, reqs, q, k_new, v_new, out, lse, stream);
  ctx->part_o = saved_o;
  ctx->part_lse = saved_lse;
  ctx->part_slots = saved_slots;
  if (rc == TPA_ERR_CAPACITY && g_err == "partial slots exhausted")
    rc = fail(TPA_ERR_CAPACITY,
              "decode needs more split partials than the %zu-byte static scratch holds "
              "(%lld slots of head_dim %d)",
              bytes, static_cast<long long>(slots), ctx->d);
  return rc;
}

int tpa_gather(tpa_ctx* ctx, int32_t id, int32_t is_request, void* k_out, void* v_out,
               void* stream) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  const std::vector<int32_t>* pages;
  int len;
  if (is_request) {
    if (id < 0 || id >= ctx->cfg.max_requests) return fail(TPA_ERR_INVALID_ARG, "request id %d", id);
    if (!ctx->reqs[id].open) return fail(TPA_ERR_STATE, "request %d is not open", id);
    pages = &ctx->reqs[id].pages;
    len = ctx->reqs[id].len;
  } else {
    if (id < 0 || id >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", id);
    const Agent& a = ctx->agents[id];
    if (a.len < 0) return fail(TPA_ERR_STATE, "agent %d is not registered", id);
    if (!a.resident) return fail(TPA_ERR_NOT_RESIDENT, "agent %d is not resident", id);
    pages = &a.pages;
    len = a.len;
  }
  if (len == 0) return TPA_OK;
  if (!k_out || !v_out) return fail(TPA_ERR_INVALID_ARG, "null destination");
  const void* kd = k_out;
  const void* vd = v_out;
  if (!ctx->plan_only) {
    int rc;
    if ((rc = resolve_host_ptr(k_out, &kd)) || (rc = resolve_host_ptr(v_out, &vd))) return rc;
  }
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  const uint64_t ready = is_request ? 0 : ctx->agents[id].ready_seq;
  const int rc = page_copy_call(ctx, *pages, len, 0, nullptr, nullptr, const_cast<void*>(kd),
                                const_cast<void*>(vd), s, true, ready, nullptr);
  if (rc) return rc;
  if (is_request) ctx->reqs[id].last_use = ctx->seq;
  else ctx->agents[id].last_use = ctx->seq;
  return TPA_OK;
}

int tpa_query(tpa_ctx* ctx, int32_t what, int32_t id, int64_t* value) {
  if (!ctx || !value) return fail(TPA_ERR_INVALID_ARG, "null argument");
  switch (what) {
    case TPA_Q_FREE_PAGES: *value = free_count(ctx); return TPA_OK;
    case TPA_Q_PREFIX_LEN:
    case TPA_Q_PREFIX_RESIDENT:
    case TPA_Q_PAGE_OF:
      if (id < 0 || id >= ctx->cfg.max_agents) return fail(TPA_ERR_INVALID_ARG, "agent id %d", id);
      if (what == TPA_Q_PREFIX_LEN) *value = ctx->agents[id].len;
      else if (what == TPA_Q_PREFIX_RESIDENT)
        *value = ctx->agents[id].len < 0 ? -1 : (ctx->agents[id].resident ? 1 : 0);
      else
        *value = ctx->agents[id].pages.empty() ? -1 : ctx->agents[id].pages[0];
      return TPA_OK;
    case TPA_Q_SUFFIX_LEN:
      if (id < 0 || id >= ctx->cfg.max_requests) return fail(TPA_ERR_INVALID_ARG, "request id %d", id);
      *value = ctx->reqs[id].open ? ctx->reqs[id].len : -1;
      return TPA_OK;
    case TPA_Q_NUM_SMS: *value = ctx->num_sms; return TPA_OK;
    case TPA_Q_LAST_DENSE_ITEMS: *value = ctx->last_dense; return TPA_OK;
    case TPA_Q_LAST_SUFFIX_ITEMS: *value = ctx->last_suffix; return TPA_OK;
    case TPA_Q_LAST_LAUNCHES: *value = ctx->last_launches; return TPA_OK;
    default: return fail(TPA_ERR_INVALID_ARG, "unknown query %d", what);
  }
}

int tpa_set_option(tpa_ctx* ctx, int32_t option, int64_t value) {
  if (!ctx) return fail(TPA_ERR_INVALID_ARG, "null context");
  switch (option) {
    case TPA_OPT_DECODE_MODE:
      if (value != 0 && value != 1) return fail(TPA_ERR_INVALID_ARG, "decode mode %lld", (long long)value);
      ctx->decode_mode = static_cast<int>(value);
      return TPA_OK;
    case TPA_OPT_PREFIX_SPLITS:
      if (value < 0 || value > 1024) return fail(TPA_ERR_INVALID_ARG, "prefix splits %lld", (long long)value);
      ctx->prefix_splits = static_cast<int>(value);
      return TPA_OK;
    case TPA_OPT_SUFFIX_SPLIT_KEYS:
      if (value < 0 || value % kPage || value > (1 << 20))
        return fail(TPA_ERR_INVALID_ARG, "split keys must be a multiple of 16");
      ctx->suffix_split_keys = static_cast<int>(value);
      return TPA_OK;
    case TPA_OPT_KERNEL_TIMING:
      ctx->timing = value ? 1 : 0;
      return TPA_OK;
    case TPA_OPT_TEST_PLAN_WAIT:
      ctx->test_plan_wait = value ? 1 : 0;
      return TPA_OK;
    case TPA_OPT_TEST_BAD_PAGE:
      ctx->test_bad_page = value ? 1 : 0;
      return TPA_OK;
    case TPA_OPT_TEST_BAD_SLOT:
      ctx->test_bad_slot = value ? 1 : 0;
      return TPA_OK;
    case TPA_OPT_MOVEMENT_STAGED:
      ctx->staged_movement = value != 0;
      return TPA_OK;
    case TPA_OPT_PREFILL_TILE_ROWS:
      if (value != 128 && value != 256) return fail(TPA_ERR_INVALID_ARG, "prefill tile rows %lld", (long long)value);
      ctx->prefill_rows = static_cast<int>(value);
      return TPA_OK;
    default: return fail(TPA_ERR_INVALID_ARG, "unknown option %d", option);
  }
}

int tpa_kernel_times(tpa_ctx* ctx, int32_t n, double* total_ms, int64_t* launches, int32_t reset) {
  if (!ctx || n < 0 || (n > 0 && (!total_ms || !launches)))
    return fail(TPA_ERR_INVALID_ARG, "bad arguments");
  int rc = resolve_timing(ctx);
  if (rc) return rc;
  for (int k = 0; k < n; ++k) {
    total_ms[k] = k < kKernelKinds ? ctx->k_ms[k] : 0.0;
    launches[k] = k < kKernelKinds ? ctx->k_n[k] : 0;
  }
  if (reset)
    for (int k = 0; k < kKernelKinds; ++k) {
      ctx->k_ms[k] = 0.0;
      ctx->k_n[k] = 0;
    }
  return TPA_OK;
}

int tpa_device_status(tpa_ctx* ctx, void* stream, uint32_t* status) {
  if (!ctx || !status) return fail(TPA_ERR_INVALID_ARG, "null argument");
  *status = 0;
  if (ctx->plan_only) return TPA_OK;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  CUDA_TRY(cudaStreamSynchronize(s));
  CUDA_TRY(cudaMemcpy(status, ctx->status, sizeof(uint32_t), cudaMemcpyDeviceToHost));
  CUDA_TRY(cudaMemset(ctx->status, 0, sizeof(uint32_t)));
  if (*status & (kStatusDenseTimeout | kStatusSuffixTimeout | kStatusPlanTimeout))
    return fail(TPA_ERR_TIMEOUT, "a device-side wait timed out (status 0x%x)", *status);
  return TPA_OK;
}

}  // extern "C"

namespace tpa {
int set_error(int code, const char* msg) { return fail(code, "%s", msg); }

cudaError_t init_kernels() {
  static bool done = false;
  if (done) return cudaSuccess;
  cudaError_t e = init_dense_kernels();
  if (e != cudaSuccess) return e;
  e = init_suffix_kernels();
  if (e != cudaSuccess) return e;
  e = init_prefill_pair();
  if (e == cudaSuccess) done = true;
  return e;
}
}  // namespace tpa
