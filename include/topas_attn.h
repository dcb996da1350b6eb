/*
 * topas_attn.h -- C ABI of a GB300 (sm_103a) library for attention over a
 * paged KV pool in which many requests share one resident agent prefix.
 *
 * Setting (TOPAS, "Workflow-Aware Prefix-State Scheduling for Multi-Agent
 * LLM Serving"): every request r belongs to an agent a(r); all requests of
 * agent a share a static system-prompt prefix of ell_a tokens whose KV cache
 * is kept resident once per agent, and each request adds its own dynamic
 * suffix and decode tokens (Sec. I; Sec. III, joint prefix-request state
 * and Eq. 2, where the resident prefix is paid once per agent plus d_r(t)
 * per request under the budget B_t).  Prefixes enter and leave the GPU as
 * the resident set changes, moving between GPU and CPU memory (Sec. IV-B,
 * prefix-movement delay, Eq. 7).
 *
 * The library computes exact attention (scores q.k/sqrt(d), softmax, value
 * average, natural-log LSE) with bf16 inputs and fp32 accumulation.  Decode
 * is a two-level cascade: the queries of all requests of one agent are
 * stacked and read that agent's prefix KV once as a dense tcgen05 GEMM,
 * each request's suffix goes through a split-KV paged kernel, and the
 * partial results are merged exactly by log-sum-exp.
 *
 * Conventions
 *   - bf16 means IEEE bfloat16 stored as 2-byte values; all arrays are
 *     row-major and densely packed.
 *   - KV pool: k_pool and v_pool are caller-owned device arrays
 *     bf16 [num_pages][num_kv_heads][page_size][head_dim].  Page size is 16.
 *   - Grouped-query attention: q head h reads kv head h / (Hq / Hkv).
 *   - Streams and events are cudaStream_t / cudaEvent_t passed as void*.
 *     All device work is asynchronous on the given stream; no call
 *     synchronises the host with the device unless documented.
 *   - Ownership: all device memory (pools, workspace, inputs, outputs),
 *     streams and events belong to the caller and are never freed by the
 *     library.  The library owns its host-side tables and a small ring of
 *     pinned host staging buffers allocated in tpa_create.
 *   - Errors: every call returns a TPA_* status.  A call that fails leaves
 *     the tables as they were.  tpa_last_error() returns a thread-local
 *     message for the last failure on the calling thread.
 *   - Thread safety: one context must not be used from two host threads
 *     at the same time.
 */
#ifndef TOPAS_ATTN_H
#define TOPAS_ATTN_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define TPA_API __attribute__((visibility("default")))
#else
#define TPA_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

enum {
  TPA_OK = 0,
  TPA_ERR_INVALID_ARG = 1,   /* bad pointer, id, length, duplicate id in a batch, unpinned host memory */
  TPA_ERR_NO_SPACE = 2,      /* free pages cannot hold the request (the budget of Eq. 2) */
  TPA_ERR_NOT_RESIDENT = 3,  /* the agent's prefix is not resident on the GPU */
  TPA_ERR_STATE = 4,         /* lifecycle misuse: registered twice, request not open, ... */
  TPA_ERR_UNSUPPORTED = 5,   /* shape outside head_dim {64,128}, group {4,8}, page 16 */
  TPA_ERR_CUDA = 6,          /* a CUDA runtime call failed (message in tpa_last_error) */
  TPA_ERR_TIMEOUT = 7,       /* a device-side wait gave up; see tpa_device_status */
  TPA_ERR_CAPACITY = 8       /* the call exceeds capacities fixed at tpa_create */
};

/* tpa_config.flags */
#define TPA_FLAG_PLAN_ONLY 1 /* host tables and planning only: no CUDA call, no device work */

typedef struct tpa_ctx tpa_ctx;

typedef struct tpa_config {
  int32_t num_q_heads;       /* Hq */
  int32_t num_kv_heads;      /* Hkv; Hq / Hkv must be 4 or 8 */
  int32_t head_dim;          /* d: 64 or 128 */
  int32_t page_size;         /* must be 16 */
  int64_t num_pages;         /* pages in each of k_pool, v_pool */
  void* k_pool;              /* device bf16 [num_pages][Hkv][16][d], 16-byte aligned */
  void* v_pool;              /* device bf16 [num_pages][Hkv][16][d], 16-byte aligned */
  void* workspace;           /* device, >= tpa_workspace_size(cfg) bytes, 256-byte aligned */
  size_t workspace_bytes;
  int32_t max_agents;        /* agent ids are 0 .. max_agents-1 */
  int32_t max_requests;      /* request ids are 0 .. max_requests-1 */
  int32_t max_tokens;        /* most query/KV token rows in one append, prefill or decode call */
  int32_t max_seq_len;       /* longest prefix and longest suffix, in tokens */
  int32_t max_splits;        /* most partial results per (token, head) in decode; 0 -> 32.
                                The partial-result workspace holds
                                min(max_tokens, max_requests) * Hq * max_splits slots */
  int32_t flags;             /* TPA_FLAG_* */
  uint64_t page_order_seed;  /* 0: free pages handed out in id order; else a seeded permutation
                                (a fragmented pool, as after many evictions and reloads) */
} tpa_config;

/* Bytes of device workspace the context needs (plan ring, partial results,
 * status word, and the prefix-movement staging area: K and V of a
 * max_seq_len-token prefix).  Returns 0 for an invalid or unsupported
 * configuration. */
TPA_API size_t tpa_workspace_size(const tpa_config* cfg);

/* Create a context over the caller's pools and workspace.  Builds the free
 * page list, the TMA descriptors of the pools and the pinned staging ring.
 * Errors: INVALID_ARG, UNSUPPORTED, CUDA. */
TPA_API int tpa_create(const tpa_config* cfg, tpa_ctx** out);

/* Synchronises with the context's outstanding work, then frees the host
 * side.  The caller's device memory is untouched. */
TPA_API int tpa_destroy(tpa_ctx* ctx);

/* ---- agent prefixes: the resident set R_t (Sec. III) ---------------- */

/* Register agent `agent` with a prefix of `len` >= 0 tokens (ell_a) and make
 * it resident: ceil(len/16) pages are taken from the free list.  The page
 * contents are undefined until tpa_prefix_write or tpa_prefix_reload.
 * Errors: INVALID_ARG (id/len), STATE (already registered), NO_SPACE. */
TPA_API int tpa_prefix_register(tpa_ctx* ctx, int32_t agent, int32_t len);

/* Write a resident prefix's K/V from contiguous bf16 [len][Hkv][d] arrays
 * `k`, `v` (device memory, or pinned host memory) into its pages on
 * `stream`.  The source must stay valid until the stream passes the call.
 * Errors: INVALID_ARG, STATE (not registered), NOT_RESIDENT, CUDA. */
TPA_API int tpa_prefix_write(tpa_ctx* ctx, int32_t agent, const void* k, const void* v, void* stream);

/* Drop a prefix from the resident set: its pages return to the free list
 * (after the work already queued that reads them).  Open requests of the
 * agent stay open but cannot attend until the prefix is reloaded.
 * Errors: STATE (not registered), NOT_RESIDENT (already evicted). */
TPA_API int tpa_prefix_evict(tpa_ctx* ctx, int32_t agent);

/* Prefix movement CPU -> GPU (Sec. IV-B, Eq. 7): take ceil(len/16) free
 * pages (in free-list order, so possibly scattered) and copy the pinned
 * host arrays bf16 [len][Hkv][d] `host_k`, `host_v` into them on
 * `side_stream`: the copy engine moves them into the workspace's staging
 * area, then a short kernel scatters them into the pages, so the transfer
 * over the host link holds no SM.  Movement calls share the staging area
 * and are ordered on the device.  If `done_event` is not NULL it is
 * recorded after the copy.  Later calls that read this prefix, on any
 * stream, wait for the copy on the device; a prefill call runs the chunks
 * of other agents first.  Host memory must be pinned (cudaHostAlloc /
 * cudaHostRegister) and stay valid until the copy completes.
 * Errors: INVALID_ARG (not pinned), STATE, NO_SPACE, CUDA. */
TPA_API int tpa_prefix_reload(tpa_ctx* ctx, int32_t agent, const void* host_k, const void* host_v,
                      void* side_stream, void* done_event);

/* Prefix movement GPU -> CPU: copy a resident prefix into pinned host
 * arrays bf16 [len][Hkv][d] on `side_stream` (a gather kernel into the
 * staging area, then a copy-engine copy to the host), record `done_event`
 * (if not NULL), then evict it as tpa_prefix_evict does.  Errors as reload. */
TPA_API int tpa_prefix_offload(tpa_ctx* ctx, int32_t agent, void* host_k, void* host_v,
                       void* side_stream, void* done_event);

/* ---- requests: the running set Q_t (Sec. III) ----------------------- */

/* Open request `req` of agent `agent` with an empty suffix.
 * Errors: INVALID_ARG, STATE (already open, agent not registered). */
TPA_API int tpa_request_open(tpa_ctx* ctx, int32_t req, int32_t agent);

/* Close a request; its suffix pages return to the free list (after the
 * work already queued that reads them).  Errors: INVALID_ARG, STATE. */
TPA_API int tpa_request_close(tpa_ctx* ctx, int32_t req);

/* Discard the tails of the suffixes of `n` distinct open requests so that
 * lens[i] tokens remain in request reqs[i] (0 <= lens[i] <= its length;
 * host arrays).  Pages past ceil(lens[i]/16) return to the free list after
 * the work already queued that reads them.  This is the table step of
 * dropping decode KV, as when a preempted request's generated tokens are
 * discarded (Sec. IV-B, discarded decode work, Eq. 8) or a speculative tail
 * is rejected.  No device work.  All or nothing.  Errors: INVALID_ARG, STATE. */
TPA_API int tpa_request_truncate(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* lens);

/* Append KV tokens to the suffixes of `n` distinct open requests.
 * reqs[i], ntok[i] (host arrays): request ids and token counts (>= 0).
 * k_new, v_new: device bf16 [sum ntok][Hkv][d], request i's tokens
 * contiguous and in call order.  Suffixes always start on a fresh page, so
 * shared prefix pages are never written.  Errors: INVALID_ARG, STATE,
 * NO_SPACE, CAPACITY, CUDA. */
TPA_API int tpa_kv_append(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* ntok,
                  const void* k_new, const void* v_new, void* stream);

/* Chunked causal suffix prefill (chunked prefill, Sec. VI).  For each of
 * `n` distinct open requests with a resident prefix, append the chunk's
 * K/V and compute attention of its queries: the row of suffix position p
 * sees all ell_a prefix keys and suffix positions 0..p (diagonal
 * included).
 *   chunk_len[i] (host): tokens in request i's chunk (>= 1)
 *   q      bf16 [sum chunk_len][Hq][d]
 *   k_new  bf16 [sum chunk_len][Hkv][d]   (v_new likewise)
 *   out    bf16 [sum chunk_len][Hq][d]
 *   lse    fp32 [sum chunk_len][Hq]  natural-log LSE of the scaled scores
 * Device memory, or pinned host memory as for tpa_decode (the kernels then
 * move those bytes over the CPU-GPU link; the results are bit-identical).
 * Errors: INVALID_ARG, STATE, NOT_RESIDENT, NO_SPACE, CAPACITY, CUDA. */
TPA_API int tpa_prefill_chunk(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const int32_t* chunk_len,
                      const void* q, const void* k_new, const void* v_new,
                      void* out, float* lse, void* stream);

/* One decode step for `n` distinct open requests with resident prefixes:
 * append each request's new token K/V, then attend each query to its
 * prefix, its suffix and the new token.
 *   q      bf16 [n][Hq][d];   k_new, v_new bf16 [n][Hkv][d]
 *   out    bf16 [n][Hq][d];   lse fp32 [n][Hq]
 * These five arrays are device memory, or pinned host memory from
 * cudaHostAlloc (mapped: its host address is its device address).  With
 * host memory the kernels read the step's inputs and write its outputs
 * over the CPU-GPU link themselves, with no staging copy; the results are
 * bit-identical to the device-memory call.  The caller keeps host arrays
 * valid and unread until the stream passes the call.
 * Errors: INVALID_ARG, STATE, NOT_RESIDENT, NO_SPACE, CAPACITY, CUDA. */
TPA_API int tpa_decode(tpa_ctx* ctx, int32_t n, const int32_t* reqs, const void* q,
               const void* k_new, const void* v_new, void* out, float* lse, void* stream);

/* tpa_decode with its split partial results in a fixed device array
 * instead of the context's workspace.  The paper has no counterpart: this
 * is an allocation-free variant of the decode step for callers that want
 * its scratch to come from static device memory.
 *   Arguments, layouts and results are those of tpa_decode, and the outputs
 *   are bit-identical to it.  The scratch is a 256-byte aligned file-scope
 *   __device__ array of 16 MiB per device inside this library: fp32 partial
 *   outputs [slots][d] followed by their fp32 LSEs, so it holds
 *   slots = (16 MiB - 256) / (4 (d + 1)) partials (32510 at d = 128).  Its
 *   address is looked up once per device (with that device current) and
 *   cached; the call allocates no device or pinned memory.  Under lazy
 *   module loading (CUDA's default) only a context that runs this entry
 *   point loads the array; with CUDA_MODULE_LOADING=EAGER every context that
 *   loads the library holds it.  The cached address is the primary
 *   context's: after cudaDeviceReset do not call this entry point again.
 *   Nothing in the array has to start at zero: every partial a call reads
 *   is written earlier in the same call.
 *   All calls of this entry point on one device share the array: calls
 *   whose kernels overlap in time (other streams, other contexts, other
 *   threads) race on it and their outputs are undefined.  Order them on
 *   one stream, or use tpa_decode.
 * Errors: those of tpa_decode; CAPACITY (message names the limit) when the
 * step needs more partial slots than the array holds; CUDA when the array's
 * address cannot be looked up. */
TPA_API int tpa_decode_static_scratch(tpa_ctx* ctx, int32_t n, const int32_t* reqs,
                                      const void* q, const void* k_new, const void* v_new,
                                      void* out, float* lse, void* stream);

/* Copy a prefix (is_request = 0) or a request suffix (is_request = 1) out of
 * its pages into contiguous bf16 [len][Hkv][d] arrays `k_out`, `v_out`
 * (device or pinned host memory).  Errors: INVALID_ARG, STATE, NOT_RESIDENT. */
TPA_API int tpa_gather(tpa_ctx* ctx, int32_t id, int32_t is_request, void* k_out, void* v_out,
               void* stream);

/* ---- introspection and options -------------------------------------- */

enum {
  TPA_Q_FREE_PAGES = 0,     /* id ignored */
  TPA_Q_PREFIX_LEN = 1,     /* agent id: ell_a, or -1 if not registered */
  TPA_Q_PREFIX_RESIDENT = 2,/* agent id: 1 resident, 0 evicted, -1 not registered */
  TPA_Q_SUFFIX_LEN = 3,     /* request id: suffix tokens, or -1 if not open */
  TPA_Q_NUM_SMS = 4,        /* SMs used for grid sizing */
  TPA_Q_LAST_DENSE_ITEMS = 5,   /* work items of the last call's dense (tensor-core) kernel */
  TPA_Q_LAST_SUFFIX_ITEMS = 6,  /* work items of the last call's split-KV suffix kernel */
  TPA_Q_LAST_LAUNCHES = 7,      /* kernels the last call launched */
  TPA_Q_PAGE_OF = 8             /* first page id of agent `id` (for layout tests) */
};
TPA_API int tpa_query(tpa_ctx* ctx, int32_t what, int32_t id, int64_t* value);

enum {
  TPA_OPT_DECODE_MODE = 0,      /* 0: cascade (default): one persistent launch over stacked
                                   prefix tiles (tensor cores) and per-request suffixes
                                   (split-KV, with the KV append), then the LSE merge launched as
                                   its programmatic dependent; 1: flat cross-check -- KV append,
                                   every key (prefix included) through the split-KV kernel, then
                                   the merge */
  TPA_OPT_PREFIX_SPLITS = 1,    /* cascade: key splits per stacked prefix tile; 0 = automatic */
  TPA_OPT_SUFFIX_SPLIT_KEYS = 2,/* keys per suffix work item, a multiple of 16; 0 = automatic */
  TPA_OPT_KERNEL_TIMING = 4,    /* 1: bracket every kernel with CUDA events (tpa_kernel_times) */
  TPA_OPT_TEST_PLAN_WAIT = 5,   /* test hook, 1: the next cascade decode's kernel waits for a
                                   plan flag that is never written, so every CTA gives up at the
                                   device wait limit (2 s) without touching the pool and
                                   tpa_device_status reports TIMEOUT.  The context stays usable;
                                   truncate that call's requests back to their lengths before it */
  TPA_OPT_TEST_BAD_PAGE = 7,    /* test hook, 1: the next decode's plan lists its first resident
                                   prefix's first page as the pool size (one past the last page).
                                   Every kernel bounds-checks page ids: those reads go to page 0 and
                                   the device status gets bit 4; that step's outputs for the agent's
                                   tokens are wrong, and later steps are unaffected */
  TPA_OPT_PREFILL_TILE_ROWS = 6,/* query rows per prefill work item: 256 (default) pairs two
                                   128-row tiles of 256/G consecutive tokens that share every K/V
                                   tile (one CTA, two softmax warpgroups, the tensor pipe
                                   alternating between them); 128 runs single tiles through the
                                   dense kernel of the decode's level 1 */
  TPA_OPT_MOVEMENT_STAGED = 8,  /* prefix reload / offload: 1 (default) moves the prefix over the
                                   host link with the copy engine, through the workspace's
                                   staging area, and scatters / gathers the pages on the device;
                                   0 runs the page kernel on the mapped host arrays directly (it
                                   holds its SMs for the whole link-bound transfer) */
  TPA_OPT_TEST_BAD_SLOT = 9     /* test hook, 1: the next decode's plan gives its first token
                                   partial slots past the end of the partial buffer.  Every
                                   kernel checks partial slots: that token's partials are neither
                                   written nor read, its outputs are left unwritten and the
                                   device status gets bit 16; later steps are unaffected */
};
TPA_API int tpa_set_option(tpa_ctx* ctx, int32_t option, int64_t value);

/* Per-kernel device time, for profiling.  While TPA_OPT_KERNEL_TIMING is 1
 * every kernel launch of the library is bracketed by CUDA events on the
 * stream it runs on.  This call synchronises with those events and returns,
 * for each kernel kind k < n (0 KV append, 1 dense tensor-core attention,
 * 2 split-KV attention, 3 LSE merge, 4 page-run copy, 5 paired-tile
 * tensor-core prefill), the accumulated time
 * in milliseconds and the number of launches since the last reset
 * (`reset` != 0 clears the totals after reading).  Errors: INVALID_ARG, CUDA. */
TPA_API int tpa_kernel_times(tpa_ctx* ctx, int32_t n, double* total_ms, int64_t* launches,
                             int32_t reset);

/* Synchronise `stream`, then read and clear the device status word.
 * *status = 0 when no kernel reported a problem; otherwise a bit set:
 * 1 a dense-kernel wait timed out, 2 a suffix-kernel wait timed out,
 * 4 a page id outside the pool was met (the access was redirected to page
 * 0), 8 a kernel gave up waiting for its plan upload (it did no work),
 * 16 a partial slot outside the partial buffer was met (not written or read).
 * Returns TIMEOUT if bit 1, 2 or 8 is set, CUDA on a CUDA error. */
TPA_API int tpa_device_status(tpa_ctx* ctx, void* stream, uint32_t* status);

/* Thread-local message describing the last failed call on this thread. */
TPA_API const char* tpa_last_error(void);

#ifdef __cplusplus
}
#endif
#endif /* TOPAS_ATTN_H */
