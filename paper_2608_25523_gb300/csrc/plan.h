// Work-list records built by the host planner and read by the kernels.
// One call's plan is a single blob uploaded with one host-to-device copy.
#pragma once
#include <stdint.h>

namespace tpa {

constexpr int kPage = 16;          // tokens per page
constexpr int kTileRows = 128;     // query rows of a dense (tensor-core) tile
constexpr int kTileKeys = 128;     // keys per dense tile (8 pages)

// Status bits of the device status word.
constexpr uint32_t kStatusDenseTimeout = 1u;
constexpr uint32_t kStatusSuffixTimeout = 2u;
constexpr uint32_t kStatusBadPage = 4u;
constexpr uint32_t kStatusPlanTimeout = 8u;  // a plan upload never arrived
constexpr uint32_t kStatusBadSlot = 16u;     // a partial slot outside the partial buffer (skipped)

// A run of a KV write within one page: source rows src .. src + n - 1 of
// the K/V arrays go to slots slot .. slot + n - 1 of page `page` (n <= 16).
struct AppendRow {
  int32_t src;
  int32_t page;
  int32_t slot;
  int32_t n;
};

// Per-token data of a dense tile.
struct DenseTok {
  int32_t q_row;       // row of q / out / lse ([rows][Hq][d])
  int32_t causal_pos;  // causal segment: key index k visible iff k <= causal_pos
  int32_t slot_base;   // partial slot of (token, head 0, split 0)
  int32_t n_slots;     // splits per (token, head); slot = slot_base + head * n_slots + split
};

// One 128-row query tile (128/G tokens x G heads of one kv head) against up
// to two key segments, each a run of pages of one prefix or one suffix.
struct DenseItem {
  int32_t tok_base;       // first DenseTok of the tile (< 0: consecutive tokens, below)
  int32_t n_tok;          // tokens in the tile (<= 128 / G)
  int32_t kv_head;
  int32_t split;          // split index for partial slots (out_mode 0)
  int32_t out_mode;       // 0: fp32 partial (o, lse); 1: bf16 out + fp32 lse
  int32_t n_tiles;        // total key tiles over both segments
  int32_t seg_pages[2];   // offset in the page list of the segment's page 0
  int32_t seg_k0[2];      // first key of the range (multiple of 16)
  int32_t seg_k1[2];      // one past the last key of the range (k1 == k0: empty)
  int32_t seg_causal[2];  // 1: causal mask on this segment
  // tok_base < 0 (paired prefill items): the tile's tokens are consecutive
  // rows of one chunk, token i at q row row0 + i and causal position pos0 + i,
  // with no DenseTok records
  int32_t row0;
  int32_t pos0;
};
static_assert(sizeof(DenseItem) == 64, "DenseItem layout");

// One warp of the split-KV kernel: the G query rows of one token against a
// key range of one page run (a request suffix, or a prefix in flat mode).
struct SuffixItem {
  int32_t q_row;
  int32_t kv_head;
  int32_t pages;      // offset in the page list of the range's first page
  int32_t n_keys;     // keys in the range (>= 1), starting at that page's slot 0
  int32_t slot_base;  // partial slot of (token, head 0, split 0)
  int32_t n_slots;
  int32_t split;
  int32_t app_src;    // decode: row of k_new/v_new appended before the range is read (-1: none)
  int32_t app_dst;    // page * 16 + slot the appended row goes to
  int32_t pad[3];
};
static_assert(sizeof(SuffixItem) == 48, "SuffixItem layout");

// Per-token record of the cascade decode's split-KV level: the suffix of
// one token's request, cut into key ranges of `split_keys` keys; the work
// items (token, range, kv head) are derived from these on the device.
struct SplitTok {
  int32_t q_row;      // token row (q / out / lse) and row of k_new / v_new
  int32_t pages;      // page-list offset of the request's suffix page 0
  int32_t keys;       // suffix keys, the step's token included
  int32_t slot_base;  // partial slot of (token, head 0, split 0)
  int32_t n_slots;    // partials per (token, head): prefix splits + suffix ranges
  int32_t split0;     // split index of the first suffix range (= prefix splits)
  int32_t app_dst;    // page * 16 + slot of the step's token
  int32_t pad;
};

// LSE merge of all partials of one token (every q head).
struct MergeTok {
  int32_t q_row;
  int32_t slot_base;
  int32_t n_slots;
  int32_t pad;
};

// Header of an uploaded plan blob; offsets in bytes from the blob start.
struct PlanHeader {
  int32_t n_pages, n_append, n_dense_tok, n_dense, n_suffix, n_merge;
  int32_t off_pages, off_append, off_dense_tok, off_dense, off_suffix, off_merge;
  uint32_t queue[4];  // zero on upload: atomic work counters of persistent kernels
};

}  // namespace tpa
