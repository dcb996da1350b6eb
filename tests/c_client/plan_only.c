/* A plain C99 client of libtopas_attn.so, built and run by
 * tests/test_c_client.py with no GPU: it includes only the public header and
 * drives a plan-only context (TPA_FLAG_PLAN_ONLY: host tables and planning,
 * no CUDA call).  It prints one line per check and "ok" at the end; any
 * failed check prints its line and exits 1. */
#include <stdio.h>
#include <string.h>

#include "topas_attn.h"

static int failures = 0;

static void check(int cond, const char* what) {
  printf("%s %s\n", cond ? "pass" : "FAIL", what);
  if (!cond) ++failures;
}

static int64_t query(tpa_ctx* ctx, int32_t what, int32_t id) {
  int64_t v = -999;
  if (tpa_query(ctx, what, id, &v) != TPA_OK) return -999;
  return v;
}

int main(void) {
  tpa_config cfg;
  memset(&cfg, 0, sizeof cfg);
  cfg.num_q_heads = 32;
  cfg.num_kv_heads = 8;
  cfg.head_dim = 128;
  cfg.page_size = 16;
  cfg.num_pages = 12;
  cfg.max_agents = 2;
  cfg.max_requests = 4;
  cfg.max_tokens = 64;
  cfg.max_seq_len = 256;
  cfg.flags = TPA_FLAG_PLAN_ONLY;

  check(tpa_workspace_size(&cfg) > 0, "workspace size of a supported shape");
  tpa_config bad = cfg;
  bad.head_dim = 96;
  check(tpa_workspace_size(&bad) == 0, "workspace size 0 for head_dim 96");

  tpa_ctx* ctx = NULL;
  check(tpa_create(&cfg, &ctx) == TPA_OK && ctx != NULL, "create a plan-only context");
  if (!ctx) return 1;
  check(query(ctx, TPA_Q_FREE_PAGES, 0) == 12, "12 free pages");

  /* the budget of Eq. 2: a 33-token prefix takes ceil(33/16) = 3 pages */
  check(tpa_prefix_register(ctx, 0, 33) == TPA_OK, "register a 33-token prefix");
  check(query(ctx, TPA_Q_FREE_PAGES, 0) == 9, "3 pages taken");
  check(tpa_prefix_register(ctx, 1, 257) == TPA_ERR_INVALID_ARG,
        "a prefix longer than max_seq_len is refused");
  check(tpa_prefix_register(ctx, 1, 160) == TPA_ERR_NO_SPACE, "10 pages do not fit in 9");
  check(strlen(tpa_last_error()) > 0, "the failure is described");
  check(query(ctx, TPA_Q_FREE_PAGES, 0) == 9 && query(ctx, TPA_Q_PREFIX_LEN, 1) == -1,
        "a failed call changes nothing");
  check(tpa_prefix_register(ctx, 1, 0) == TPA_OK, "an empty prefix takes no page");

  /* requests, an append and a decode step (plan only: pointers untouched) */
  check(tpa_request_open(ctx, 0, 0) == TPA_OK, "open request 0");
  check(tpa_request_open(ctx, 1, 0) == TPA_OK, "open request 1");
  check(tpa_request_open(ctx, 1, 0) == TPA_ERR_STATE, "open twice is a state error");
  int32_t reqs[2] = {0, 1};
  int32_t ntok[2] = {17, 40};
  int dummy = 0;
  check(tpa_kv_append(ctx, 2, reqs, ntok, &dummy, &dummy, NULL) == TPA_OK, "append 17 + 40 tokens");
  check(query(ctx, TPA_Q_SUFFIX_LEN, 0) == 17 && query(ctx, TPA_Q_SUFFIX_LEN, 1) == 40,
        "suffix lengths after the append");
  check(tpa_decode(ctx, 2, reqs, NULL, NULL, NULL, NULL, NULL, NULL) == TPA_OK, "plan a decode step");
  check(query(ctx, TPA_Q_SUFFIX_LEN, 0) == 18 && query(ctx, TPA_Q_SUFFIX_LEN, 1) == 41,
        "the decode appended one token each");
  check(query(ctx, TPA_Q_LAST_DENSE_ITEMS, 0) > 0, "the shared prefix went to the dense level");
  check(query(ctx, TPA_Q_LAST_SUFFIX_ITEMS, 0) >= 2 * 8, "every (token, kv head) has a suffix item");
  int32_t dup[2] = {1, 1};
  check(tpa_decode(ctx, 2, dup, NULL, NULL, NULL, NULL, NULL, NULL) == TPA_ERR_INVALID_ARG,
        "a request twice in one batch is refused");

  /* eviction makes the agent's requests unable to attend */
  check(tpa_prefix_evict(ctx, 0) == TPA_OK, "evict the prefix");
  check(tpa_decode(ctx, 2, reqs, NULL, NULL, NULL, NULL, NULL, NULL) == TPA_ERR_NOT_RESIDENT,
        "decode without the prefix is refused");
  check(tpa_prefix_reload(ctx, 0, &dummy, &dummy, NULL, NULL) == TPA_OK, "reload it");
  check(query(ctx, TPA_Q_PREFIX_RESIDENT, 0) == 1, "resident again");

  int32_t lens[2] = {5, 0};
  check(tpa_request_truncate(ctx, 2, reqs, lens) == TPA_OK, "truncate (preemption)");
  check(query(ctx, TPA_Q_SUFFIX_LEN, 0) == 5 && query(ctx, TPA_Q_SUFFIX_LEN, 1) == 0,
        "truncated lengths");
  check(tpa_request_close(ctx, 0) == TPA_OK && tpa_request_close(ctx, 1) == TPA_OK, "close both");
  check(query(ctx, TPA_Q_FREE_PAGES, 0) == 9, "only the prefix's pages remain taken");
  check(tpa_destroy(ctx) == TPA_OK, "destroy");

  if (failures) return 1;
  printf("ok\n");
  return 0;
}
