/*
 * topas_sched.h -- one TOPAS scheduling decision on the host (C ABI).
 *
 * The paper's scheduler (Sec. IV) picks, at every scheduling event, a
 * post-decision prefix-request state S' = (R', Q'): which agent prefixes
 * stay or become resident and which requests run under them, subject to
 * the joint KV budget of Eq. 2 (sum of the resident prefixes' lengths plus
 * the running requests' reservations <= B_t; a prefix is paid once for all
 * of its agent's requests; no idle prefix is resident).  This call scores
 * candidate states with Eq. 12
 *
 *   Score = J_admit^age - J_move - J_redo - J_revoke + V_reuse
 *
 *   J_admit  sum over admitted requests of g_i(t) (Eq. 11) times the
 *            conditional reduction of the task's expected longest remaining
 *            LLM-service path (Eqs. 3-6);
 *   J_move   mu / B_swap times the moved prefix tokens (in and out), times
 *            the distinct admitted tasks waiting for an incoming prefix (Eq. 7);
 *   J_redo   T_decode y_r over preempted requests (Eq. 8);
 *   J_revoke the preempted requests' stored credits lambda_r (Eq. 9);
 *   V_reuse  beta sum over resident agents of n_a(t) mu l_a / B_swap (Eq. 10),
 *
 * generates them with GreedyPack and the hierarchical prefix-set search
 * (Algorithm 1: every subset of the active agents when there are at most
 * M of them, else greedy single additions, one pair pass and drop/swap
 * repairs; caps K on admissions and on preemptions) and returns the
 * highest-scoring one (Eq. 13, first generated wins ties).
 *
 * The call is stateless: the caller passes the whole state as flat arrays
 * (host memory, caller-owned, only read during the call) and applies the
 * decision itself -- e.g. with tpa_prefix_evict / tpa_prefix_reload for the
 * prefix moves and tpa_request_* / tpa_prefill_chunk / tpa_decode for the
 * requests (topas_attn.h).  The arithmetic is IEEE double in a fixed
 * order, so the same snapshot always gives the same decision.
 *
 * Readings where the paper is silent:
 *  - the expectation of Eq. 4 is a mean over `mc_samples` joint draws of
 *    the stage residuals; draw k of stage v of task i takes residual sample
 *    splitmix64(splitmix64(splitmix64(seed ^ task_id) ^ v) ^ k) mod n
 *    (SplitMix64, S. Vigna), the same draws for every hypothetical set;
 *  - a started stage already served beyond every sample has residual 0;
 *  - LP of a realization: lp[v] = z_v + max(0, max over successors lp[s]),
 *    stages in topological order, LP = max over v;
 *  - D_r (a request's expected service, s) is an input;
 *  - GreedyPack admits the fitting request with the largest g_i Delta / d_r,
 *    ties to a request whose task already has an admission, then to the
 *    lowest index; an uncovered agent of R reserves its ready request with
 *    the smallest d_r;
 *  - n_a(t) counts unstarted stages of agent a whose only unfinished
 *    predecessor has started;
 *  - the bounded search starts from R_t restricted to the active agents;
 *  - the age t - tau_i is clamped at 0;
 *  - when no state is generated at all (the caps forbid every change and
 *    the incumbent's requests do not all fit), the incumbent is kept.
 */
#ifndef TOPAS_SCHED_H
#define TOPAS_SCHED_H

#include <stddef.h>
#include <stdint.h>

#include "topas_attn.h"

#ifdef __cplusplus
extern "C" {
#endif

typedef struct {
  double budget;      /* B_t: token-equivalent KV capacity */
  double mu;          /* KV bytes per prefix token */
  double b_swap;      /* swap bandwidth, bytes/s (> 0) */
  double t_decode;    /* profiled decode time per token, s */
  double beta;        /* V_reuse pressure (Eq. 10) */
  double rho;         /* aging strength (Eq. 11) */
  double h_age;       /* aging scale, s (> 0) */
  int32_t M;          /* enumerate all prefix sets when the active agents are <= M (M <= 20) */
  int32_t K;          /* cap on admissions and on preemptions; 0 = no cap */
  int32_t mc_samples; /* joint draws of the Eq. 4 expectation (>= 1) */
  int32_t pad;
  uint64_t seed;
} tpa_sched_params;

/* Stages are listed in topological order (every predecessor index is
 * smaller than its stage).  [i * n_stages + v] indexes task i, stage v. */
typedef struct {
  double t;                     /* scheduling time, s */
  int32_t n_stages, n_agents, n_tasks, n_reqs;   /* n_agents <= 64 */
  const int32_t* stage_agent;   /* [n_stages] agent executing each stage */
  const int32_t* pred_off;      /* [n_stages + 1] CSR offsets into pred_idx */
  const int32_t* pred_idx;      /* predecessors of each stage, ascending */
  const int64_t* prefix_len;    /* [n_agents] l_a, tokens */
  const int32_t* sample_off;    /* [n_stages + 1] CSR offsets into samples (>= 1 per stage) */
  const double* samples;        /* empirical total LLM service of each stage, s (F_{a,v}) */
  const uint64_t* task_id;      /* [n_tasks] stable ids (the draws key on them) */
  const double* task_arrival;   /* [n_tasks] tau_i */
  const int8_t* stage_state;    /* [n_tasks * n_stages] 0 unstarted, 1 started, 2 done */
  const double* stage_served;   /* [n_tasks * n_stages] e_{i,v}(t), s */
  const int32_t* req_task;      /* [n_reqs] task index */
  const int32_t* req_stage;     /* [n_reqs] stage index */
  const double* req_kv;         /* [n_reqs] d_r(t) > 0, tokens */
  const double* req_dhat;       /* [n_reqs] D_r(t) >= 0, s */
  const double* req_redo;       /* [n_reqs] y_r(t), tokens to rebuild if preempted */
  const double* req_credit;     /* [n_reqs] lambda_r of running requests */
  const uint8_t* req_running;   /* [n_reqs] 1: in Q_t; 0: ready (W_t) */
  const uint8_t* resident;      /* [n_agents] 1: in R_t */
} tpa_sched_snapshot;

typedef struct {
  /* caller-provided outputs */
  uint8_t* agents;      /* [n_agents] R' */
  uint8_t* running;     /* [n_reqs] Q' */
  int32_t* admitted;    /* [n_reqs] A, in admission order (first n_admitted entries) */
  double* credits;      /* [n_reqs] lambda of each admitted request, same order */
  /* filled by the call */
  int32_t n_admitted, n_preempted;
  double score, j_admit, j_move, j_redo, j_revoke, v_reuse;
  int64_t n_candidates; /* states generated (Algorithm 1's C_t) */
} tpa_sched_decision;

/* Select the next state.  Errors: INVALID_ARG (null pointer, size or index
 * out of range, a predecessor not before its stage, a stage without
 * samples, non-positive b_swap, h_age, d_r or mc_samples, M > 20).
 * A generated state satisfies the budget; with no nonempty feasible state
 * the result may be empty (Q' = {}); with none at all it is the incumbent. */
TPA_API int tpa_sched_decide(const tpa_sched_params* params, const tpa_sched_snapshot* snap,
                             tpa_sched_decision* out);

#ifdef __cplusplus
}
#endif
#endif /* TOPAS_SCHED_H */
