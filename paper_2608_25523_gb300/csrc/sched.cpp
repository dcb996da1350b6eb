// One TOPAS scheduling decision on the host (topas_sched.h): the
// transition score of Eq. 12 over candidate prefix-request states generated
// by GreedyPack and the hierarchical prefix-set search of Algorithm 1
// (Sec. IV of the paper).  Stateless: everything comes from the snapshot.
//
// All arithmetic is IEEE double in a fixed order, and this file is compiled
// without floating-point contraction, so a snapshot always gives the same
// decision on any host.
#include <cmath>
#include <cstdint>
#include <cstdio>
#include <limits>
#include <vector>

#include "../../include/topas_sched.h"

namespace tpa {
int set_error(int code, const char* msg);
}  // namespace tpa

namespace {

using Mask = uint64_t;  // a set of agents (bit a = agent a)
constexpr double kNegInf = -std::numeric_limits<double>::infinity();

// SplitMix64 (S. Vigna): one output of the generator for a 64-bit state.
inline uint64_t splitmix64(uint64_t x) {
  uint64_t z = x + 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

struct Cand {
  Mask agents;
  std::vector<int> keep;      // retained running requests, ascending
  std::vector<int> admitted;  // greedy order
  std::vector<double> gains;  // g_i * Delta of each admission
  double score, j_admit, j_move, j_redo, j_revoke, v_reuse;
  bool nonempty;
};

class Decider {
 public:
  Decider(const tpa_sched_params& p, const tpa_sched_snapshot& s) : p_(p), s_(s) {
    const int n = s.n_stages;
    succ_.assign(n, {});
    for (int v = 0; v < n; ++v)
      for (int k = s.pred_off[v]; k < s.pred_off[v + 1]; ++k) succ_[s.pred_idx[k]].push_back(v);
    // residual supports (Eq. 3), one list per (task, stage)
    vals_.resize(static_cast<size_t>(s.n_tasks) * n);
    for (int i = 0; i < s.n_tasks; ++i)
      for (int v = 0; v < n; ++v) {
        std::vector<double>& out = vals_[static_cast<size_t>(i) * n + v];
        const int st = s.stage_state[static_cast<size_t>(i) * n + v];
        if (st == 2) {
          out.push_back(0.0);
        } else if (st == 0) {
          for (int k = s.sample_off[v]; k < s.sample_off[v + 1]; ++k) out.push_back(s.samples[k]);
        } else {
          const double e = s.stage_served[static_cast<size_t>(i) * n + v];
          for (int k = s.sample_off[v]; k < s.sample_off[v + 1]; ++k)
            if (s.samples[k] > e) out.push_back(s.samples[k] - e);
          if (out.empty()) out.push_back(0.0);
        }
      }
    // the draws: per (task, stage, k) the chosen residual value
    draw_.resize(static_cast<size_t>(s.n_tasks) * n * p.mc_samples);
    for (int i = 0; i < s.n_tasks; ++i)
      for (int v = 0; v < n; ++v) {
        const std::vector<double>& vv = vals_[static_cast<size_t>(i) * n + v];
        const uint64_t h0 = splitmix64(p.seed ^ s.task_id[i]);
        const uint64_t h1 = splitmix64(h0 ^ static_cast<uint64_t>(v));
        for (int k = 0; k < p.mc_samples; ++k) {
          const uint64_t h = splitmix64(h1 ^ static_cast<uint64_t>(k));
          draw_[(static_cast<size_t>(i) * n + v) * p.mc_samples + k] = vv[h % vv.size()];
        }
      }
    // n_a(t): unstarted stages whose only unfinished predecessor has started
    n_a_.assign(s.n_agents, 0);
    for (int i = 0; i < s.n_tasks; ++i)
      for (int v = 0; v < n; ++v) {
        if (state(i, v) != 0) continue;
        int unfinished = 0, last = -1;
        for (int k = s.pred_off[v]; k < s.pred_off[v + 1]; ++k)
          if (state(i, s.pred_idx[k]) != 2) {
            ++unfinished;
            last = s.pred_idx[k];
          }
        if (unfinished == 1 && state(i, last) == 1) ++n_a_[s.stage_agent[v]];
      }
    for (int r = 0; r < s.n_reqs; ++r) {
      if (s.req_running[r]) running_.push_back(r);
      active_ |= Mask(1) << agent_of(r);
    }
    for (int a = 0; a < s.n_agents; ++a)
      if (s.resident[a]) r_now_ |= Mask(1) << a;
    age_.resize(s.n_tasks);
    for (int i = 0; i < s.n_tasks; ++i) {
      const double age = s.t - s.task_arrival[i];
      age_[i] = 1.0 + p.rho * std::log(1.0 + (age > 0.0 ? age : 0.0) / p.h_age);
    }
    z_.resize(n);
    lp_.resize(n);
  }

  void run(tpa_sched_decision* out);

 private:
  int state(int i, int v) const { return s_.stage_state[static_cast<size_t>(i) * s_.n_stages + v]; }
  int agent_of(int r) const { return s_.stage_agent[s_.req_stage[r]]; }

  // Eq. 4 for task i with the hypothetical service `done` removed per stage
  double remaining_path(int i, const std::vector<double>& done) {
    const int n = s_.n_stages;
    double total = 0.0;
    for (int k = 0; k < p_.mc_samples; ++k) {
      for (int v = 0; v < n; ++v) {
        const double x = draw_[(static_cast<size_t>(i) * n + v) * p_.mc_samples + k];
        const double d = done[v];
        z_[v] = x - d > 0.0 ? x - d : 0.0;
      }
      double best = 0.0;
      for (int v = n - 1; v >= 0; --v) {
        double m = 0.0;
        for (int w : succ_[v])
          if (lp_[w] > m) m = lp_[w];
        lp_[v] = z_[v] + m;
        if (lp_[v] > best) best = lp_[v];
      }
      total += best;
    }
    return total / p_.mc_samples;
  }

  // Eq. 5: progress of r given the earlier admissions of its task
  double progress(int r, const std::vector<int>& admitted) {
    const int i = s_.req_task[r];
    std::vector<double> done(s_.n_stages, 0.0);
    for (int q : admitted)
      if (s_.req_task[q] == i) done[s_.req_stage[q]] = done[s_.req_stage[q]] + s_.req_dhat[q];
    const double before = remaining_path(i, done);
    done[s_.req_stage[r]] = done[s_.req_stage[r]] + s_.req_dhat[r];
    return before - remaining_path(i, done);
  }

  void score(Cand& c);
  void greedy_pack(Mask agents, std::vector<Cand>& out);
  double add(Mask agents);

  const tpa_sched_params& p_;
  const tpa_sched_snapshot& s_;
  std::vector<std::vector<int>> succ_;
  std::vector<std::vector<double>> vals_;
  std::vector<double> draw_;
  std::vector<int> n_a_;
  std::vector<int> running_;
  std::vector<double> age_;
  std::vector<double> z_, lp_;
  Mask active_ = 0, r_now_ = 0;
  std::vector<Cand> cands_;
};

// Eq. 12 of the state (c.agents, c.keep + c.admitted)
void Decider::score(Cand& c) {
  double j_admit = 0.0;
  for (double g : c.gains) j_admit += g;
  const Mask r_in = c.agents & ~r_now_, r_out = r_now_ & ~c.agents;
  double moved = 0.0;
  for (int a = 0; a < s_.n_agents; ++a)
    if (r_out >> a & 1) moved += static_cast<double>(s_.prefix_len[a]);
  for (int a = 0; a < s_.n_agents; ++a)
    if (r_in >> a & 1) moved += static_cast<double>(s_.prefix_len[a]);
  const double t_move = p_.mu / p_.b_swap * moved;
  std::vector<int> tasks_in;
  for (int r : c.admitted)
    if (r_in >> agent_of(r) & 1) {
      bool seen = false;
      for (int x : tasks_in) seen = seen || x == s_.req_task[r];
      if (!seen) tasks_in.push_back(s_.req_task[r]);
    }
  const double j_move = t_move * static_cast<double>(tasks_in.size());
  double j_redo = 0.0, j_revoke = 0.0;
  size_t kk = 0;
  for (int r : running_) {  // preempted: running and not kept (both ascending)
    if (kk < c.keep.size() && c.keep[kk] == r) {
      ++kk;
      continue;
    }
    j_redo += p_.t_decode * s_.req_redo[r];
    j_revoke += s_.req_credit[r];
  }
  double v_reuse = 0.0;
  for (int a = 0; a < s_.n_agents; ++a)
    if (c.agents >> a & 1)
      v_reuse += p_.beta * static_cast<double>(n_a_[a]) * p_.mu * static_cast<double>(s_.prefix_len[a]) /
                 p_.b_swap;
  c.j_admit = j_admit;
  c.j_move = j_move;
  c.j_redo = j_redo;
  c.j_revoke = j_revoke;
  c.v_reuse = v_reuse;
  c.score = j_admit - j_move - j_redo - j_revoke + v_reuse;
  c.nonempty = !c.keep.empty() || !c.admitted.empty();
}

// GreedyPack(R): every feasible intermediate allocation, in order
void Decider::greedy_pack(Mask agents, std::vector<Cand>& out) {
  Cand c;
  c.agents = agents;
  for (int r : running_)
    if (agents >> agent_of(r) & 1) c.keep.push_back(r);
  const int n_pre = static_cast<int>(running_.size() - c.keep.size());
  if (p_.K > 0 && n_pre > p_.K) return;
  double used = 0.0;
  for (int a = 0; a < s_.n_agents; ++a)
    if (agents >> a & 1) used += static_cast<double>(s_.prefix_len[a]);
  for (int r : c.keep) used += s_.req_kv[r];
  if (used > p_.budget) return;
  std::vector<int> pool;  // ready requests of agents in R, ascending
  for (int r = 0; r < s_.n_reqs; ++r)
    if (!s_.req_running[r] && (agents >> agent_of(r) & 1)) pool.push_back(r);
  Mask covered = 0;
  for (int r : c.keep) covered |= Mask(1) << agent_of(r);
  std::vector<double> reserve(s_.n_agents, 0.0);
  Mask uncovered = 0;
  for (int a = 0; a < s_.n_agents; ++a) {
    if (!(agents >> a & 1) || (covered >> a & 1)) continue;
    bool any = false;
    double mn = 0.0;
    for (int r : pool)
      if (agent_of(r) == a && (!any || s_.req_kv[r] < mn)) {
        mn = s_.req_kv[r];
        any = true;
      }
    if (!any) return;  // an uncoverable prefix
    reserve[a] = mn;
    uncovered |= Mask(1) << a;
  }
  double total_res = 0.0;
  int n_unc = 0;
  for (int a = 0; a < s_.n_agents; ++a)
    if (uncovered >> a & 1) {
      total_res += reserve[a];
      ++n_unc;
    }
  if (used + total_res > p_.budget || (p_.K > 0 && n_unc > p_.K)) return;
  if (!uncovered) {
    score(c);
    out.push_back(c);
  }
  while (true) {
    int best = -1, best_rep = 0;
    double best_ratio = 0.0, best_gain = 0.0;
    for (int r : pool) {
      // fits: room for r and for the reservations of the other uncovered agents
      double rest = 0.0;
      int slots = 0;
      for (int a = 0; a < s_.n_agents; ++a)
        if ((uncovered >> a & 1) && a != agent_of(r)) {
          rest += reserve[a];
          ++slots;
        }
      if (p_.K > 0 && static_cast<int>(c.admitted.size()) + 1 + slots > p_.K) continue;
      if (!(used + s_.req_kv[r] + rest <= p_.budget)) continue;
      const double gain = age_[s_.req_task[r]] * progress(r, c.admitted);
      const double ratio = gain / s_.req_kv[r];
      int rep = 0;
      for (int q : c.admitted) rep = rep || s_.req_task[q] == s_.req_task[r];
      // key (ratio, represented, -index), largest wins; pool is ascending
      if (best < 0 || ratio > best_ratio || (ratio == best_ratio && rep > best_rep)) {
        best = r;
        best_ratio = ratio;
        best_rep = rep;
        best_gain = gain;
      }
    }
    if (best < 0) break;
    c.admitted.push_back(best);
    c.gains.push_back(best_gain);
    for (size_t k = 0; k < pool.size(); ++k)
      if (pool[k] == best) {
        pool.erase(pool.begin() + static_cast<long>(k));
        break;
      }
    used += s_.req_kv[best];
    uncovered &= ~(Mask(1) << agent_of(best));
    if (!uncovered) {
      score(c);
      out.push_back(c);
    }
  }
}

// adds GreedyPack(R)'s states to the candidates; returns Phi(R)
double Decider::add(Mask agents) {
  std::vector<Cand> sts;
  greedy_pack(agents, sts);
  double phi = kNegInf;
  for (Cand& c : sts) {
    if (c.score > phi) phi = c.score;
    cands_.push_back(std::move(c));
  }
  return phi;
}

void Decider::run(tpa_sched_decision* out) {
  std::vector<int> act;
  for (int a = 0; a < s_.n_agents; ++a)
    if (active_ >> a & 1) act.push_back(a);
  const int na = static_cast<int>(act.size());
  // Single-agent edits of a prefix set (Sec. IV, the Repair neighbourhood):
  // every drop, then every swap of a member for an active non-member.
  auto add_repairs = [&](Mask R) {
    for (int a = 0; a < s_.n_agents; ++a)
      if (R >> a & 1) add(R & ~(Mask(1) << a));
    for (int a = 0; a < s_.n_agents; ++a)
      if (R >> a & 1)
        for (int b : act)
          if (!(R >> b & 1)) add((R & ~(Mask(1) << a)) | (Mask(1) << b));
  };
  // Every superset of R with `extra` (1 or 2) more active agents, in agent
  // order; each adds its GreedyPack states.  Returns the best set's Phi and
  // the set (the first one on ties), or -inf when R has no such superset.
  auto best_superset = [&](Mask R, int extra, Mask* best_R) {
    double best = kNegInf;
    bool have = false;
    auto consider = [&](Mask S) {
      const double v = add(S);
      if (!have || v > best) {
        best = v;
        *best_R = S;
        have = true;
      }
    };
    for (int x = 0; x < na; ++x) {
      if (R >> act[x] & 1) continue;
      if (extra == 1) {
        consider(R | (Mask(1) << act[x]));
        continue;
      }
      for (int y = x + 1; y < na; ++y)
        if (!(R >> act[y] & 1)) consider(R | (Mask(1) << act[x]) | (Mask(1) << act[y]));
    }
    return have ? best : kNegInf;
  };
  if (na <= p_.M) {
    // small pool: every prefix set of the active agents
    for (uint64_t mask = 0; mask < (uint64_t(1) << na); ++mask) {
      Mask R = 0;
      for (int j = 0; j < na; ++j)
        if (mask >> j & 1) R |= Mask(1) << act[j];
      add(R);
    }
  } else {
    // large pool (Algorithm 1): a hill climb on Phi from the resident active
    // prefixes.  It moves to the best one-agent superset while that raises
    // Phi; where none does, it may take the best two-agent superset, once per
    // decision; it stops when neither helps.  The start and the end point
    // also contribute their Repair neighbourhoods, and the incumbent stays.
    Mask rg = r_now_ & active_;
    add(rg);
    add_repairs(rg);
    double phi_g;
    {
      std::vector<Cand> tmp;
      greedy_pack(rg, tmp);
      phi_g = kNegInf;
      for (const Cand& c : tmp)
        if (c.score > phi_g) phi_g = c.score;
    }
    int two_agent_steps = 1;
    for (;;) {
      Mask next = 0;
      double v = best_superset(rg, 1, &next);
      if (!(v > phi_g)) {
        if (two_agent_steps == 0) break;
        --two_agent_steps;
        v = best_superset(rg, 2, &next);
        if (!(v > phi_g)) break;
      }
      rg = next;
      phi_g = v;
    }
    add_repairs(rg);
    Cand inc;
    inc.agents = r_now_;
    inc.keep = running_;
    score(inc);
    cands_.push_back(inc);
  }
  if (cands_.empty()) {  // nothing feasible was generated: keep the incumbent
    Cand inc;
    inc.agents = r_now_;
    inc.keep = running_;
    score(inc);
    cands_.push_back(inc);
  }
  bool any_nonempty = false;
  for (const Cand& c : cands_) any_nonempty = any_nonempty || c.nonempty;
  const Cand* best = nullptr;
  for (const Cand& c : cands_) {
    if (any_nonempty && !c.nonempty) continue;
    if (!best || c.score > best->score) best = &c;
  }
  out->n_candidates = static_cast<int64_t>(cands_.size());
  for (int a = 0; a < s_.n_agents; ++a) out->agents[a] = 0;
  for (int r = 0; r < s_.n_reqs; ++r) out->running[r] = 0;
  out->n_admitted = out->n_preempted = 0;
  out->score = out->j_admit = out->j_move = out->j_redo = out->j_revoke = out->v_reuse = 0.0;
  for (int a = 0; a < s_.n_agents; ++a) out->agents[a] = (best->agents >> a & 1) ? 1 : 0;
  for (int r : best->keep) out->running[r] = 1;
  for (size_t k = 0; k < best->admitted.size(); ++k) {
    out->running[best->admitted[k]] = 1;
    out->admitted[k] = best->admitted[k];
    out->credits[k] = best->gains[k];
  }
  out->n_admitted = static_cast<int32_t>(best->admitted.size());
  out->n_preempted = static_cast<int32_t>(running_.size() - best->keep.size());
  out->score = best->score;
  out->j_admit = best->j_admit;
  out->j_move = best->j_move;
  out->j_redo = best->j_redo;
  out->j_revoke = best->j_revoke;
  out->v_reuse = best->v_reuse;
}

int invalid(const char* msg) { return tpa::set_error(TPA_ERR_INVALID_ARG, msg); }

int validate(const tpa_sched_params* p, const tpa_sched_snapshot* s, const tpa_sched_decision* o) {
  if (!p || !s || !o) return invalid("null argument");
  if (!(p->b_swap > 0.0) || !(p->h_age > 0.0) || p->mc_samples < 1 || p->M < 0 || p->M > 20 || p->K < 0)
    return invalid("bad parameters (b_swap, h_age > 0; mc_samples >= 1; 0 <= M <= 20; K >= 0)");
  if (s->n_stages < 1 || s->n_agents < 1 || s->n_agents > 64 || s->n_tasks < 0 || s->n_reqs < 0)
    return invalid("bad snapshot sizes (n_agents in 1..64)");
  if (!s->stage_agent || !s->pred_off || !s->prefix_len || !s->sample_off || !s->samples ||
      !s->resident || (s->n_tasks && (!s->task_id || !s->task_arrival || !s->stage_state ||
                                      !s->stage_served)) ||
      (s->n_reqs && (!s->req_task || !s->req_stage || !s->req_kv || !s->req_dhat || !s->req_redo ||
                     !s->req_credit || !s->req_running || !o->agents || !o->running ||
                     !o->admitted || !o->credits)) ||
      !o->agents)
    return invalid("null snapshot or output array");
  if (s->pred_off[0] != 0 || s->sample_off[0] != 0) return invalid("CSR offsets must start at 0");
  for (int v = 0; v < s->n_stages; ++v) {
    if (s->stage_agent[v] < 0 || s->stage_agent[v] >= s->n_agents) return invalid("stage agent out of range");
    if (s->pred_off[v + 1] < s->pred_off[v]) return invalid("predecessor offsets decrease");
    if (s->pred_off[v + 1] > s->pred_off[v] && !s->pred_idx) return invalid("null predecessor array");
    for (int k = s->pred_off[v]; k < s->pred_off[v + 1]; ++k)
      if (s->pred_idx[k] < 0 || s->pred_idx[k] >= v) return invalid("a predecessor is not before its stage");
    if (s->sample_off[v + 1] <= s->sample_off[v]) return invalid("a stage without samples");
  }
  for (int a = 0; a < s->n_agents; ++a)
    if (s->prefix_len[a] < 0) return invalid("negative prefix length");
  for (size_t k = 0; k < static_cast<size_t>(s->n_tasks) * s->n_stages; ++k)
    if (s->stage_state[k] < 0 || s->stage_state[k] > 2) return invalid("stage state not 0, 1 or 2");
  for (int r = 0; r < s->n_reqs; ++r) {
    if (s->req_task[r] < 0 || s->req_task[r] >= s->n_tasks) return invalid("request task out of range");
    if (s->req_stage[r] < 0 || s->req_stage[r] >= s->n_stages) return invalid("request stage out of range");
    if (!(s->req_kv[r] > 0.0) || !(s->req_dhat[r] >= 0.0)) return invalid("request needs d_r > 0 and D_r >= 0");
  }
  return TPA_OK;
}

}  // namespace

extern "C" TPA_API int tpa_sched_decide(const tpa_sched_params* params, const tpa_sched_snapshot* snap,
                                        tpa_sched_decision* out) {
  const int rc = validate(params, snap, out);
  if (rc) return rc;
  Decider d(*params, *snap);
  d.run(out);
  return TPA_OK;
}
