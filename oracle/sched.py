"""Plain CPU restatement of the TOPAS scheduling decision (test infrastructure).

Imported only by tests/ and bench.py's baseline legs; the library never
imports it.  It evaluates one scheduling event from a flat snapshot of the
serving state, following Sec. IV of the paper:

  * stage residuals Z = X - e | X > e over the empirical stage-service
    samples (Eq. 3), hypothetical completions [Z - D_r]_+ (Sec. IV-B);
  * the expected longest remaining path E[LP(G, Z)] in reverse topological
    order (Eq. 4) and the conditional progress of a request (Eq. 5);
  * J_admit with task aging (Eqs. 6, 11), J_move (Eq. 7), J_redo (Eq. 8),
    J_revoke (Eq. 9), V_reuse (Eq. 10) and the full score (Eq. 12);
  * GreedyPack and the hierarchical prefix-set search (Sec. IV-E,
    Algorithm 1) with the caps M and K and deterministic ties (Eq. 13).

Readings where the paper is silent (each is also what the native module
does):

  R1  The expectation in Eq. 4 is a Monte-Carlo mean over `mc_samples`
      joint draws.  Draw k of stage v of task i picks residual sample
      splitmix64(splitmix64(splitmix64(seed ^ task_id) ^ v) ^ k) mod n,
      the same draws for every hypothetical set (common random numbers),
      so conditional progress is never negative.  splitmix64 is the
      generator published by S. Vigna (constants 0x9E3779B97F4A7C15,
      0xBF58476D1CE4E5B9, 0x94D049BB133111EB; shifts 30, 27, 31).
  R2  A started stage that has already received more service than every
      sample has residual 0; done stages have residual 0; unstarted stages
      take the samples themselves.
  R3  The longest remaining path is lp[v] = z_v + max(0, max over
      successors lp[s]), over stages listed in topological order
      (every predecessor index smaller), and LP = max over v of lp[v].
  R4  D_r (the expected service of a request) is an input: the caller
      forms it from the request-service history of its agent-stage pair,
      or from the profile T_prefill(input) + T_decode * max_new.
  R5  GreedyPack admits, at each step, the fitting ready request of an
      agent in R with the largest g_i * Delta / d_r; ties go to a request
      whose task already has an admission in this allocation, then to the
      lowest request index.  A request fits when, after it, every agent
      of R still without a request can get its reserved request (the
      agent's ready request with the smallest d_r) within the budget and
      within the admission cap K.
  R6  States are generated in a fixed order (prefix sets in increasing
      bitmask order over the agent ids sorted ascending; within a set, the
      allocation before any admission, then after each admission); the
      first state with the largest score wins.  "Improves Phi" is strictly
      greater.
  R7  n_a(t) counts unstarted stages of agent a whose unfinished
      predecessors are exactly one, and that one started (running).
  R8  The incumbent's running requests keep their stored credit lambda_r
      (age-weighted, Sec. IV-D); an admitted request's credit is
      g_i(t) * Delta at this event.
  R9  The bounded search of Algorithm 1 starts from R_t restricted to the
      active agents A_t (a resident prefix without requests cannot be
      covered, so it always leaves); repairs drop one agent of R or swap
      one for an agent of A_t outside R.
  R10 When no state is generated at all (the caps forbid every change and
      the incumbent's requests do not all fit), the incumbent is kept.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List

MASK64 = (1 << 64) - 1


def splitmix64(x: int) -> int:
    """One step of SplitMix64 (Vigna), as a pure function of a 64-bit input."""
    z = (x + 0x9E3779B97F4A7C15) & MASK64
    z = ((z ^ (z >> 30)) * 0xBF58476D1CE4E5B9) & MASK64
    z = ((z ^ (z >> 27)) * 0x94D049BB133111EB) & MASK64
    return z ^ (z >> 31)


def draw_index(seed: int, task_id: int, stage: int, k: int, n: int) -> int:
    """R1: index of the residual sample of draw k (stage, task)."""
    h = splitmix64((seed ^ task_id) & MASK64)
    h = splitmix64(h ^ stage)
    h = splitmix64(h ^ k)
    return h % n


@dataclass
class Params:
    budget: float          # B_t, token-equivalent KV capacity
    mu: float              # KV bytes per prefix token
    b_swap: float          # swap bandwidth, bytes/s
    t_decode: float        # profiled decode time per token, s
    beta: float = 1.0      # V_reuse pressure (Eq. 10)
    rho: float = 0.0       # aging strength (Eq. 11)
    h_age: float = 1.0     # aging scale, s
    M: int = 6             # enumerate all prefix sets when |A_t| <= M
    K: int = 0             # cap on admissions and on preemptions (0 = none)
    mc_samples: int = 32   # draws of the expectation (R1)
    seed: int = 0


@dataclass
class Snapshot:
    t: float
    stage_agent: List[int]            # agent of each stage (stages topologically ordered)
    stage_preds: List[List[int]]      # predecessors of each stage (indices < the stage)
    prefix_len: List[int]             # l_a per agent, tokens
    stage_samples: List[List[float]]  # empirical total-service samples per stage (>= 1 each)
    task_id: List[int]                # stable id of each task (the draws key on it)
    task_arrival: List[float]         # tau_i
    stage_state: List[List[int]]      # [task][stage]: 0 unstarted, 1 started, 2 done
    stage_served: List[List[float]]   # [task][stage]: e_{i,v}(t)
    req_task: List[int]               # index into the task arrays
    req_stage: List[int]
    req_kv: List[float]               # d_r(t): request-specific KV reservation, tokens
    req_dhat: List[float]             # D_r(t), s (R4)
    req_redo: List[float]             # y_r(t), tokens to rebuild if preempted
    req_running: List[bool]           # in Q_t (else ready, in W_t)
    req_credit: List[float]           # lambda_r of running requests
    resident: List[bool]              # R_t per agent


@dataclass
class State:
    agents: tuple                     # R', sorted agent ids
    running: tuple                    # Q', sorted request indices
    admitted: tuple                   # A in greedy order
    preempted: tuple                  # P, sorted
    score: float
    j_admit: float
    j_move: float
    j_redo: float
    j_revoke: float
    v_reuse: float
    credits: tuple = field(default=())  # lambda of each admitted request, greedy order


# ------------------------------------------------------------ remaining paths

def _residual_values(s: Snapshot, i: int, v: int) -> List[float]:
    """R2: support of Z_{i,v}(t) (Eq. 3), in sample order."""
    st = s.stage_state[i][v]
    if st == 2:
        return [0.0]
    if st == 0:
        return list(s.stage_samples[v])
    e = s.stage_served[i][v]
    vals = [x - e for x in s.stage_samples[v] if x > e]
    return vals if vals else [0.0]


def _succs(s: Snapshot) -> List[List[int]]:
    n = len(s.stage_agent)
    succ = [[] for _ in range(n)]
    for v in range(n):
        for u in s.stage_preds[v]:
            succ[u].append(v)
    return succ


def longest_path(z: List[float], succ: List[List[int]]) -> float:
    """R3: longest remaining path of one residual realization."""
    n = len(z)
    lp = [0.0] * n
    best = 0.0
    for v in range(n - 1, -1, -1):
        m = 0.0
        for w in succ[v]:
            if lp[w] > m:
                m = lp[w]
        lp[v] = z[v] + m
        if lp[v] > best:
            best = lp[v]
    return best


def expected_remaining_path(s: Snapshot, p: Params, i: int, done: dict) -> float:
    """Eq. 4: L_i(H, t), H given as {stage: total D of its hypothetical completions}."""
    n = len(s.stage_agent)
    succ = _succs(s)
    vals = [_residual_values(s, i, v) for v in range(n)]
    total = 0.0
    for k in range(p.mc_samples):
        z = []
        for v in range(n):
            x = vals[v][draw_index(p.seed, s.task_id[i], v, k, len(vals[v]))]
            d = done.get(v, 0.0)
            z.append(x - d if x - d > 0.0 else 0.0)
        total += longest_path(z, succ)
    return total / p.mc_samples


def aging(s: Snapshot, p: Params, i: int) -> float:
    """Eq. 11: g_i(t)."""
    age = s.t - s.task_arrival[i]
    return 1.0 + p.rho * math.log(1.0 + (age if age > 0.0 else 0.0) / p.h_age)


def progress(s: Snapshot, p: Params, r: int, admitted: List[int]) -> float:
    """Eq. 5: Delta_task(r | A_i^{<r}), the earlier admissions of r's task."""
    i = s.req_task[r]
    before = {}
    for q in admitted:
        if s.req_task[q] == i:
            before[s.req_stage[q]] = before.get(s.req_stage[q], 0.0) + s.req_dhat[q]
    after = dict(before)
    after[s.req_stage[r]] = after.get(s.req_stage[r], 0.0) + s.req_dhat[r]
    return expected_remaining_path(s, p, i, before) - expected_remaining_path(s, p, i, after)


def reuse_counts(s: Snapshot) -> List[int]:
    """R7: n_a(t) per agent."""
    n_a = [0] * len(s.prefix_len)
    for i in range(len(s.task_id)):
        for v in range(len(s.stage_agent)):
            if s.stage_state[i][v] != 0:
                continue
            unfinished = [u for u in s.stage_preds[v] if s.stage_state[i][u] != 2]
            if len(unfinished) == 1 and s.stage_state[i][unfinished[0]] == 1:
                n_a[s.stage_agent[v]] += 1
    return n_a


# ------------------------------------------------------------ scoring

def _agent(s: Snapshot, r: int) -> int:
    return s.stage_agent[s.req_stage[r]]


def score_state(s: Snapshot, p: Params, agents: set, keep: List[int], admitted: List[int],
                gains: List[float], n_a: List[int]) -> State:
    """Eq. 12 for the state (R' = agents, Q' = keep + admitted)."""
    running = [r for r in range(len(s.req_task)) if s.req_running[r]]
    preempted = sorted(r for r in running if r not in keep)
    j_admit = 0.0
    for gain in gains:
        j_admit += gain
    r_now = {a for a in range(len(s.prefix_len)) if s.resident[a]}
    r_in = sorted(a for a in agents if a not in r_now)
    r_out = sorted(a for a in r_now if a not in agents)
    moved = 0.0
    for a in r_out:
        moved += s.prefix_len[a]
    for a in r_in:
        moved += s.prefix_len[a]
    t_move = p.mu / p.b_swap * moved
    tasks_in = {s.req_task[r] for r in admitted if _agent(s, r) in r_in}
    j_move = t_move * len(tasks_in)
    j_redo = 0.0
    j_revoke = 0.0
    for r in preempted:
        j_redo += p.t_decode * s.req_redo[r]
        j_revoke += s.req_credit[r]
    v_reuse = 0.0
    for a in sorted(agents):
        v_reuse += p.beta * n_a[a] * p.mu * s.prefix_len[a] / p.b_swap
    score = j_admit - j_move - j_redo - j_revoke + v_reuse
    return State(tuple(sorted(agents)), tuple(sorted(keep + admitted)), tuple(admitted),
                 tuple(preempted), score, j_admit, j_move, j_redo, j_revoke, v_reuse,
                 tuple(gains))


def greedy_pack(s: Snapshot, p: Params, agents: set, n_a: List[int]) -> List[State]:
    """GreedyPack(R) (Sec. IV-E, R5): every feasible intermediate allocation."""
    nreq = len(s.req_task)
    running = [r for r in range(nreq) if s.req_running[r]]
    keep = [r for r in running if _agent(s, r) in agents]
    n_pre = len(running) - len(keep)
    if p.K > 0 and n_pre > p.K:
        return []
    used = 0.0
    for a in sorted(agents):
        used += s.prefix_len[a]
    for r in keep:
        used += s.req_kv[r]
    if used > p.budget:
        return []
    ready = [r for r in range(nreq) if not s.req_running[r] and _agent(s, r) in agents]
    covered = {_agent(s, r) for r in keep}
    reserve = {}
    for a in sorted(agents):
        if a in covered:
            continue
        cand = [s.req_kv[r] for r in ready if _agent(s, r) == a]
        if not cand:
            return []       # an uncoverable prefix: R' must equal {a(r) : r in Q'}
        reserve[a] = min(cand)

    def fits(r, n_adm):
        rest = 0.0
        slots = 0
        for a in sorted(reserve):
            if a != _agent(s, r):
                rest += reserve[a]
                slots += 1
        if p.K > 0 and n_adm + 1 + slots > p.K:
            return False
        return used + s.req_kv[r] + rest <= p.budget

    total_res = 0.0
    for a in sorted(reserve):
        total_res += reserve[a]
    if used + total_res > p.budget or (p.K > 0 and len(reserve) > p.K):
        return []
    out = []
    admitted, gains = [], []
    if not reserve:
        out.append(score_state(s, p, agents, keep, admitted, gains, n_a))
    pool = list(ready)
    while True:
        best = None
        best_key = None
        tasks_adm = {s.req_task[q] for q in admitted}
        for r in pool:
            if not fits(r, len(admitted)):
                continue
            gain = aging(s, p, s.req_task[r]) * progress(s, p, r, admitted)
            ratio = gain / s.req_kv[r]
            key = (ratio, 1 if s.req_task[r] in tasks_adm else 0, -r)
            if best_key is None or key > best_key:
                best, best_key, best_gain = r, key, gain
        if best is None:
            break
        admitted.append(best)
        gains.append(best_gain)
        pool.remove(best)
        used += s.req_kv[best]
        reserve.pop(_agent(s, best), None)
        if not reserve:
            out.append(score_state(s, p, agents, keep, admitted, gains, n_a))
    return out


def _phi(states: List[State]) -> float:
    return max((st.score for st in states), default=-math.inf)


def decide(s: Snapshot, p: Params) -> State:
    """Algorithm 1: generate candidate states and select by Eq. 13."""
    n_a = reuse_counts(s)
    nreq = len(s.req_task)
    active = sorted({_agent(s, r) for r in range(nreq)})
    cands: List[State] = []
    r_now = {a for a in range(len(s.prefix_len)) if s.resident[a]}

    def add(sets):
        best = -math.inf
        for R in sets:
            sts = greedy_pack(s, p, set(R), n_a)
            cands.extend(sts)
            best = max(best, _phi(sts))
        return best

    def repair(R):
        sets = []
        for a in sorted(R):
            sets.append(R - {a})
        for a in sorted(R):
            for b in active:
                if b not in R:
                    sets.append((R - {a}) | {b})
        return sets

    if len(active) <= p.M:
        for mask in range(1 << len(active)):
            add([{active[j] for j in range(len(active)) if mask >> j & 1}])
    else:
        rg = set(r_now) & set(active)
        add([rg] + repair(rg))
        phi_g = _phi(greedy_pack(s, p, rg, n_a))
        pair_tried = False
        while True:
            singles = [rg | {a} for a in active if a not in rg]
            best_v, best_R = -math.inf, None
            for R in singles:
                v = add([R])
                if v > best_v:
                    best_v, best_R = v, R
            if best_R is not None and best_v > phi_g:
                rg, phi_g = best_R, best_v
                continue
            if pair_tried:
                break
            pair_tried = True
            rest = [a for a in active if a not in rg]
            best_v, best_R = -math.inf, None
            for x in range(len(rest)):
                for y in range(x + 1, len(rest)):
                    R = rg | {rest[x], rest[y]}
                    v = add([R])
                    if v > best_v:
                        best_v, best_R = v, R
            if best_R is not None and best_v > phi_g:
                rg, phi_g = best_R, best_v
            else:
                break
        add(repair(rg))
        # the incumbent itself
        inc_keep = [r for r in range(nreq) if s.req_running[r]]
        cands.append(score_state(s, p, r_now, inc_keep, [], [], n_a))
    if not cands:   # R10
        cands.append(score_state(s, p, r_now, [r for r in range(nreq) if s.req_running[r]],
                                 [], [], n_a))
    nonempty = [st for st in cands if st.running]
    if nonempty:
        cands = nonempty
    best = None
    for st in cands:
        if best is None or st.score > best.score:
            best = st
    return best
