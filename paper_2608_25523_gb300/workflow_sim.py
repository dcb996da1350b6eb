"""Multi-agent workflow tasks served by TOPAS decisions on one library context.

A discrete-event driver: tasks of one DAG workflow (Sec. III; e.g. the
paper's Chain-3 shape) arrive by a seeded Poisson process, each stage issues
one LLM request under its agent's static prefix, and at every scheduling
event the driver builds the state snapshot, asks the native scheduler
(tpa_sched_decide, Sec. IV) for the next prefix-request state and applies it
through the library:

  prefixes that leave R     tpa_prefix_offload (to pinned host) / evict
  prefixes that enter R     tpa_prefix_register + write the first time,
                            tpa_prefix_reload from the host copy later
  preempted requests        tpa_request_close (their KV is rebuilt on
                            re-admission by chunked prefill of input + y_r)
  admitted requests         tpa_request_open + tpa_prefill_chunk
  the running set           one tpa_decode step per simulated step

Service times are synthetic (a time per prefill token, per decode step and
the movement cost mu / B_swap per prefix token); the library does the real
page-table work (its NO_SPACE check holds the scheduler to the budget of
Eq. 2) and, on a GPU context, the real attention kernels on synthetic Q/K/V.
A plan-only context (TPA_FLAG_PLAN_ONLY) runs the same driver without a GPU.
"""
from __future__ import annotations

import time
from dataclasses import dataclass, field
from typing import Callable, List, Optional

import numpy as np

from . import binding as B

PAGE = 16


def _pages(tokens: int) -> int:
    return (tokens + PAGE - 1) // PAGE


@dataclass
class Workflow:
    name: str
    stage_agent: List[int]
    stage_preds: List[List[int]]
    prefix_len: List[int]        # l_a, tokens
    input_tokens: List[int]      # per stage: new suffix tokens of its request
    output_tokens: List[int]     # per stage: decode tokens of its request


def chain3() -> Workflow:
    """Three agents in a line with fixed per-stage queries and generations
    (the shape of the paper's Chain-3 workload; sizes are this driver's)."""
    return Workflow("chain3", [0, 1, 2], [[], [0], [1]], [2048, 4096, 3072],
                    [512, 384, 256], [128, 192, 96])


def dag4() -> Workflow:
    """A fork/join: planner -> {coder, tester} -> reviewer."""
    return Workflow("dag4", [0, 1, 2, 3], [[], [0], [0], [1, 2]], [2048, 3072, 3072, 1536],
                    [384, 256, 256, 192], [96, 160, 64, 96])


@dataclass
class Timing:
    t_prefill_token: float = 2.0e-5   # s per prefilled token
    t_decode_step: float = 0.02       # s per decode step of the running batch
    mu: float = 4096.0                # KV bytes per prefix token (one layer's)
    b_swap: float = 20e9              # bytes/s of prefix movement


@dataclass
class SchedKnobs:
    beta: float = 1.0
    rho: float = 0.5
    h_age: float = 10.0
    M: int = 6
    K: int = 0
    mc_samples: int = 16
    seed: int = 1


@dataclass
class _Req:
    task: int
    stage: int
    generated: int = 0      # decode tokens produced in the current attempt
    redo: int = 0           # tokens whose KV a re-admission rebuilds (y_r at preemption)
    served: float = 0.0     # LLM service received, s
    running: bool = False
    lib_id: int = -1
    credit: float = 0.0


@dataclass
class Result:
    jct: List[float] = field(default_factory=list)
    decisions: int = 0
    decide_us: List[float] = field(default_factory=list)
    candidates: int = 0
    prefix_in: int = 0
    prefix_out: int = 0
    preemptions: int = 0
    steps: int = 0
    decode_tokens: int = 0
    prefill_tokens: int = 0
    sim_time: float = 0.0
    wall_s: float = 0.0

    def summary(self) -> dict:
        j = sorted(self.jct)
        lat = sorted(self.decide_us)
        pick = lambda xs, q: xs[min(len(xs) - 1, int(q * len(xs)))] if xs else None
        return {"tasks": len(j), "mean_jct_s": round(float(np.mean(j)), 3) if j else None,
                "p99_jct_s": round(float(pick(j, 0.99)), 3) if j else None, "decisions": self.decisions,
                "decide_us_mean": round(float(np.mean(lat)), 1) if lat else None,
                "decide_us_p99": round(pick(lat, 0.99), 1) if lat else None,
                "candidates_per_decision": round(self.candidates / max(1, self.decisions), 1),
                "prefix_moves_in": self.prefix_in, "prefix_moves_out": self.prefix_out,
                "preemptions": self.preemptions, "steps": self.steps,
                "decode_tokens": self.decode_tokens, "prefill_tokens": self.prefill_tokens,
                "sim_time_s": round(self.sim_time, 3), "wall_s": round(self.wall_s, 3)}


class WorkflowSim:
    """Serve `n_tasks` tasks of `wf` on `ctx` (a GPU or plan-only Context
    with Hq/Hkv/d of `dims`).  On a GPU context `device` must be set."""

    def __init__(self, wf: Workflow, ctx: B.Context, *, n_tasks: int, rate: float, seed: int,
                 dims=(8, 2, 64), budget_pages: int, max_tokens: int, max_requests: int,
                 timing: Timing = Timing(), knobs: SchedKnobs = SchedKnobs(),
                 device: Optional[str] = None, record: Optional[list] = None,
                 on_launch: Optional[Callable] = None):
        self.wf, self.ctx, self.tm, self.kn = wf, ctx, timing, knobs
        self.record = record   # if a list: every decision's (params, snapshot, decision)
        # Called after every prefill chunk as on_launch(self, "prefill", (lib_id, offset, c))
        # and after every decode step as on_launch(self, "decode", ids), with the
        # launches still in flight.  kv_log[lib_id] lists what the request's suffix
        # holds, in order: ("pf", c) = rows 0..c-1 of k_pf / v_pf (one prefill
        # chunk), ("dec", j) = row j of k_dec / v_dec (one decode token); events
        # lists ("reload", agent), ("preempt", lib_id) and ("rebuild", lib_id,
        # tokens) in the order they happened.
        self.on_launch = on_launch
        self.kv_log = {}
        self.lib_agent = {}     # lib_id -> agent of the request it holds
        self.events = []
        self.hq, self.hkv, self.d = dims
        self.budget_tokens = budget_pages * PAGE
        self.max_tokens = max_tokens
        rng = np.random.default_rng(seed)
        gaps = rng.exponential(1.0 / rate, size=n_tasks)
        self.arrivals = list(np.cumsum(gaps))
        self.task_ids = [int(x) for x in rng.integers(0, 2**62, size=n_tasks)]
        ns = len(wf.stage_agent)
        # stage-service profile: a point mass at T_prefill(input) + T_decode * max_new
        self.samples = [[timing.t_prefill_token * wf.input_tokens[v] +
                         timing.t_decode_step * wf.output_tokens[v]] for v in range(ns)]
        self.observed = [[] for _ in range(ns)]
        self.free_ids = list(range(max_requests))[::-1]
        self.device = device
        self.agent_state = ["new"] * len(wf.prefix_len)   # new | resident | host
        self.host_kv = {}
        self.res = Result()
        if device is not None:
            import torch
            g = torch.Generator(device="cpu").manual_seed(seed)
            def rnd(*shape):
                return torch.randn(*shape, generator=g).to(torch.bfloat16)
            self.q_pf = rnd(max_tokens, self.hq, self.d).to(device)
            self.k_pf = rnd(max_tokens, self.hkv, self.d).to(device)
            self.v_pf = rnd(max_tokens, self.hkv, self.d).to(device)
            self.o_pf = torch.empty_like(self.q_pf)
            self.l_pf = torch.empty(max_tokens, self.hq, dtype=torch.float32, device=device)
            nb = max_requests
            self.q_dec = rnd(nb, self.hq, self.d).to(device)
            self.k_dec = rnd(nb, self.hkv, self.d).to(device)
            self.v_dec = rnd(nb, self.hkv, self.d).to(device)
            self.o_dec = torch.empty_like(self.q_dec)
            self.l_dec = torch.empty(nb, self.hq, dtype=torch.float32, device=device)
            for a, L in enumerate(wf.prefix_len):
                hk = rnd(L, self.hkv, self.d).pin_memory()
                hv = rnd(L, self.hkv, self.d).pin_memory()
                self.host_kv[a] = (hk, hv)

    # ------------------------------------------------------------ library
    def _prefix_in(self, a):
        L = self.wf.prefix_len[a]
        if self.agent_state[a] == "new":
            self.ctx.prefix_register(a, L)
            if self.device is not None:
                hk, hv = self.host_kv[a]
                self.ctx.prefix_write(a, hk, hv)
        else:
            hk, hv = self.host_kv.get(a, (1, 1))
            self.ctx.prefix_reload(a, hk, hv)
            self.events.append(("reload", a))
        self.agent_state[a] = "resident"
        self.res.prefix_in += 1

    def _prefix_out(self, a):
        hk, hv = self.host_kv.get(a, (1, 1))
        self.ctx.prefix_offload(a, hk, hv)
        self.agent_state[a] = "host"
        self.res.prefix_out += 1

    def _prefill(self, lib_id, ntok):
        done = 0
        while done < ntok:
            c = min(self.max_tokens, ntok - done)
            if self.device is not None:
                self.ctx.prefill_chunk([lib_id], [c], self.q_pf, self.k_pf, self.v_pf,
                                       self.o_pf, self.l_pf)
            else:
                self.ctx.prefill_chunk([lib_id], [c], 1, 1, 1, 1, 1)
            self.kv_log.setdefault(lib_id, []).append(("pf", c))
            if self.on_launch is not None:
                self.on_launch(self, "prefill", (lib_id, done, c))
            done += c
        self.res.prefill_tokens += ntok

    def _decode(self, ids):
        if self.device is not None:
            n = len(ids)
            self.ctx.decode(ids, self.q_dec[:n], self.k_dec[:n], self.v_dec[:n],
                            self.o_dec[:n], self.l_dec[:n])
        else:
            self.ctx.decode(ids, 1, 1, 1, 1, 1)
        for j, i in enumerate(ids):
            self.kv_log.setdefault(i, []).append(("dec", j))
        if self.on_launch is not None:
            self.on_launch(self, "decode", list(ids))
        self.res.decode_tokens += len(ids)

    # ------------------------------------------------------------ state
    def _kv(self, r: _Req) -> float:
        """d_r: the request's whole suffix (input and every output token), page-rounded."""
        v = r.stage
        return float(_pages(self.wf.input_tokens[v] + self.wf.output_tokens[v]) * PAGE)

    def _dhat(self, r: _Req) -> float:
        obs = self.observed[r.stage]
        mean = (sum(obs) / len(obs)) if obs else self.samples[r.stage][0]
        return max(0.0, mean - r.served)

    def run(self) -> Result:
        wf = self.wf
        ns = len(wf.stage_agent)
        t = 0.0
        nxt = 0                              # next arrival
        tasks = {}                           # index -> dict(state, served)
        reqs: List[_Req] = []
        t0 = time.perf_counter()
        resident = set()
        event = False
        while nxt < len(self.arrivals) or tasks:
            # arrivals up to t
            while nxt < len(self.arrivals) and self.arrivals[nxt] <= t:
                tasks[nxt] = {"state": [0] * ns, "served": [0.0] * ns, "arrival": self.arrivals[nxt]}
                for v in range(ns):
                    if not wf.stage_preds[v]:
                        tasks[nxt]["state"][v] = 1
                        reqs.append(_Req(nxt, v))
                nxt += 1
                event = True
            if not reqs:
                if nxt < len(self.arrivals):
                    t = max(t, self.arrivals[nxt])
                    continue
                break
            if event:
                t += self._decide(t, tasks, reqs, resident)
                event = False
            running = [r for r in reqs if r.running]
            if not running:
                # nothing admissible now: wait for the next arrival
                if nxt < len(self.arrivals):
                    t = max(t, self.arrivals[nxt])
                    event = True
                    continue
                raise RuntimeError("no state admits any ready request (budget too small)")
            # one decode step of the running batch
            self._decode([r.lib_id for r in running])
            self.res.steps += 1
            t += self.tm.t_decode_step
            for r in running:
                r.generated += 1
                r.served += self.tm.t_decode_step
                tasks[r.task]["served"][r.stage] += self.tm.t_decode_step
            # completions (committed before the next decision)
            for r in [r for r in running if r.generated >= wf.output_tokens[r.stage]]:
                self.ctx.request_close(r.lib_id)
                self.kv_log.pop(r.lib_id, None)
                self.free_ids.append(r.lib_id)
                reqs.remove(r)
                tk = tasks[r.task]
                tk["state"][r.stage] = 2
                self.observed[r.stage].append(r.served)
                for v in range(ns):
                    if tk["state"][v] == 0 and all(tk["state"][u] == 2 for u in wf.stage_preds[v]):
                        tk["state"][v] = 1
                        reqs.append(_Req(r.task, v))
                if all(x == 2 for x in tk["state"]):
                    self.res.jct.append(float(t - tk["arrival"]))
                    del tasks[r.task]
                event = True
        self.res.sim_time = float(t)
        self.res.wall_s = time.perf_counter() - t0
        if self.device is not None:
            import torch
            torch.cuda.synchronize()
        return self.res

    def _decide(self, t, tasks, reqs, resident) -> float:
        """One scheduling event: snapshot, decision, application.  Returns the
        simulated time the transition takes (prefix moves, then the admitted
        requests' prefills, serialized)."""
        wf = self.wf
        ns = len(wf.stage_agent)
        order = sorted(tasks)
        index = {k: i for i, k in enumerate(order)}
        for v in range(ns):
            if self.observed[v]:
                self.samples[v] = list(self.observed[v])
        snap = _Snap(
            t=t, stage_agent=wf.stage_agent, stage_preds=wf.stage_preds,
            prefix_len=[_pages(L) * PAGE for L in wf.prefix_len],
            stage_samples=self.samples, task_id=[self.task_ids[k] for k in order],
            task_arrival=[tasks[k]["arrival"] for k in order],
            stage_state=[tasks[k]["state"] for k in order],
            stage_served=[tasks[k]["served"] for k in order],
            req_task=[index[r.task] for r in reqs], req_stage=[r.stage for r in reqs],
            req_kv=[self._kv(r) for r in reqs], req_dhat=[self._dhat(r) for r in reqs],
            req_redo=[float(r.generated) for r in reqs], req_running=[r.running for r in reqs],
            req_credit=[r.credit for r in reqs],
            resident=[a in resident for a in range(len(wf.prefix_len))])
        prm = _Prm(budget=float(self.budget_tokens), mu=self.tm.mu, b_swap=self.tm.b_swap,
                   t_decode=self.tm.t_decode_step, beta=self.kn.beta, rho=self.kn.rho,
                   h_age=self.kn.h_age, M=self.kn.M, K=self.kn.K, mc_samples=self.kn.mc_samples,
                   seed=self.kn.seed)
        c0 = time.perf_counter()
        dec = B.sched_decide(prm, snap)
        self.res.decide_us.append((time.perf_counter() - c0) * 1e6)
        if self.record is not None:
            import copy
            self.record.append((copy.deepcopy(prm), copy.deepcopy(snap), dec))
        self.res.decisions += 1
        self.res.candidates += dec["n_candidates"]
        keep = set(dec["running"])
        # preemptions first (their pages return), then prefixes out, then in
        for i, r in enumerate(reqs):
            if r.running and i not in keep:
                self.ctx.request_close(r.lib_id)
                self.kv_log.pop(r.lib_id, None)
                self.events.append(("preempt", r.lib_id))
                self.free_ids.append(r.lib_id)
                r.running, r.lib_id, r.credit = False, -1, 0.0
                r.redo = r.generated          # y_r: rebuilt on re-admission
                r.generated = 0
                self.res.preemptions += 1
        new_r = set(dec["agents"])
        moved = 0
        for a in sorted(resident - new_r):
            self._prefix_out(a)
            moved += wf.prefix_len[a]
        for a in sorted(new_r - resident):
            self._prefix_in(a)
            moved += wf.prefix_len[a]
        resident.clear()
        resident.update(new_r)
        dt = self.tm.mu / self.tm.b_swap * moved
        for i, lam in zip(dec["admitted"], dec["credits"]):
            r = reqs[i]
            r.lib_id = self.free_ids.pop()
            self.ctx.request_open(r.lib_id, wf.stage_agent[r.stage])
            self.kv_log[r.lib_id] = []
            self.lib_agent[r.lib_id] = wf.stage_agent[r.stage]
            ntok = self.wf.input_tokens[r.stage] + r.redo
            if r.redo:
                self.events.append(("rebuild", r.lib_id, ntok))
            self._prefill(r.lib_id, ntok)
            r.generated, r.redo = r.redo, 0
            r.running, r.credit = True, lam
            tp = self.tm.t_prefill_token * ntok
            dt += tp
            r.served += tp
            tasks[r.task]["served"][r.stage] += tp
        return dt


@dataclass
class _Prm:
    budget: float
    mu: float
    b_swap: float
    t_decode: float
    beta: float
    rho: float
    h_age: float
    M: int
    K: int
    mc_samples: int
    seed: int


@dataclass
class _Snap:
    t: float
    stage_agent: list
    stage_preds: list
    prefix_len: list
    stage_samples: list
    task_id: list
    task_arrival: list
    stage_state: list
    stage_served: list
    req_task: list
    req_stage: list
    req_kv: list
    req_dhat: list
    req_redo: list
    req_running: list
    req_credit: list
    resident: list
