"""Seeded synthetic scheduling snapshots (inputs only, no scoring).

Both the oracle and the native scheduler read the same generated snapshot;
nothing here computes any part of the decision.  Workflow shapes follow the
paper's workloads in kind (Sec. V: a chain, a fork/join, a wide fan-out, a
star that returns to a central agent); sizes are small so the plain oracle
stays fast.
"""
from dataclasses import dataclass
from typing import List

import numpy as np

SHAPES = ("chain3", "dag4", "wide6", "star5", "random6")


@dataclass
class Params:
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
class Snapshot:
    t: float
    stage_agent: List[int]
    stage_preds: List[List[int]]
    prefix_len: List[int]
    stage_samples: List[List[float]]
    task_id: List[int]
    task_arrival: List[float]
    stage_state: List[List[int]]
    stage_served: List[List[float]]
    req_task: List[int]
    req_stage: List[int]
    req_kv: List[float]
    req_dhat: List[float]
    req_redo: List[float]
    req_running: List[bool]
    req_credit: List[float]
    resident: List[bool]


def workflow(shape, rng):
    """(stage_agent, stage_preds, n_agents) of a workflow shape."""
    if shape == "chain3":
        return [0, 1, 2], [[], [0], [1]], 3
    if shape == "dag4":
        return [0, 1, 2, 3], [[], [0], [0], [1, 2]], 4
    if shape == "wide6":
        return [0, 1, 2, 3, 4, 5], [[], [0], [0], [0], [0], [1, 2, 3, 4]], 6
    if shape == "star5":
        # a central agent 0 between specialists 1, 2
        return [0, 1, 0, 2, 0], [[], [0], [1], [2], [3]], 3
    # random DAG over 6 stages and 4 agents, predecessors among earlier stages
    preds = [[]]
    for v in range(1, 6):
        k = int(rng.integers(1, min(v, 2) + 1))
        preds.append(sorted(int(x) for x in rng.choice(v, size=k, replace=False)))
    return [int(rng.integers(0, 4)) for _ in range(6)], preds, 4


def snapshot(seed: int, shape: str = None):
    rng = np.random.default_rng(seed)
    shape = shape or SHAPES[seed % len(SHAPES)]
    stage_agent, preds, n_agents = workflow(shape, rng)
    ns = len(stage_agent)
    prefix_len = [int(rng.integers(200, 8000)) for _ in range(n_agents)]
    samples = [[float(np.round(rng.uniform(1.0, 20.0), 3)) for _ in range(int(rng.integers(1, 5)))]
               for _ in range(ns)]
    t = float(np.round(rng.uniform(50.0, 100.0), 3))
    n_tasks = int(rng.integers(1, 6))
    task_id = [int(rng.integers(0, 2**63)) for _ in range(n_tasks)]
    arrival = [float(np.round(rng.uniform(0.0, t), 3)) for _ in range(n_tasks)]
    states, served = [], []
    for _ in range(n_tasks):
        st, sv = [], []
        for v in range(ns):
            ok = all(st[u] == 2 for u in preds[v])
            x = int(rng.choice([2, 1, 0], p=[0.35, 0.35, 0.3])) if ok else 0
            st.append(x)
            sv.append(float(np.round(rng.uniform(0.0, 1.2 * max(samples[v])), 3)) if x == 1 else 0.0)
        states.append(st)
        served.append(sv)
    req_task, req_stage = [], []
    for i in range(n_tasks):
        for v in range(ns):
            ready = states[i][v] == 1 or (states[i][v] == 0 and all(states[i][u] == 2 for u in preds[v]))
            if ready:
                for _ in range(int(rng.integers(1, 3)) if states[i][v] == 1 else 1):
                    req_task.append(i)
                    req_stage.append(v)
    nr = len(req_task)
    req_kv = [float(rng.integers(100, 3000)) for _ in range(nr)]
    req_dhat = [float(np.round(rng.uniform(0.3, 10.0), 3)) for _ in range(nr)]
    running = [bool(rng.random() < 0.4) for _ in range(nr)]
    redo = [float(rng.integers(0, 300)) if running[r] else 0.0 for r in range(nr)]
    credit = [float(np.round(rng.uniform(0.0, 5.0), 3)) if running[r] else 0.0 for r in range(nr)]
    resident = [False] * n_agents
    for r in range(nr):
        if running[r]:
            resident[stage_agent[req_stage[r]]] = True
    if rng.random() < 0.2:
        resident[int(rng.integers(0, n_agents))] = True   # an idle resident prefix
    full = sum(prefix_len) + sum(req_kv)
    params = Params(budget=float(np.round(full * rng.uniform(0.25, 1.1))), mu=4096.0,
                    b_swap=float(rng.choice([2e9, 20e9, 200e9])), t_decode=0.02,
                    beta=float(rng.choice([0.0, 0.5, 2.0])), rho=float(rng.choice([0.0, 0.5])),
                    h_age=10.0, M=int(rng.choice([1, 2, 3, 6])), K=int(rng.choice([0, 0, 1, 2, 3])),
                    mc_samples=int(rng.choice([1, 4, 8])), seed=int(rng.integers(0, 2**63)))
    snap = Snapshot(t, stage_agent, preds, prefix_len, samples, task_id, arrival, states, served,
                    req_task, req_stage, req_kv, req_dhat, redo, running, credit, resident)
    return params, snap
