"""Pins of the scheduling oracle (oracle/sched.py) against closed forms.

Each case fixes the answer by hand from the paper's definitions (Sec. IV):
point-mass stage services make Eq. 4 deterministic, so the remaining path
of a chain is the sum of its residuals and that of a fork/join the larger
branch; Eqs. 7-11 are plain arithmetic on the chosen state.  The generator
behind the Monte-Carlo expectation is pinned to SplitMix64's published
output sequence.
"""
import math

import pytest

from oracle import sched as S

pytestmark = pytest.mark.filterwarnings("ignore")


def chain(n_stages, agents=None):
    agents = agents if agents is not None else list(range(n_stages))
    return agents, [[v - 1] if v else [] for v in range(n_stages)]


def snap(stage_agent, preds, prefix_len, samples, tasks, reqs, resident, t=0.0):
    """tasks: list of (id, arrival, states, served); reqs: list of dicts."""
    return S.Snapshot(
        t=t, stage_agent=stage_agent, stage_preds=preds, prefix_len=prefix_len,
        stage_samples=samples,
        task_id=[x[0] for x in tasks], task_arrival=[x[1] for x in tasks],
        stage_state=[list(x[2]) for x in tasks], stage_served=[list(x[3]) for x in tasks],
        req_task=[r["task"] for r in reqs], req_stage=[r["stage"] for r in reqs],
        req_kv=[float(r.get("kv", 100)) for r in reqs], req_dhat=[float(r["dhat"]) for r in reqs],
        req_redo=[float(r.get("redo", 0)) for r in reqs],
        req_running=[bool(r.get("running", False)) for r in reqs],
        req_credit=[float(r.get("credit", 0.0)) for r in reqs], resident=resident)


P0 = S.Params(budget=1e9, mu=4096.0, b_swap=20e9, t_decode=0.02, mc_samples=8)


# ------------------------------------------------------------ generator

def test_splitmix64_published_sequence():
    # SplitMix64 from state 0: the state advances by the golden-ratio
    # increment and each output mixes the new state
    golden = 0x9E3779B97F4A7C15
    outs, x = [], 0
    for _ in range(3):
        outs.append(S.splitmix64(x))
        x = (x + golden) & S.MASK64
    assert outs == [0xE220A8397B1DCDAF, 0x6E789E6AA1B965F4, 0x06C45D188009454F]


def test_draws_are_uniform_over_samples():
    # single-stage task, samples {10, 30}: the mean over many draws tends to 20
    sa, pr = chain(1)
    s = snap(sa, pr, [0], [[10.0, 30.0]], [(7, 0.0, [0], [0.0])], [], [False])
    p = S.Params(budget=1e9, mu=1.0, b_swap=1.0, t_decode=0.0, mc_samples=4096)
    est = S.expected_remaining_path(s, p, 0, {})
    assert abs(est - 20.0) < 0.6   # 6 standard errors of the mean (sd 10)


# ------------------------------------------------------------ Eq. 3, 4, 5

def test_chain_remaining_path_is_sum_of_residuals():
    sa, pr = chain(3)
    # stage 0 done, stage 1 started with 4 s served of 10, stage 2 unstarted (7)
    s = snap(sa, pr, [0, 0, 0], [[5.0], [10.0], [7.0]],
             [(1, 0.0, [2, 1, 0], [5.0, 4.0, 0.0])], [], [False] * 3)
    assert S.expected_remaining_path(s, P0, 0, {}) == pytest.approx(6.0 + 7.0, abs=1e-12)


def test_residual_conditions_on_service_received():
    # Eq. 3 with samples {10, 30}: after 15 s only 30 remains possible -> 15
    sa, pr = chain(1)
    s = snap(sa, pr, [0], [[10.0, 30.0]], [(3, 0.0, [1], [15.0])], [], [False])
    assert S.expected_remaining_path(s, P0, 0, {}) == pytest.approx(15.0, abs=1e-12)
    # beyond every sample: residual 0 (R2)
    s.stage_served[0][0] = 31.0
    assert S.expected_remaining_path(s, P0, 0, {}) == 0.0


def test_chain_progress_is_clipped_reduction():
    sa, pr = chain(2)
    s = snap(sa, pr, [0, 0], [[10.0], [8.0]], [(1, 0.0, [1, 0], [4.0, 0.0])],
             [{"task": 0, "stage": 0, "dhat": 2.5}, {"task": 0, "stage": 0, "dhat": 9.0}],
             [False] * 2)
    # residual of stage 0 is 6: a request worth 2.5 s advances the path 2.5,
    # one worth 9 s only the remaining 6
    assert S.progress(s, P0, 0, []) == pytest.approx(2.5, abs=1e-12)
    assert S.progress(s, P0, 1, []) == pytest.approx(6.0, abs=1e-12)
    # conditional on the first one: 6 - 2.5 = 3.5 remain for the second
    assert S.progress(s, P0, 1, [0]) == pytest.approx(3.5, abs=1e-12)


def fork_join():
    # 0 -> {1, 2} -> 3 ; agents 0, 1, 2, 3
    return [0, 1, 2, 3], [[], [0], [0], [1, 2]]


def test_fork_join_longest_branch_and_slack():
    sa, pr = fork_join()
    # stage 0 done; branch 1 needs 10, branch 2 needs 4; join 3 needs 5
    s = snap(sa, pr, [0] * 4, [[1.0], [10.0], [4.0], [5.0]],
             [(1, 0.0, [2, 0, 0, 0], [1.0, 0, 0, 0])],
             [{"task": 0, "stage": 2, "dhat": 3.0}, {"task": 0, "stage": 1, "dhat": 3.0},
              {"task": 0, "stage": 1, "dhat": 8.0}],
             [False] * 4)
    assert S.expected_remaining_path(s, P0, 0, {}) == pytest.approx(15.0, abs=1e-12)
    # a non-bottleneck branch: no task progress (the paper's fork/join point)
    assert S.progress(s, P0, 0, []) == pytest.approx(0.0, abs=1e-12)
    # the bottleneck branch: full reduction while it stays critical
    assert S.progress(s, P0, 1, []) == pytest.approx(3.0, abs=1e-12)
    # 8 s on branch 1 leaves 2 < 4: the path drops only to the other branch
    assert S.progress(s, P0, 2, []) == pytest.approx(6.0, abs=1e-12)


def test_progress_never_negative_under_common_draws():
    sa, pr = fork_join()
    s = snap(sa, pr, [0] * 4, [[1.0, 3.0], [2.0, 12.0, 5.0], [4.0, 9.0], [5.0, 1.0]],
             [(11, 0.0, [1, 0, 0, 0], [0.5, 0, 0, 0])],
             [{"task": 0, "stage": v, "dhat": d} for v, d in ((0, 0.4), (1, 3.0), (2, 2.0), (3, 1.0))],
             [False] * 4)
    p = S.Params(budget=1e9, mu=1.0, b_swap=1.0, t_decode=0.0, mc_samples=64, seed=5)
    for r in range(4):
        for before in ([], [0], [1, 2]):
            if r not in before:
                assert S.progress(s, p, r, before) >= 0.0


# ------------------------------------------------------------ Eq. 7 - 11

def test_aging_weight():
    sa, pr = chain(1)
    s = snap(sa, pr, [0], [[1.0]], [(1, 2.0, [0], [0.0])], [], [False], t=2.0 + (math.e - 1) * 4.0)
    assert S.aging(s, S.Params(1, 1, 1, 0, rho=1.0, h_age=4.0), 0) == pytest.approx(2.0, abs=1e-12)
    assert S.aging(s, S.Params(1, 1, 1, 0, rho=0.0, h_age=4.0), 0) == 1.0


def test_reuse_counts_fork_join_chain():
    sa, pr = fork_join()
    # task A: stage 0 running -> children 1 and 2 both about to become ready
    # task B: 1 running, 2 unstarted -> the join 3 has two unfinished preds: 0
    # task C: 1 done, 2 running -> the join counts for agent 3
    s = snap(sa, pr, [0] * 4, [[1.0]] * 4,
             [(1, 0, [1, 0, 0, 0], [0] * 4), (2, 0, [2, 1, 0, 0], [0] * 4),
              (3, 0, [2, 2, 1, 0], [0] * 4)], [], [False] * 4)
    assert S.reuse_counts(s) == [0, 1, 1, 1]


def test_score_terms_by_hand():
    # agents 0 (l=1000) and 1 (l=3000); R_t = {0} with a running request of
    # task 0 (y = 50 tokens to redo, credit 0.7); a ready request of task 1 on
    # agent 1.  The state R' = {1}, Q' = {ready}: moves both prefixes, charges
    # one incoming task, preempts the running one.
    sa, pr = [0, 1], [[], [0]]
    s = snap(sa, pr, [1000, 3000], [[4.0], [6.0]],
             [(1, 0.0, [1, 0], [1.0, 0.0]), (2, 0.0, [2, 0], [4.0, 0.0])],
             [{"task": 0, "stage": 0, "dhat": 1.0, "running": True, "redo": 50, "credit": 0.7, "kv": 10},
              {"task": 1, "stage": 1, "dhat": 2.0, "kv": 20}],
             [True, False])
    p = S.Params(budget=1e9, mu=4096.0, b_swap=20e9, t_decode=0.02, beta=0.5, mc_samples=4)
    n_a = S.reuse_counts(s)
    assert n_a == [0, 1]     # task 0's stage 0 runs; its stage 1 (agent 1) is next
    sts = S.greedy_pack(s, p, {1}, n_a)
    st = sts[-1]
    assert st.admitted == (1,) and st.preempted == (0,)
    t_move = 4096.0 / 20e9 * (1000 + 3000)
    assert st.j_move == pytest.approx(t_move * 1, rel=1e-12)
    assert st.j_redo == pytest.approx(0.02 * 50, rel=1e-12)
    assert st.j_revoke == pytest.approx(0.7, rel=1e-12)
    assert st.v_reuse == pytest.approx(0.5 * 1 * 4096.0 * 3000 / 20e9, rel=1e-12)
    assert st.j_admit == pytest.approx(2.0, abs=1e-12)   # a chain residual of 6 > 2
    assert st.score == pytest.approx(st.j_admit - st.j_move - st.j_redo - st.j_revoke + st.v_reuse,
                                     rel=1e-12)


# ------------------------------------------------------------ GreedyPack, Algorithm 1

def _feasible(s, p, st):
    used = sum(s.prefix_len[a] for a in st.agents) + sum(s.req_kv[r] for r in st.running)
    assert used <= p.budget
    assert set(st.agents) == {s.stage_agent[s.req_stage[r]] for r in st.running}
    if p.K:
        assert len(st.admitted) <= p.K and len(st.preempted) <= p.K


def test_shared_prefix_is_paid_once():
    # budget fits one prefix and three requests, not two prefixes
    # (two independent stages; tasks 0-2 have only stage 0 left, task 3 only stage 1)
    sa, pr = [0, 1], [[], []]
    tasks = [(i, 0.0, [0, 2] if i < 3 else [2, 0], [0.0, 0.0]) for i in range(4)]
    reqs = [{"task": 0, "stage": 0, "dhat": 1.0, "kv": 100}, {"task": 1, "stage": 0, "dhat": 1.0, "kv": 100},
            {"task": 2, "stage": 0, "dhat": 1.0, "kv": 100}, {"task": 3, "stage": 1, "dhat": 1.0, "kv": 100}]
    s = snap(sa, pr, [1000, 1000], [[2.0], [2.0]], tasks, reqs, [False, False])
    p = S.Params(budget=1300.0, mu=1.0, b_swap=1e12, t_decode=0.0, mc_samples=2)
    st = S.decide(s, p)
    _feasible(s, p, st)
    assert st.agents == (0,) and st.running == (0, 1, 2)


def test_critical_branch_preferred_over_slack_branch():
    sa, pr = fork_join()
    tasks = [(1, 0.0, [2, 1, 1, 0], [1.0, 0.0, 0.0, 0.0])]
    reqs = [{"task": 0, "stage": 1, "dhat": 3.0, "kv": 100}, {"task": 0, "stage": 2, "dhat": 3.0, "kv": 100}]
    s = snap(sa, pr, [0, 500, 500, 0], [[1.0], [10.0], [4.0], [5.0]], tasks, reqs, [False] * 4)
    # room for one prefix and one request only
    p = S.Params(budget=650.0, mu=1.0, b_swap=1e12, t_decode=0.0, mc_samples=2)
    st = S.decide(s, p)
    _feasible(s, p, st)
    assert st.admitted == (0,) and st.agents == (1,)


def test_admission_cap_and_intermediate_states():
    sa, pr = chain(1)
    tasks = [(i, float(i), [0], [0.0]) for i in range(5)]
    reqs = [{"task": i, "stage": 0, "dhat": 1.0 + i, "kv": 10} for i in range(5)]
    s = snap(sa, pr, [100], [[10.0]], tasks, reqs, [False], t=10.0)
    p = S.Params(budget=1e6, mu=1.0, b_swap=1e12, t_decode=0.0, K=2, mc_samples=2)
    sts = S.greedy_pack(s, p, {0}, S.reuse_counts(s))
    assert [len(x.admitted) for x in sts] == [1, 2]      # every feasible intermediate
    # largest progress per KV first (ties impossible here)
    assert sts[-1].admitted == (4, 3)
    st = S.decide(s, p)
    _feasible(s, p, st)
    assert len(st.admitted) == 2


def test_uncoverable_prefix_set_is_rejected():
    sa, pr = [0, 1], [[], []]
    s = snap(sa, pr, [100, 100], [[1.0], [1.0]], [(0, 0.0, [0, 0], [0.0, 0.0])],
             [{"task": 0, "stage": 0, "dhat": 1.0, "kv": 10}], [False, False])
    assert S.greedy_pack(s, P0, {0, 1}, [0, 0]) == []    # agent 1 has no request
    assert len(S.greedy_pack(s, P0, {0}, [0, 0])) == 1


def test_bounded_search_matches_enumeration_on_easy_pool():
    # five agents, one cheap request each, budget for everything: both the
    # full enumeration (M = 5) and the bounded search (M = 2) admit all
    n = 5
    sa, pr = list(range(n)), [[] for _ in range(n)]
    # task i has only stage i left
    tasks = [(i, 0.0, [0 if v == i else 2 for v in range(n)], [0.0] * n) for i in range(n)]
    reqs = [{"task": i, "stage": i, "dhat": 1.0 + 0.1 * i, "kv": 10} for i in range(n)]
    s = snap(sa, pr, [50] * n, [[5.0]] * n, tasks, reqs, [False] * n)
    for M in (5, 2):
        p = S.Params(budget=1e6, mu=1.0, b_swap=1e12, t_decode=0.0, M=M, mc_samples=2)
        st = S.decide(s, p)
        _feasible(s, p, st)
        assert st.agents == tuple(range(n)) and len(st.admitted) == n


def test_incumbent_kept_when_moving_costs_more():
    # a running request on resident agent 0; a ready request on agent 1 whose
    # prefix is huge to move; the budget allows only one prefix
    sa, pr = [0, 1], [[], []]
    tasks = [(0, 0.0, [1, 2], [0.5, 0.0]), (1, 0.0, [2, 0], [0.0, 0.0])]
    reqs = [{"task": 0, "stage": 0, "dhat": 1.0, "kv": 10, "running": True, "credit": 1.0, "redo": 10},
            {"task": 1, "stage": 1, "dhat": 2.0, "kv": 10}]
    s = snap(sa, pr, [100, 10_000_000], [[2.0], [3.0]], tasks, reqs, [True, False])
    p = S.Params(budget=10_000_050.0, mu=4096.0, b_swap=20e9, t_decode=0.02, mc_samples=2)
    st = S.decide(s, p)
    _feasible(s, p, st)
    # switching would gain 2 s of progress but cost 2.05 s of movement, 0.2 s
    # of redo and the revoked credit 1.0
    assert st.running == (0,) and st.preempted == ()
    # with a cheap prefix the switch pays
    s.prefix_len[1] = 1000
    p.budget = 1050.0
    st = S.decide(s, p)
    _feasible(s, p, st)
    assert st.running == (1,) and st.preempted == (0,)
