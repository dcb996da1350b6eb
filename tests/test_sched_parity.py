"""The native scheduler (tpa_sched_decide) against the oracle, decision by decision.

Both evaluate the same seeded snapshots (tests/_sched_cases.py) in IEEE
double with the same operation order, so the selected state, the admission
order, the credits and every score term must agree exactly.  No GPU: the
scheduler is host code in the same library.
"""
import pytest

from oracle import sched as S
from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build

from _sched_cases import SHAPES, snapshot

pytestmark = pytest.mark.filterwarnings("ignore")


@pytest.fixture(scope="module", autouse=True)
def lib():
    build()
    return B.load()


def _oracle(params, snap):
    p = S.Params(**vars(params))
    s = S.Snapshot(**vars(snap))
    return S.decide(s, p)


@pytest.mark.parametrize("seed", range(150))
def test_decision_matches_oracle(seed):
    params, snap = snapshot(seed)
    want = _oracle(params, snap)
    got = B.sched_decide(params, snap)
    assert got["agents"] == want.agents
    assert got["running"] == want.running
    assert got["admitted"] == want.admitted
    assert got["credits"] == want.credits
    assert got["n_preempted"] == len(want.preempted)
    for k in ("score", "j_admit", "j_move", "j_redo", "j_revoke", "v_reuse"):
        assert got[k] == getattr(want, k), k


@pytest.mark.parametrize("shape", SHAPES)
def test_selected_state_is_feasible(shape):
    for seed in range(20):
        params, snap = snapshot(1000 + seed, shape)
        got = B.sched_decide(params, snap)
        agent = [snap.stage_agent[v] for v in snap.req_stage]
        used = sum(snap.prefix_len[a] for a in got["agents"]) + sum(snap.req_kv[r] for r in got["running"])
        incumbent = (got["agents"] == tuple(a for a, x in enumerate(snap.resident) if x) and
                     got["running"] == tuple(r for r, x in enumerate(snap.req_running) if x))
        if incumbent:
            continue    # Algorithm 1 may keep the current state as it is
        assert used <= params.budget
        assert set(got["agents"]) == {agent[r] for r in got["running"]}
        if params.K:
            assert len(got["admitted"]) <= params.K and got["n_preempted"] <= params.K
        assert all(not snap.req_running[r] for r in got["admitted"])


def test_invalid_snapshots_are_refused():
    params, snap = snapshot(3)
    bad = snapshot(3)[1]
    bad.stage_preds = [[1]] + bad.stage_preds[1:]     # a predecessor after its stage
    with pytest.raises(B.TpaError) as e:
        B.sched_decide(params, bad)
    assert e.value.code == B.TPA_ERR_INVALID_ARG
    bad = snapshot(3)[1]
    bad.stage_samples = [[]] + bad.stage_samples[1:]  # a stage without samples
    with pytest.raises(B.TpaError):
        B.sched_decide(params, bad)
    params.mc_samples = 0
    with pytest.raises(B.TpaError):
        B.sched_decide(params, snap)
