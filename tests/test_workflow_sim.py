"""The workflow driver (workflow_sim.py): TOPAS decisions applied to the library.

CPU (plan-only contexts: the page table, no kernels): every task completes
under budgets from roomy to tight, the library never runs out of pages (its
NO_SPACE check holds each chosen state to Eq. 2), no task finishes faster
than its critical path of synthetic service, tight budgets move prefixes and
preempt, and every decision the driver took equals the oracle's on the same
snapshot.  GPU: the same driver with the attention kernels running.
"""
import pytest

from oracle import sched as S
from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build
from paper_2608_25523_gb300.workflow_sim import Timing, WorkflowSim, chain3, dag4

pytestmark = pytest.mark.filterwarnings("ignore")


@pytest.fixture(scope="module", autouse=True)
def lib():
    build()
    return B.load()


def _ctx(pages, flags):
    cfg = B.make_config(num_q_heads=8, num_kv_heads=2, head_dim=64, num_pages=pages, max_agents=8,
                        max_requests=64, max_tokens=1024, max_seq_len=8192, flags=flags)
    return B.Context(cfg)


def _critical_path(wf, tm):
    # longest path of per-stage service T_prefill(input) + T_step * output
    ns = len(wf.stage_agent)
    svc = [tm.t_prefill_token * wf.input_tokens[v] + tm.t_decode_step * wf.output_tokens[v]
           for v in range(ns)]
    best = [0.0] * ns
    for v in range(ns):
        best[v] = svc[v] + max([best[u] for u in wf.stage_preds[v]], default=0.0)
    return max(best)


@pytest.mark.parametrize("pages", [1400, 800, 560])
@pytest.mark.parametrize("make", [chain3, dag4], ids=["chain3", "dag4"])
def test_all_tasks_complete_within_budget(make, pages):
    wf = make()
    ctx = _ctx(pages, B.TPA_FLAG_PLAN_ONLY)
    rec = []
    sim = WorkflowSim(wf, ctx, n_tasks=24, rate=1.5, seed=5, budget_pages=pages, max_tokens=1024,
                      max_requests=64, record=rec)
    res = sim.run()
    assert len(res.jct) == 24
    cp = _critical_path(wf, Timing())
    assert min(res.jct) >= cp - 1e-9
    assert res.decisions == len(rec) > 0
    if pages <= 800:
        assert res.prefix_in > len(wf.prefix_len)     # prefixes moved back in at least once
    # the driver's decisions are the oracle's
    for prm, snap, dec in rec[:40]:
        want = S.decide(S.Snapshot(**vars(snap)), S.Params(**vars(prm)))
        assert dec["running"] == want.running and dec["admitted"] == want.admitted
        assert dec["score"] == want.score
    ctx.close()


@pytest.mark.gpu
def test_driver_on_gpu_kernels():
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    wf = chain3()
    ctx = B.allocate(num_q_heads=8, num_kv_heads=2, head_dim=64, num_pages=800, max_agents=8,
                     max_requests=64, max_tokens=1024, max_seq_len=8192)
    sim = WorkflowSim(wf, ctx, n_tasks=12, rate=1.5, seed=6, budget_pages=800, max_tokens=1024,
                      max_requests=64, device="cuda")
    res = sim.run()
    torch.cuda.synchronize()
    assert len(res.jct) == 12
    assert ctx.device_status() == 0
    assert res.decode_tokens > 0 and res.prefill_tokens > 0
    ctx.close()
