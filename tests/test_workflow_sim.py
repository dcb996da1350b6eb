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


class _Checker:
    """on_launch hook of the GPU driver test.  After a prefix reload and after
    a preempted request's rebuild it checks, at the next launches that use
    them (reading the device after a synchronize):

      * the resident prefix, gathered from its (fragmented) pages, equals the
        host copy bit for bit;
      * each checked request's suffix, gathered from its pages, equals the
        rows the driver appended (its kv_log) bit for bit;
      * the rebuild's prefill chunks and the decode step's outputs match the
        fp64 oracle over the host copies of the same K/V.
    """

    def __init__(self, max_decode=6, max_prefill=4):
        self.seen = 0
        self.reloaded, self.rebuilt = set(), set()
        self.max_decode, self.max_prefill = max_decode, max_prefill
        self.done = {"decode": 0, "prefill": 0, "reload": 0, "rebuild": 0}

    @staticmethod
    def _h(x):
        import numpy as np
        return x.float().cpu().numpy().astype(np.float64)

    def _suffix(self, sim, lib, upto=None):
        import torch
        ks, vs = [], []
        for kind, n in sim.kv_log[lib][:upto]:
            if kind == "pf":
                ks.append(sim.k_pf[:n])
                vs.append(sim.v_pf[:n])
            else:
                ks.append(sim.k_dec[n:n + 1])
                vs.append(sim.v_dec[n:n + 1])
        if not ks:
            e = sim.k_pf[:0]
            return e, e
        return torch.cat(ks), torch.cat(vs)

    def _gathered(self, sim, ident, is_req, length):
        import torch
        k = torch.empty(length, sim.hkv, sim.d, dtype=torch.bfloat16, device=sim.device)
        v = torch.empty_like(k)
        sim.ctx.gather(ident, is_req, k, v)
        torch.cuda.synchronize()
        return k, v

    def _prefix_ok(self, sim, a):
        import torch
        hk, hv = sim.host_kv[a]
        k, v = self._gathered(sim, a, False, hk.shape[0])
        assert torch.equal(k.cpu().view(torch.int16), hk.view(torch.int16)), a
        assert torch.equal(v.cpu().view(torch.int16), hv.view(torch.int16)), a
        return self._h(hk), self._h(hv)

    def __call__(self, sim, kind, info):
        import torch
        import oracle
        from _util import compare
        for e in sim.events[self.seen:]:
            if e[0] == "reload":
                self.reloaded.add(e[1])
            elif e[0] == "rebuild":
                self.rebuilt.add(e[1])
            elif e[0] == "preempt":
                self.rebuilt.discard(e[1])
        self.seen = len(sim.events)
        if kind == "prefill":
            lib, off, c = info
            if lib not in self.rebuilt or self.done["prefill"] >= self.max_prefill:
                return
            torch.cuda.synchronize()
            assert sim.ctx.device_status() == 0
            pk, pv = self._prefix_ok(sim, sim.lib_agent[lib])
            sk, sv = self._suffix(sim, lib, upto=-1)
            assert sk.shape[0] == off
            o_ref, l_ref = oracle.prefill_chunk(self._h(sim.q_pf[:c]), pk, pv, self._h(sk),
                                                self._h(sv), self._h(sim.k_pf[:c]),
                                                self._h(sim.v_pf[:c]))
            compare(sim.o_pf[:c], sim.l_pf[:c], o_ref, l_ref, f"rebuild chunk lib {lib} off {off}")
            self.done["prefill"] += 1
            return
        ids = info
        due = [i for i in ids if i in self.rebuilt or sim.lib_agent[i] in self.reloaded]
        if not due or self.done["decode"] >= self.max_decode:
            return
        torch.cuda.synchronize()
        assert sim.ctx.device_status() == 0
        for j, lib in enumerate(ids):
            if lib not in due:
                continue
            a = sim.lib_agent[lib]
            pk, pv = self._prefix_ok(sim, a)
            sk, sv = self._suffix(sim, lib)
            gk, gv = self._gathered(sim, lib, True, sk.shape[0])
            assert torch.equal(gk.view(torch.int16), sk.view(torch.int16)), lib
            assert torch.equal(gv.view(torch.int16), sv.view(torch.int16)), lib
            o_ref, l_ref = oracle.decode_step(self._h(sim.q_dec[j]), pk, pv, self._h(sk[:-1]),
                                              self._h(sv[:-1]), self._h(sk[-1]), self._h(sv[-1]))
            compare(sim.o_dec[j:j + 1], sim.l_dec[j:j + 1], o_ref[None], l_ref[None],
                    f"decode lib {lib} agent {a}")
            if lib in self.rebuilt:
                self.rebuilt.discard(lib)
                self.done["rebuild"] += 1
            if a in self.reloaded:
                self.reloaded.discard(a)
                self.done["reload"] += 1
        self.done["decode"] += 1


@pytest.mark.gpu
def test_driver_on_gpu_kernels():
    """The driver on the attention kernels: every task completes with device
    status 0, and after prefix reloads into fragmented pages and preemption
    rebuilds by chunked prefill the pages and outputs are checked (_Checker)."""
    import torch
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    wf = chain3()
    ctx = B.allocate(num_q_heads=8, num_kv_heads=2, head_dim=64, num_pages=800, max_agents=8,
                     max_requests=64, max_tokens=1024, max_seq_len=8192, page_order_seed=9)
    chk = _Checker()
    sim = WorkflowSim(wf, ctx, n_tasks=12, rate=1.5, seed=6, budget_pages=800, max_tokens=1024,
                      max_requests=64, device="cuda", on_launch=chk)
    res = sim.run()
    torch.cuda.synchronize()
    assert len(res.jct) == 12
    assert ctx.device_status() == 0
    assert res.decode_tokens > 0 and res.prefill_tokens > 0
    # at least one reloaded prefix and one rebuilt request were checked on a later step
    assert chk.done["reload"] >= 1 and chk.done["rebuild"] >= 1, chk.done
    assert chk.done["prefill"] >= 1, chk.done
    ctx.close()
