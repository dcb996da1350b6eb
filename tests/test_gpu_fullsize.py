"""Parity at the full workload sizes, in the launch configuration bench.py times.

Inputs are drawn on the device by the seeded generator (workloads.tensors_torch);
only the slices the oracle needs are copied to the host, in float64.  Rows
are checked against the fp64 oracle:

  * llama3_8b_decode: the bench's 4-copy context, the steps of copies 0
    and 3, every row;
  * llama3_70b_decode: one step, all 512 requests (every head; so every
    dense tile and every split-KV item of the launch);
  * chunked_prefill: every 512-token chunk round of the 256 new requests,
    the first, the last and one seeded row of every chunk;
  * mixed: reload of 2 evicted prefixes on a side stream (bit-exact), the
    8 prefill chunks (32 rows each, first and last included) and all 256
    Zipf decode requests in one step;
  * the co-residency points of the bench (one 16384-token prefix with 16
    requests of 2048 tokens, two with 8, eight 4096-token prefixes with one
    request each), every row of both copies' steps.

A causal prefill row at suffix position p sees the whole prefix and suffix
positions 0..p, which is the oracle's decode step with suffix[0:p] cached
and suffix[p] as the step's own token.  For the large sets of rows the
oracle's answer is assembled from two oracle.attend calls, one over the
agent's prefix (all of that agent's rows at once) and one over the
request's suffix rows, joined by oracle.lse_merge: the exact merge the
oracle's pins check against single-pass attention (tests/test_oracle_pins.py).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build
from paper_2608_25523_gb300.session import Session
from paper_2608_25523_gb300.workloads import (config, copy_requests, replicate, small_case,
                                               tensors_torch)

from _util import compare

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    build()
    B.load()


def _h(x):
    return x.float().cpu().numpy().astype(np.float64)


_PREFIX = {}


def _prefix_host(w, t, a):
    key = (id(t), a)
    if key not in _PREFIX:
        _PREFIX.clear()
        pk, pv = t.prefix(a, w)
        _PREFIX[key] = (_h(pk), _h(pv))
    return _PREFIX[key]


def _decode_ref(w, t, r, q_row):
    """Oracle decode step of request r (query rows q_row [Hq, d], device)."""
    pk, pv = _prefix_host(w, t, w.req_agent[r])
    n = w.req_ctx[r] + w.req_prefill[r]
    sk, sv = t.suffix(r, w, 0, n)
    nk, nv = t.suffix(r, w, n, n + 1)
    return oracle.decode_step(_h(q_row), pk, pv, _h(sk), _h(sv), _h(nk[0]), _h(nv[0]))


def _refs_by_parts(w, t, items):
    """fp64 oracle output of query rows.  items: (request r, keys k, q_row
    [Hq, d] float64), a row that sees the whole prefix of r's agent and r's
    suffix rows 0..k-1.  Computed as oracle.attend over the prefix (all rows
    of one agent and kv head in one call), oracle.attend over the suffix
    rows, and oracle.lse_merge of the two.  Returns o [n, Hq, d], lse [n, Hq]."""
    hq, hkv, d, G = w.num_q_heads, w.num_kv_heads, w.head_dim, w.group
    n = len(items)
    Q = np.stack([q for _, _, q in items])
    o_pre = np.zeros((n, hq, d))
    l_pre = np.zeros((n, hq))
    by_agent, by_req = {}, {}
    for i, (r, _, _) in enumerate(items):
        by_agent.setdefault(w.req_agent[r], []).append(i)
        by_req.setdefault(r, []).append(i)
    for a, idx in by_agent.items():
        if w.prefix_len[a] == 0:
            continue
        pk, pv = t.prefix(a, w)
        for g in range(hkv):
            rows = Q[idx][:, g * G:(g + 1) * G].reshape(-1, d)
            o, l = oracle.attend(rows, _h(pk[:, g]), _h(pv[:, g]))
            o_pre[idx, g * G:(g + 1) * G] = o.reshape(len(idx), G, d)
            l_pre[idx, g * G:(g + 1) * G] = l.reshape(len(idx), G)
    O = np.empty((n, hq, d))
    L = np.empty((n, hq))
    for r, idx in by_req.items():
        sk, sv = t.suffix(r, w, 0, max(items[i][1] for i in idx))
        SK, SV = _h(sk), _h(sv)
        for i in idx:
            k = items[i][1]
            o_s = np.empty((hq, d))
            l_s = np.empty(hq)
            for g in range(hkv):
                o_s[g * G:(g + 1) * G], l_s[g * G:(g + 1) * G] = oracle.attend(
                    Q[i, g * G:(g + 1) * G], SK[:k, g], SV[:k, g])
            if w.prefix_len[w.req_agent[r]] == 0:
                O[i], L[i] = o_s, l_s
            else:
                O[i], L[i] = oracle.lse_merge([(o_pre[i], l_pre[i]), (o_s, l_s)])
    return O, L


def _check_rows(out, lse, refs, what):
    o_ref = np.stack([o for o, _ in refs])
    l_ref = np.stack([l for _, l in refs])
    return compare(out, lse, o_ref, l_ref, what)


def test_llama3_8b_decode_bench_context():
    base = config(1)
    copies = 4
    w = replicate(base, copies)
    t = tensors_torch(w, "cuda")
    s = Session(w, t, extra_tokens=16)
    dec = w.decode_requests()
    for c in (0, 3):
        pos = copy_requests(w, copies, c)
        ids, q, kn, vn = s.decode_inputs(pos)
        out, lse = s.new_outputs(len(ids))
        s.decode(ids, q, kn, vn, out, lse)
        torch.cuda.synchronize()
        assert s.ctx.device_status() == 0
        assert s.ctx.query(B.Q_LAST_DENSE_ITEMS) > 0      # the cascade ran its tensor-core level
        refs = [_decode_ref(w, t, dec[p], q[k]) for k, p in enumerate(pos)]
        _check_rows(out, lse, refs, f"llama3_8b_decode copy {c}")
    s.ctx.close()


def test_llama3_70b_decode_all_requests():
    w = config(4)
    t = tensors_torch(w, "cuda")
    s = Session(w, t, extra_tokens=16, max_tokens=len(w.decode_requests()))
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    assert s.ctx.device_status() == 0
    assert s.ctx.query(B.Q_LAST_DENSE_ITEMS) > 0 and s.ctx.query(B.Q_LAST_SUFFIX_ITEMS) > 0
    qh = _h(q)
    items = [(r, w.req_ctx[r] + 1, qh[k]) for k, r in enumerate(ids)]
    o_ref, l_ref = _refs_by_parts(w, t, items)
    compare(out, lse, o_ref, l_ref, "llama3_70b_decode, all 512 requests")
    s.ctx.close()


def test_chunked_prefill_all_rounds_every_chunk():
    w = config(2)
    t = tensors_torch(w, "cuda")
    s = Session(w, t, extra_tokens=0)
    rng = np.random.default_rng(303)
    for rnd in range(w.prefill_rounds()):
        chunks, ids, lens, q, k, v = s.prefill_inputs(rnd)
        out, lse = s.new_outputs(sum(lens))
        s.prefill(ids, lens, q, k, v, out, lse)
        torch.cuda.synchronize()
        assert s.ctx.device_status() == 0
        starts = np.cumsum([0] + lens[:-1])
        rows, items = [], []
        for ci, (r, off, c) in enumerate(chunks):
            for i in sorted({0, c - 1, int(rng.integers(0, c))}):
                row = int(starts[ci]) + i
                rows.append(row)
                items.append((r, off + i + 1, _h(q[row])))
        o_ref, l_ref = _refs_by_parts(w, t, items)
        idx = torch.tensor(rows, device="cuda")
        compare(out[idx], lse[idx], o_ref, l_ref, f"chunked_prefill round {rnd}, {len(rows)} rows")
    s.ctx.close()


def test_mixed_step():
    w = config(3)
    t = tensors_torch(w, "cuda")
    s = Session(w, t, extra_tokens=16)
    s.offload_for_reload()
    main = torch.cuda.current_stream()
    side = torch.cuda.Stream()
    done = torch.cuda.Event()
    chunks, pids, plens, pq, pk, pv = s.prefill_inputs(0)
    pout, plse = s.new_outputs(sum(plens))
    dids, dq, dkn, dvn = s.decode_inputs()
    dout, dlse = s.new_outputs(len(dids))
    s.reload(side_stream=side, done_event=done)
    s.prefill(pids, plens, pq, pk, pv, pout, plse, main)
    s.decode(dids, dq, dkn, dvn, dout, dlse, main)
    torch.cuda.synchronize()
    assert s.ctx.device_status() == 0
    # the reloaded prefixes are bit-exact copies of the host ones
    for a in w.reload_agents:
        hk, hv = s.host_prefix[a]
        gk = torch.empty(hk.shape, dtype=hk.dtype, device="cuda")
        gv = torch.empty_like(gk)
        s.ctx.gather(a, False, gk, gv)
        torch.cuda.synchronize()
        assert torch.equal(gk.cpu().view(torch.int16), hk.view(torch.int16))
        assert torch.equal(gv.cpu().view(torch.int16), hv.view(torch.int16))
    rng = np.random.default_rng(202)
    refs = [_decode_ref(w, t, r, dq[k]) for k, r in enumerate(dids)]
    _check_rows(dout, dlse, refs, "mixed decode")
    starts = np.cumsum([0] + plens[:-1])
    rows, items = [], []
    for ci, (r, off, c) in enumerate(chunks):
        pick = {0, c - 1} | {int(x) for x in rng.choice(c, size=min(c, 30), replace=False)}
        for i in sorted(pick):
            row = int(starts[ci]) + i
            rows.append(row)
            items.append((r, off + i + 1, _h(pq[row])))
    o_ref, l_ref = _refs_by_parts(w, t, items)
    idx = torch.tensor(rows, device="cuda")
    compare(pout[idx], plse[idx], o_ref, l_ref, f"mixed prefill, {len(rows)} rows")
    s.ctx.close()


@pytest.mark.parametrize("lp,k", [(16384, 1), (16384, 2), (4096, 8)],
                         ids=["grouped_16384x1", "alternating_16384x2", "prefixes_4096x8"])
def test_coresidency_points(lp, k):
    """The co-residency bench's shapes: a 49152-token budget, 2048-token
    suffixes, k resident prefixes of lp tokens and the batch the budget
    admits, two copies cycled as the bench does."""
    budget, ls = 49152, 2048
    n = (budget - k * lp) // ls
    base = small_case(7, hq=32, hkv=8, d=128, prefix_len=[lp] * k, req_agent=[i % k for i in range(n)],
                      req_ctx=[ls - 1] * n, req_prefill=[0] * n, req_decode=[1] * n)
    w = replicate(base, 2)
    t = tensors_torch(w, "cuda")
    s = Session(w, t, extra_tokens=16)
    for c in (0, 1):
        ids, q, kn, vn = s.decode_inputs(copy_requests(w, 2, c))
        out, lse = s.new_outputs(len(ids))
        s.decode(ids, q, kn, vn, out, lse)
        torch.cuda.synchronize()
        assert s.ctx.device_status() == 0
        qh = _h(q)
        items = [(r, w.req_ctx[r] + 1, qh[j]) for j, r in enumerate(ids)]
        o_ref, l_ref = _refs_by_parts(w, t, items)
        compare(out, lse, o_ref, l_ref, f"coresidency {k} x {lp}, batch {n}, copy {c}")
    s.ctx.close()
