"""Parity at the full workload sizes, in the launch configuration bench.py times.

Inputs are drawn on the device by the seeded generator (workloads.tensors_torch);
only the slices the oracle needs are copied to the host, in float64.  Rows
are checked against the fp64 oracle one by one:

  * llama3_8b_decode: the bench's 4-copy context, the steps of copies 0
    and 3, every row;
  * llama3_70b_decode: one step, a seeded sample of 64 of the 512 requests
    (every head);
  * chunked_prefill: every 512-token chunk round of the 256 new requests,
    with a seeded sample of rows per round (first and last row of a chunk
    included);
  * mixed: reload of 2 evicted prefixes on a side stream (bit-exact), the
    8 prefill chunks (sampled rows) and all 256 Zipf decode requests in one
    step.

A causal prefill row at suffix position p sees the whole prefix and suffix
positions 0..p, which is the oracle's decode step with suffix[0:p] cached
and suffix[p] as the step's own token; sampled rows are checked that way.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build
from paper_2608_25523_gb300.session import Session
from paper_2608_25523_gb300.workloads import config, copy_requests, replicate, tensors_torch

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


def _prefill_row_ref(w, t, r, p, q_row):
    """Oracle output of request r's prefill row at suffix position p."""
    pk, pv = _prefix_host(w, t, w.req_agent[r])
    sk, sv = t.suffix(r, w, 0, p)
    nk, nv = t.suffix(r, w, p, p + 1)
    return oracle.decode_step(_h(q_row), pk, pv, _h(sk), _h(sv), _h(nk[0]), _h(nv[0]))


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


def test_llama3_70b_decode_sampled():
    w = config(4)
    t = tensors_torch(w, "cuda")
    s = Session(w, t, extra_tokens=16)
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    assert s.ctx.device_status() == 0
    rng = np.random.default_rng(404)
    pick = sorted(rng.choice(len(ids), size=64, replace=False).tolist())
    refs = [_decode_ref(w, t, ids[k], q[k]) for k in pick]
    idx = torch.tensor(pick, device="cuda")
    _check_rows(out[idx], lse[idx], refs, "llama3_70b_decode sample")
    s.ctx.close()


def test_chunked_prefill_all_rounds_sampled():
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
        rows, refs = [], []
        for ci in sorted(rng.choice(len(chunks), size=min(16, len(chunks)), replace=False).tolist()):
            r, off, c = chunks[ci]
            for i in sorted({0, c - 1, int(rng.integers(0, c))}):
                row = int(starts[ci]) + i
                rows.append(row)
                refs.append(_prefill_row_ref(w, t, r, off + i, q[row]))
        idx = torch.tensor(rows, device="cuda")
        _check_rows(out[idx], lse[idx], refs, f"chunked_prefill round {rnd}")
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
    rows, prefs = [], []
    for ci, (r, off, c) in enumerate(chunks):
        for i in sorted({0, c - 1, int(rng.integers(0, c))}):
            rows.append(int(starts[ci]) + i)
            prefs.append(_prefill_row_ref(w, t, r, off + i, pq[int(starts[ci]) + i]))
    idx = torch.tensor(rows, device="cuda")
    _check_rows(pout[idx], plse[idx], prefs, "mixed prefill sample")
    s.ctx.close()
