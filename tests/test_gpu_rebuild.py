"""Preemption and rebuild of a request's suffix by chunked prefill (Sec. IV-B, Eq. 8).

The paper charges a preempted request T_decode * y_r for redoing its y_r
decode tokens one step at a time; the library can instead drop the
request's decode KV (tpa_request_truncate) and rebuild those tokens with
tpa_prefill_chunk.  On a permuted (fragmented) pool, three requests:

  1. prefill their inputs in one chunk round;
  2. take y = 50 decode steps, each appending one token;
  3. are preempted: truncated part-way into a page (request 0), to an empty
     suffix (request 1: the whole suffix, input included, is rebuilt) and
     exactly onto a page boundary (request 2);
  4. rebuild the dropped tokens in two chunk rounds of uneven lengths;
  5. take one more decode step.

Every chunk output and every decode step is compared with the fp64 oracle,
and after the rebuild each suffix gathered from its pages must equal the
generator's rows bit for bit.  The same token positions give the same keys
whichever call wrote them, so the rebuilt state is the state before the
preemption.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build
from paper_2608_25523_gb300.session import Session, to_device
from paper_2608_25523_gb300.workloads import small_case, tensors_numpy

from _util import compare

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    build()
    B.load()


def _bits(x):
    return x.contiguous().view(torch.int16)


INPUT = [64, 40, 100]      # input tokens prefilled first
Y = 50                     # decode steps before the preemption
KEEP = [64 + 13, 0, 144]   # suffix length kept by the preemption (77: mid-page; 144 = 9 pages)
ROUNDS = [[20, 40, 3], [17, 50, 3]]   # rebuild chunk lengths per round and request


@pytest.mark.parametrize("rows", [256, 128], ids=["pairs", "single"])
def test_preempted_suffix_rebuilt_by_chunked_prefill(rows):
    n = len(INPUT)
    total = [i + Y for i in INPUT]
    assert all(KEEP[r] + sum(c[r] for c in ROUNDS) == total[r] for r in range(n))
    # suffix rows of request r: input, the Y decoded tokens, then one more decode token;
    # q_prefill rows 0..total-1 are the queries at those positions
    w = small_case(61, hq=8, hkv=2, d=128, prefix_len=[333, 129], req_agent=[0, 1, 0],
                   req_ctx=[0] * n, req_prefill=total, req_decode=[1] * n, chunk=64, permute=True)
    t = tensors_numpy(w)
    s = Session(w, to_device(t, "cuda"))
    s.ctx.set_option(B.OPT_PREFILL_TILE_ROWS, rows)
    td = s.t
    ids = list(range(n))

    def q_rows(r, lo, hi):
        o = td.qpf_off[r]
        return td.q_prefill[o + lo:o + hi]

    def run_chunks(offsets, lens, what):
        q = torch.cat([q_rows(r, offsets[r], offsets[r] + lens[r]) for r in ids if lens[r]])
        kv = [td.suffix(r, w, offsets[r], offsets[r] + lens[r]) for r in ids if lens[r]]
        rq = [r for r in ids if lens[r]]
        out, lse = s.new_outputs(sum(lens))
        s.prefill(rq, [lens[r] for r in rq], q, torch.cat([k for k, _ in kv]),
                  torch.cat([v for _, v in kv]), out, lse)
        torch.cuda.synchronize()
        assert s.ctx.device_status() == 0
        row = 0
        for r in rq:
            pk, pv = t.prefix(w.req_agent[r], w)
            sk, sv = t.suffix(r, w, 0, offsets[r])
            nk, nv = t.suffix(r, w, offsets[r], offsets[r] + lens[r])
            qo = t.qpf_off[r] + offsets[r]
            o_ref, l_ref = oracle.prefill_chunk(t.q_prefill[qo:qo + lens[r]], pk, pv, sk, sv, nk, nv)
            compare(out[row:row + lens[r]], lse[row:row + lens[r]], o_ref, l_ref,
                    f"{what} r{r} off {offsets[r]}")
            row += lens[r]

    def decode_at(pos, q, what):
        """One decode step of every request, appending suffix row pos[r]."""
        kn = torch.stack([td.suffix(r, w, pos[r], pos[r] + 1)[0][0] for r in ids])
        vn = torch.stack([td.suffix(r, w, pos[r], pos[r] + 1)[1][0] for r in ids])
        out, lse = s.new_outputs(n)
        s.decode(ids, q, kn, vn, out, lse)
        torch.cuda.synchronize()
        assert s.ctx.device_status() == 0
        refs = []
        for r in ids:
            pk, pv = t.prefix(w.req_agent[r], w)
            sk, sv = t.suffix(r, w, 0, pos[r])
            nk, nv = t.suffix(r, w, pos[r], pos[r] + 1)
            qh = q[r].float().cpu().numpy()
            refs.append(oracle.decode_step(qh, pk, pv, sk, sv, nk[0], nv[0]))
        compare(out, lse, np.stack([o for o, _ in refs]), np.stack([l for _, l in refs]), what)

    # 1. the inputs, one chunk round
    run_chunks([0] * n, INPUT, "input")
    # 2. Y decode steps; the query of position p is q_prefill row p
    for j in range(Y):
        pos = [INPUT[r] + j for r in ids]
        decode_at(pos, torch.stack([q_rows(r, pos[r], pos[r] + 1)[0] for r in ids]), f"decode {j}")
    assert [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids] == total
    # 3. preemption drops the decode KV (and, for request 1, the input's too)
    free0 = s.ctx.query(B.Q_FREE_PAGES)
    s.ctx.request_truncate(ids, KEEP)
    assert [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids] == KEEP
    freed = sum(-(-a // 16) - -(-b // 16) for a, b in zip(total, KEEP))
    assert s.ctx.query(B.Q_FREE_PAGES) == free0 + freed
    # 4. rebuild by chunked prefill in two rounds of uneven chunks
    off = list(KEEP)
    for rnd, lens in enumerate(ROUNDS):
        run_chunks(off, lens, f"rebuild round {rnd}")
        off = [o + c for o, c in zip(off, lens)]
    assert off == total
    for r in ids:
        k = torch.empty(total[r], 2, 128, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        s.ctx.gather(r, True, k, v)
        sk, sv = td.suffix(r, w, 0, total[r])
        torch.cuda.synchronize()
        assert torch.equal(_bits(k), _bits(sk)) and torch.equal(_bits(v), _bits(sv)), r
    # 5. the next decode step sees the rebuilt suffix
    decode_at(total, td.q_decode, "decode after the rebuild")
    s.ctx.close()
