"""GPU parity of the CUDA path against the fp64 oracle, through the C ABI.

Small workloads span several tiles and ragged tails: prefixes of 0, 1, 15,
16, 17, 127, 128, 129 and 1000 tokens; cached suffixes of 0..300 tokens;
more decode requests per agent than one 128-row tile holds; head_dim 64
and 128; GQA groups 4 and 8; sequential and permuted (fragmented) pools;
a "sharp" variant with Q scaled by 8 so the softmax is peaked.  Page-table
work (append, prefix write, reload, offload, gather) must be bit-exact.
"""
import zlib

import numpy as np
import pytest
import torch

import oracle
from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build
from paper_2608_25523_gb300.session import Session, to_device
from paper_2608_25523_gb300.workloads import bf16_round, config, sharp, small_case, tensors_numpy

from _util import compare, stack_decode_ref

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    build()
    B.load()


def _bits(x):
    return x.contiguous().view(torch.int16)


def _session(w, **kw):
    t = tensors_numpy(w)
    return t, Session(w, to_device(t, "cuda"), **kw)


def _check_status(s):
    assert s.ctx.device_status() == 0


DECODE_CASES = {
    # name: (hq, hkv, d, prefix lens, request agents, cached suffix lens, permuted)
    "d128_g4_mixed": (8, 2, 128, [0, 1, 129, 1000], [0, 1, 2, 3, 1, 2, 3, 3],
                      [5, 0, 15, 16, 17, 300, 64, 1], False),
    "d64_g8_edges": (16, 2, 64, [15, 16, 17, 127, 128], [0, 1, 2, 3, 4, 0, 4],
                     [1, 16, 31, 32, 33, 200, 7], True),
    "d128_g8_many": (32, 4, 128, [300], [0] * 20, list(range(0, 200, 10)), False),
    "d64_g4_two_tiles": (8, 2, 64, [257, 40], [0] * 40 + [1] * 3,
                         [(7 * i) % 90 for i in range(43)], True),
}


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
@pytest.mark.parametrize("name", sorted(DECODE_CASES))
def test_decode_small(name, mode):
    hq, hkv, d, plen, agents, ctx, perm = DECODE_CASES[name]
    w = small_case(zlib.crc32(name.encode()) % 1000, hq=hq, hkv=hkv, d=d, prefix_len=plen, req_agent=agents,
                   req_ctx=ctx, req_prefill=[0] * len(agents), req_decode=[1] * len(agents),
                   permute=perm)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    ref = oracle.workload_decode(w, t)
    o_ref, l_ref = stack_decode_ref(ref, range(len(ids)))
    compare(out, lse, o_ref, l_ref, f"{name}/{mode}")


@pytest.mark.parametrize("splits", [(1, 16), (3, 48), (0, 0)])
def test_decode_split_choices_agree(splits):
    """Any split of the prefix (dense level) and suffix (split-KV level)
    gives the oracle's result: the LSE merge is exact."""
    w = small_case(7, hq=8, hkv=2, d=128, prefix_len=[700, 33], req_agent=[0, 0, 1, 0],
                   req_ctx=[100, 257, 3, 31], req_prefill=[0] * 4, req_decode=[1] * 4)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_PREFIX_SPLITS, splits[0])
    s.ctx.set_option(B.OPT_SUFFIX_SPLIT_KEYS, splits[1])
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(out, lse, o_ref, l_ref, f"splits {splits}")


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
def test_decode_at_capacity_limits(mode):
    """A batch of exactly max_tokens requests whose suffixes reach
    max_seq_len with the step's token, under a split budget (max_splits 4)
    so small that the planner must widen the suffix items: every row matches
    the oracle.  The next step would pass max_seq_len and is refused with
    CAPACITY, with the tables left as they were."""
    n = 48
    ctx_lens = [1599 if i % 5 == 0 else (37 * i) % 1599 for i in range(n)]
    w = small_case(61, hq=8, hkv=2, d=128, prefix_len=[100, 1], req_agent=[i % 2 for i in range(n)],
                   req_ctx=ctx_lens, req_prefill=[0] * n, req_decode=[1] * n, permute=True)
    t = tensors_numpy(w)
    s = Session(w, to_device(t, "cuda"), extra_tokens=0, max_splits=4, max_tokens=n)
    s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    ids, q, kn, vn = s.decode_inputs()
    assert len(ids) == n
    out, lse = s.new_outputs(n)
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(n))
    compare(out, lse, o_ref, l_ref, f"capacity limits/{mode}")
    lens = [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids]
    assert max(lens) == 1600
    free = s.ctx.query(B.Q_FREE_PAGES)
    with pytest.raises(B.TpaError) as e:
        s.decode(ids, q, kn, vn, out, lse)
    assert e.value.code == B.TPA_ERR_CAPACITY
    assert [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids] == lens
    assert s.ctx.query(B.Q_FREE_PAGES) == free
    torch.cuda.synchronize()
    _check_status(s)


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
def test_decode_suffix_scores_far_above_the_prefix(mode):
    """Suffix keys 24x larger than the prefix keys: the partials of one
    token have LSEs tens of units apart, so the exact merge must weight the
    prefix partials down to (almost) nothing.  Must match the oracle."""
    w = small_case(43, hq=8, hkv=2, d=128, prefix_len=[700, 129], req_agent=[0, 1, 0, 1, 0],
                   req_ctx=[40, 300, 1, 17, 600], req_prefill=[0] * 5, req_decode=[1] * 5,
                   permute=True)
    t = tensors_numpy(w)
    t.suffix_k = bf16_round(t.suffix_k * np.float32(24.0))
    s = Session(w, to_device(t, "cuda"))
    s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(out, lse, o_ref, l_ref, "suffix scores far above the prefix")


def test_decode_sharp_softmax():
    w = sharp(small_case(11, hq=8, hkv=2, d=128, prefix_len=[513, 64], req_agent=[0, 1, 0, 1, 0],
                         req_ctx=[40, 2, 129, 300, 0], req_prefill=[0] * 5, req_decode=[1] * 5))
    t, s = _session(w)
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(out, lse, o_ref, l_ref, "sharp")


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
def test_decode_steps_back_to_back(mode):
    """12 decode steps issued with no host synchronisation between them, each
    appending one token per request and writing its own outputs: the steps
    run as a chain of programmatic dependents (each step's split-KV warps
    resolve their first item from the plan before waiting for the previous
    kernel) and cycle the 4-slot plan ring three times.  Every step must
    match the oracle."""
    steps = 12
    n = 6
    w = small_case(83, hq=8, hkv=2, d=128, prefix_len=[700, 129, 0], req_agent=[0, 1, 0, 2, 1, 0],
                   req_ctx=[0] * n, req_prefill=[40, 300, 17, 260, 1, 120],
                   req_decode=[1] * n, chunk=512, permute=True)
    t = tensors_numpy(w)
    s = Session(w, to_device(t, "cuda"))
    s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    td = s.t
    ids = list(range(n))
    # prefill the inputs except their last `steps` tokens, which the decode steps append
    base = [w.req_prefill[r] - steps if w.req_prefill[r] > steps else 0 for r in ids]
    pre = [r for r in ids if base[r] > 0]
    if pre:
        q = torch.cat([td.q_prefill[td.qpf_off[r]:td.qpf_off[r] + base[r]] for r in pre])
        kv = [td.suffix(r, w, 0, base[r]) for r in pre]
        out, lse = s.new_outputs(sum(base[r] for r in pre))
        s.prefill(pre, [base[r] for r in pre], q, torch.cat([k for k, _ in kv]),
                  torch.cat([v for _, v in kv]), out, lse)
    live = [r for r in ids if w.req_prefill[r] >= steps]   # requests with a token for every step
    results = []
    for j in range(steps):
        pos = [base[r] + j for r in live]
        q = torch.stack([td.q_prefill[td.qpf_off[r] + p] for r, p in zip(live, pos)])
        kn = torch.stack([td.suffix(r, w, p, p + 1)[0][0] for r, p in zip(live, pos)])
        vn = torch.stack([td.suffix(r, w, p, p + 1)[1][0] for r, p in zip(live, pos)])
        out, lse = s.new_outputs(len(live))
        s.decode(live, q, kn, vn, out, lse)
        results.append((pos, q, out, lse))
    torch.cuda.synchronize()
    _check_status(s)
    for j, (pos, q, out, lse) in enumerate(results):
        refs = []
        for r, p, qr in zip(live, pos, q):
            pk, pv = t.prefix(w.req_agent[r], w)
            sk, sv = t.suffix(r, w, 0, p)
            nk, nv = t.suffix(r, w, p, p + 1)
            refs.append(oracle.decode_step(qr.float().cpu().numpy(), pk, pv, sk, sv, nk[0], nv[0]))
        compare(out, lse, np.stack([o for o, _ in refs]), np.stack([l for _, l in refs]),
                f"back-to-back step {j}")


def test_cascade_equals_flat():
    """The two-level cascade and the flat split-KV path read the same keys
    in different groupings; they agree to fp32 reordering noise."""
    w = small_case(13, hq=32, hkv=8, d=128, prefix_len=[1024, 300],
                   req_agent=[0] * 12 + [1] * 4, req_ctx=[17 * i + 1 for i in range(16)],
                   req_prefill=[0] * 16, req_decode=[1] * 16)
    outs = []
    for mode in (0, 1):
        t, s = _session(w)
        s.ctx.set_option(B.OPT_DECODE_MODE, mode)
        ids, q, kn, vn = s.decode_inputs()
        out, lse = s.new_outputs(len(ids))
        s.decode(ids, q, kn, vn, out, lse)
        torch.cuda.synchronize()
        _check_status(s)
        outs.append((out.float().cpu(), lse.cpu()))
    assert (outs[0][1] - outs[1][1]).abs().max().item() <= 1e-4
    assert (outs[0][0] - outs[1][0]).abs().max().item() <= 8e-3


PREFILL_CASES = {
    "d128_g4": (8, 2, 128, [0, 129, 1000], [0, 1, 2, 1, 2], [1, 31, 200, 64, 130], 64),
    "d64_g8": (16, 2, 64, [17, 128], [0, 1, 1], [33, 15, 150], 48),
    "d128_g8": (32, 4, 128, [250], [0, 0], [100, 17], 32),
    # chunks of 100 tokens: pairs whose second tile holds 4, 5 and 18 tokens
    "d128_g4_ragged_pairs": (8, 2, 128, [300, 0], [0, 1, 0], [100, 37, 250], 100),
}


@pytest.mark.parametrize("rows", [256, 128], ids=["pairs", "single"])
@pytest.mark.parametrize("name", sorted(PREFILL_CASES))
def test_prefill_chunks(name, rows):
    hq, hkv, d, plen, agents, pf, chunk = PREFILL_CASES[name]
    n = len(agents)
    w = small_case(zlib.crc32(name.encode()) % 1000, hq=hq, hkv=hkv, d=d, prefix_len=plen, req_agent=agents,
                   req_ctx=[0] * n, req_prefill=pf, req_decode=[0] * n, chunk=chunk,
                   permute=True)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_PREFILL_TILE_ROWS, rows)
    for rnd in range(w.prefill_rounds()):
        chunks, ids, lens, q, k, v = s.prefill_inputs(rnd)
        out, lse = s.new_outputs(sum(lens))
        s.prefill(ids, lens, q, k, v, out, lse)
        torch.cuda.synchronize()
        _check_status(s)
        row = 0
        for r, off, c in chunks:
            o_ref, l_ref = oracle.workload_prefill_chunk(w, t, r, off, c)
            compare(out[row:row + c], lse[row:row + c], o_ref, l_ref, f"{name} r{r} off{off}")
            row += c


@pytest.mark.parametrize("rows", [256, 128], ids=["pairs", "single"])
def test_prefill_scores_rising_far_above_the_first_tile(rows):
    """Suffix keys 24x larger than the prefix keys: the scores of the
    suffix tiles lie far above the prefix tiles' row max, so the online
    softmax's reference max jumps by tens of log2 units mid-row and O and l
    are rescaled.  The outputs must still match the oracle."""
    w = small_case(41, hq=8, hkv=2, d=128, prefix_len=[300, 150], req_agent=[0, 1, 0],
                   req_ctx=[0] * 3, req_prefill=[200, 130, 64], req_decode=[0] * 3, chunk=256,
                   permute=True)
    t = tensors_numpy(w)
    t.suffix_k = bf16_round(t.suffix_k * np.float32(24.0))
    s = Session(w, to_device(t, "cuda"))
    s.ctx.set_option(B.OPT_PREFILL_TILE_ROWS, rows)
    chunks, ids, lens, q, k, v = s.prefill_inputs(0)
    out, lse = s.new_outputs(sum(lens))
    s.prefill(ids, lens, q, k, v, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    row = 0
    for r, off, c in chunks:
        o_ref, l_ref = oracle.workload_prefill_chunk(w, t, r, off, c)
        compare(out[row:row + c], lse[row:row + c], o_ref, l_ref, f"r{r} off{off}")
        row += c


@pytest.mark.parametrize("rows", [256, 128], ids=["pairs", "single"])
def test_prefill_at_capacity_limits(rows):
    """One call whose chunks total exactly max_tokens rows, one of them
    ending exactly at max_seq_len (cached suffixes before the chunks): every
    row matches the oracle.  One more token for that request is refused
    with CAPACITY, with the tables left as they were."""
    w = small_case(67, hq=8, hkv=2, d=128, prefix_len=[150, 17], req_agent=[0, 1, 0, 1],
                   req_ctx=[0, 40, 100, 7], req_prefill=[200, 150, 90, 200], req_decode=[0] * 4,
                   chunk=256, permute=True)
    t = tensors_numpy(w)
    s = Session(w, to_device(t, "cuda"), extra_tokens=0, max_tokens=640)
    s.ctx.set_option(B.OPT_PREFILL_TILE_ROWS, rows)
    assert w.prefill_rounds() == 1
    chunks, ids, lens, q, k, v = s.prefill_inputs(0)
    assert sum(lens) == 640
    out, lse = s.new_outputs(640)
    s.prefill(ids, lens, q, k, v, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    row = 0
    for r, off, c in chunks:
        o_ref, l_ref = oracle.workload_prefill_chunk(w, t, r, off, c)
        compare(out[row:row + c], lse[row:row + c], o_ref, l_ref, f"capacity r{r} off{off}")
        row += c
    assert s.ctx.query(B.Q_SUFFIX_LEN, 3) == 207
    free = s.ctx.query(B.Q_FREE_PAGES)
    with pytest.raises(B.TpaError) as e:
        s.prefill([3], [1], q[:1], k[:1], v[:1], out[:1], lse[:1])
    assert e.value.code == B.TPA_ERR_CAPACITY
    assert s.ctx.query(B.Q_SUFFIX_LEN, 3) == 207
    assert s.ctx.query(B.Q_FREE_PAGES) == free
    torch.cuda.synchronize()
    _check_status(s)


def test_tiny_workload_prefill_then_decode():
    """The tiny workload: 1 agent, 256-token prefix, 4 requests prefill a
    64-token suffix in one chunk, then take one decode step."""
    w = config(0)
    t, s = _session(w)
    chunks, ids, lens, q, k, v = s.prefill_inputs(0)
    out, lse = s.new_outputs(sum(lens))
    s.prefill(ids, lens, q, k, v, out, lse)
    torch.cuda.synchronize()
    row = 0
    for r, off, c in chunks:
        o_ref, l_ref = oracle.workload_prefill_chunk(w, t, r, off, c)
        compare(out[row:row + c], lse[row:row + c], o_ref, l_ref, f"tiny prefill r{r}")
        row += c
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(out, lse, o_ref, l_ref, "tiny decode")


# ---------------------------------------------------------------- pages --

@pytest.mark.parametrize("perm", [False, True], ids=["sequential", "permuted"])
def test_page_roundtrip_bit_exact(perm):
    w = small_case(21, hq=8, hkv=2, d=128, prefix_len=[1, 16, 17, 300, 0],
                   req_agent=[0, 1, 2, 3, 4, 3], req_ctx=[0, 1, 15, 16, 33, 250],
                   req_prefill=[0] * 6, req_decode=[1] * 6, permute=perm)
    t, s = _session(w)
    td = s.t
    for a in range(w.num_agents):
        L = w.prefix_len[a]
        if L == 0:
            continue
        k = torch.empty(L, w.num_kv_heads, w.head_dim, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        s.ctx.gather(a, False, k, v)
        pk, pv = td.prefix(a, w)
        torch.cuda.synchronize()
        assert torch.equal(_bits(k), _bits(pk)) and torch.equal(_bits(v), _bits(pv))
    # a decode step appends one token per request; gathering must show it
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    for r in range(w.num_requests):
        L = w.req_ctx[r] + 1
        k = torch.empty(L, w.num_kv_heads, w.head_dim, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        s.ctx.gather(r, True, k, v)
        sk, sv = td.suffix(r, w, 0, L)
        torch.cuda.synchronize()
        assert torch.equal(_bits(k), _bits(sk)) and torch.equal(_bits(v), _bits(sv)), r
    _check_status(s)


@pytest.mark.parametrize("staged", [1, 0], ids=["staged", "direct"])
def test_offload_reload_bit_exact_on_side_stream(staged):
    """Both movement modes: copy engine through the staging area (default)
    and the page kernel on the mapped host arrays."""
    w = small_case(23, hq=8, hkv=2, d=128, prefix_len=[333, 48], req_agent=[0, 1, 0],
                   req_ctx=[20, 5, 77], req_prefill=[0] * 3, req_decode=[1] * 3, permute=True)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_MOVEMENT_STAGED, staged)
    L = w.prefix_len[0]
    hk = torch.empty(L, 2, 128, dtype=torch.bfloat16, pin_memory=True)
    hv = torch.empty_like(hk, pin_memory=True)
    side = torch.cuda.Stream()
    ev = torch.cuda.Event()
    s.ctx.prefix_offload(0, hk, hv, side, ev)
    ev.synchronize()
    pk, pv = s.t.prefix(0, w)
    assert torch.equal(_bits(hk), _bits(pk.cpu())) and torch.equal(_bits(hv), _bits(pv.cpu()))
    assert s.ctx.query(B.Q_PREFIX_RESIDENT, 0) == 0
    ev2 = torch.cuda.Event()
    s.ctx.prefix_reload(0, hk, hv, side, ev2)
    # decode on the default stream must see the reloaded prefix without a host sync
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(out, lse, o_ref, l_ref, "after reload")
    k = torch.empty(L, 2, 128, dtype=torch.bfloat16, device="cuda")
    v = torch.empty_like(k)
    s.ctx.gather(0, False, k, v)
    torch.cuda.synchronize()
    assert torch.equal(_bits(k), _bits(pk)) and torch.equal(_bits(v), _bits(pv))


def test_decode_with_pinned_host_io_is_bit_identical():
    """q, k_new, v_new, out, lse in pinned host memory: the kernels read and
    write them over the host link, and the outputs and the appended pages
    equal those of the same step with device buffers bit for bit."""
    w = small_case(37, hq=8, hkv=2, d=128, prefix_len=[300, 17], req_agent=[0, 1, 0, 1, 0],
                   req_ctx=[10, 200, 0, 33, 97], req_prefill=[0] * 5, req_decode=[1] * 5,
                   permute=True)
    t, s = _session(w)
    ids, q, kn, vn = s.decode_inputs()
    lens = [w.req_ctx[r] for r in ids]
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    k_dev = torch.empty(w.req_ctx[ids[0]] + 1, 2, 128, dtype=torch.bfloat16, device="cuda")
    v_dev = torch.empty_like(k_dev)
    s.ctx.gather(ids[0], True, k_dev, v_dev)
    s.ctx.request_truncate(ids, lens)
    pin = lambda x: x.cpu().pin_memory()
    hq, hk, hv = pin(q), pin(kn), pin(vn)
    ho = torch.empty(out.shape, dtype=out.dtype, pin_memory=True)
    hl = torch.empty(lse.shape, dtype=lse.dtype, pin_memory=True)
    s.decode(ids, hq, hk, hv, ho, hl)
    k2 = torch.empty_like(k_dev)
    v2 = torch.empty_like(v_dev)
    s.ctx.gather(ids[0], True, k2, v2)
    torch.cuda.synchronize()
    _check_status(s)
    assert torch.equal(_bits(ho), _bits(out.cpu())) and torch.equal(hl, lse.cpu())
    assert torch.equal(_bits(k2), _bits(k_dev)) and torch.equal(_bits(v2), _bits(v_dev))
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(ho, hl, o_ref, l_ref, "pinned host io")


@pytest.mark.parametrize("rows", [256, 128], ids=["pairs", "single"])
def test_prefill_with_pinned_host_io_is_bit_identical(rows):
    """A prefill chunk round with q, k_new, v_new, out, lse in pinned host
    memory gives the same bits as with device buffers."""
    w = small_case(47, hq=8, hkv=2, d=128, prefix_len=[300, 17], req_agent=[0, 1, 0],
                   req_ctx=[0] * 3, req_prefill=[100, 64, 37], req_decode=[0] * 3, chunk=128,
                   permute=True)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_PREFILL_TILE_ROWS, rows)
    chunks, ids, lens, q, k, v = s.prefill_inputs(0)
    out, lse = s.new_outputs(sum(lens))
    s.prefill(ids, lens, q, k, v, out, lse)
    s.ctx.request_truncate(ids, [0] * len(ids))
    pin = lambda x: x.cpu().pin_memory()
    hq, hk, hv = pin(q), pin(k), pin(v)
    ho = torch.empty(out.shape, dtype=out.dtype, pin_memory=True)
    hl = torch.empty(lse.shape, dtype=lse.dtype, pin_memory=True)
    s.prefill(ids, lens, hq, hk, hv, ho, hl)
    torch.cuda.synchronize()
    _check_status(s)
    assert torch.equal(_bits(ho), _bits(out.cpu())) and torch.equal(hl, lse.cpu())


def test_concurrent_reloads_on_two_streams_share_the_staging_area():
    """Two prefixes reloaded at once on two side streams go through the one
    staging area of the workspace; the second waits for the first on the
    device.  Both land bit-exact and a decode over them matches the oracle."""
    w = small_case(31, hq=8, hkv=2, d=128, prefix_len=[500, 333, 17], req_agent=[0, 1, 2, 0, 1],
                   req_ctx=[20, 5, 77, 3, 40], req_prefill=[0] * 5, req_decode=[1] * 5, permute=True)
    t, s = _session(w)
    hosts = {}
    side = [torch.cuda.Stream(), torch.cuda.Stream()]
    for a in (0, 1):
        L = w.prefix_len[a]
        hk = torch.empty(L, 2, 128, dtype=torch.bfloat16, pin_memory=True)
        hv = torch.empty_like(hk, pin_memory=True)
        ev = torch.cuda.Event()
        s.ctx.prefix_offload(a, hk, hv, side[a], ev)
        ev.synchronize()
        hosts[a] = (hk, hv)
    with torch.cuda.stream(side[0]):
        torch.cuda._sleep(5_000_000)   # the first reload is still in flight when the second is issued
    for a in (0, 1):
        s.ctx.prefix_reload(a, hosts[a][0], hosts[a][1], side[a], None)
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(out, lse, o_ref, l_ref, "after two reloads")
    for a in (0, 1):
        L = w.prefix_len[a]
        k = torch.empty(L, 2, 128, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        s.ctx.gather(a, False, k, v)
        pk, pv = s.t.prefix(a, w)
        torch.cuda.synchronize()
        assert torch.equal(_bits(k), _bits(pk)) and torch.equal(_bits(v), _bits(pv)), a


@pytest.mark.parametrize("only_reloading", [False, True], ids=["mixed_agents", "only_reloading"])
@pytest.mark.parametrize("rows", [256, 128], ids=["pairs", "single"])
def test_prefill_runs_ready_chunks_before_a_pending_reload(rows, only_reloading):
    """A prefill call whose chunks include an agent with a reload still in
    flight on a side stream: the other agents' items run in a first launch,
    the reloading agent's in a second one after the stream waits for the
    reload.  When every chunk belongs to the reloading agent there is one
    launch, after the wait.  Every chunk must still match the oracle."""
    agents = [0, 0, 0] if only_reloading else [0, 1, 2, 0, 1]
    w = small_case(29, hq=8, hkv=2, d=128, prefix_len=[333, 200, 48],
                   req_agent=agents, req_ctx=[0] * len(agents),
                   req_prefill=[100, 70, 64, 40, 90][:len(agents)],
                   req_decode=[0] * len(agents), chunk=128, permute=True)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_PREFILL_TILE_ROWS, rows)
    L = w.prefix_len[0]
    hk = torch.empty(L, 2, 128, dtype=torch.bfloat16, pin_memory=True)
    hv = torch.empty_like(hk, pin_memory=True)
    side = torch.cuda.Stream()
    ev = torch.cuda.Event()
    s.ctx.prefix_offload(0, hk, hv, side, ev)
    ev.synchronize()
    chunks, ids, lens, q, k, v = s.prefill_inputs(0)
    out, lse = s.new_outputs(sum(lens))
    torch.cuda.synchronize()
    s.ctx.set_option(B.OPT_KERNEL_TIMING, 1)
    s.ctx.kernel_times(reset=True)
    with torch.cuda.stream(side):
        torch.cuda._sleep(20_000_000)   # keeps the reload behind it in flight (bounded spin)
    s.ctx.prefix_reload(0, hk, hv, side, None)
    s.prefill(ids, lens, q, k, v, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    kt = s.ctx.kernel_times(reset=True)
    assert kt["prefill_pair_tcgen05" if rows == 256 else "dense_tcgen05"][1] == (1 if only_reloading else 2)
    row = 0
    for r, off, c in chunks:
        o_ref, l_ref = oracle.workload_prefill_chunk(w, t, r, off, c)
        compare(out[row:row + c], lse[row:row + c], o_ref, l_ref, f"r{r} off{off}")
        row += c


def test_reload_rejects_unpinned_host_memory():
    """A reload that fails (pageable host memory) leaves the prefix evicted:
    the agent's decode is refused with NOT_RESIDENT rather than waiting, and
    after a good reload (pinned copies of the prefix) the step is exact."""
    w = small_case(25, hq=8, hkv=2, d=64, prefix_len=[40], req_agent=[0], req_ctx=[1],
                   req_prefill=[0], req_decode=[1])
    t, s = _session(w)
    pk, pv = s.t.prefix(0, w)
    hk_good, hv_good = pk.cpu().pin_memory(), pv.cpu().pin_memory()
    s.ctx.prefix_evict(0)
    hk = torch.zeros(40, 2, 64, dtype=torch.bfloat16)   # pageable
    with pytest.raises(B.TpaError) as e:
        s.ctx.prefix_reload(0, hk, hk)
    assert e.value.code == B.TPA_ERR_INVALID_ARG
    assert s.ctx.query(B.Q_PREFIX_RESIDENT, 0) == 0
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    with pytest.raises(B.TpaError) as e:
        s.decode(ids, q, kn, vn, out, lse)
    assert e.value.code == B.TPA_ERR_NOT_RESIDENT
    s.ctx.prefix_reload(0, hk_good, hv_good)
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(oracle.workload_decode(w, t), range(len(ids)))
    compare(out, lse, o_ref, l_ref, "after a failed and a good reload")


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
def test_out_of_pool_page_is_redirected_and_reported(mode):
    # A plan whose first prefix page id lies outside the pool (test hook):
    # every kernel bounds-checks page ids, so the read goes to page 0, the
    # status word gets bit 4 and nothing faults; the next step is exact.
    w = small_case(78, hq=8, hkv=2, d=128, prefix_len=[300, 40], req_agent=[0, 0, 1, 0],
                   req_ctx=[10, 200, 33, 0], req_prefill=[0] * 4, req_decode=[1] * 4)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    ids, q, kn, vn = s.decode_inputs()
    lens = [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids]
    out, lse = s.new_outputs(len(ids))
    s.ctx.set_option(B.OPT_TEST_BAD_PAGE, 1)
    s.decode(ids, q, kn, vn, out, lse)
    assert s.ctx.device_status() == 4
    s.ctx.request_truncate(ids, lens)
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    ref = oracle.workload_decode(w, t)
    o_ref, l_ref = stack_decode_ref(ref, range(len(ids)))
    compare(out, lse, o_ref, l_ref, "after an out-of-pool page id")


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
def test_out_of_range_partial_slot_is_skipped_and_reported(mode):
    # A plan whose first token's partial slots lie past the partial buffer
    # (test hook): every kernel checks partial slots, so that token's
    # partials are neither written nor read, the status word gets bit 16,
    # the other tokens' outputs are exact and the next step is exact.
    w = small_case(79, hq=8, hkv=2, d=128, prefix_len=[300, 40], req_agent=[0, 0, 1, 0],
                   req_ctx=[10, 200, 33, 0], req_prefill=[0] * 4, req_decode=[1] * 4)
    t, s = _session(w)
    s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    ids, q, kn, vn = s.decode_inputs()
    lens = [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids]
    out, lse = s.new_outputs(len(ids))
    out.fill_(3.0)
    s.ctx.set_option(B.OPT_TEST_BAD_SLOT, 1)
    s.decode(ids, q, kn, vn, out, lse)
    assert s.ctx.device_status() == 16
    ref = oracle.workload_decode(w, t)
    assert torch.all(out[0].float() == 3.0)   # the skipped token's row was not written
    o_ref, l_ref = stack_decode_ref(ref, range(1, len(ids)))
    compare(out[1:], lse[1:], o_ref, l_ref, "other tokens beside a skipped slot")
    s.ctx.request_truncate(ids, lens)
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    o_ref, l_ref = stack_decode_ref(ref, range(len(ids)))
    compare(out, lse, o_ref, l_ref, "after an out-of-range partial slot")


def test_plan_wait_timeout_is_reported_and_context_recovers():
    # A decode whose kernel never sees its plan (test hook: the flag it waits
    # for is never written) gives up at the device wait limit; the host reads
    # the timeout from the status word, and after truncating that step's
    # requests back the next step is exact again.
    w = small_case(77, hq=8, hkv=2, d=128, prefix_len=[300, 40], req_agent=[0, 0, 1, 0],
                   req_ctx=[10, 200, 33, 0], req_prefill=[0] * 4, req_decode=[1] * 4)
    t, s = _session(w)
    ids, q, kn, vn = s.decode_inputs()
    lens = [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids]
    out, lse = s.new_outputs(len(ids))
    s.ctx.set_option(B.OPT_TEST_PLAN_WAIT, 1)
    s.decode(ids, q, kn, vn, out, lse)
    status = s.ctx.device_status()
    assert status & 8, status
    assert s.ctx.device_status() == 0          # the word was cleared
    s.ctx.request_truncate(ids, lens)
    s.decode(ids, q, kn, vn, out, lse)
    torch.cuda.synchronize()
    _check_status(s)
    ref = oracle.workload_decode(w, t)
    o_ref, l_ref = stack_decode_ref(ref, range(len(ids)))
    compare(out, lse, o_ref, l_ref, "after a plan-wait timeout")
