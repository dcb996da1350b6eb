"""tpa_decode_static_scratch against tpa_decode.

The variant keeps the split partials of a decode step in the library's
static device array instead of the context workspace; everything else is
tpa_decode, so two decode steps in a row must give bit-identical outputs
and leave bit-identical KV pages, and the context workspace must keep its
partials untouched.  A step needing more partials than the
array holds is refused with a CAPACITY error that names the limit, and
changes nothing.  Collected last, so it runs both alone and after every
other GPU test in the same process.
"""
import pytest
import torch

from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build
from paper_2608_25523_gb300.session import Session, to_device
from paper_2608_25523_gb300.workloads import small_case, tensors_numpy

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    if not torch.cuda.is_available():
        pytest.skip("needs a GPU")
    build()
    B.load()


def _workload(seed):
    # 3 agents (prefix 0, 300 and 1000 tokens), 12 decode requests with
    # cached suffixes 0..297 tokens: several prefix splits and suffix ranges
    agents = [0, 1, 2, 2, 1, 2, 0, 2, 1, 2, 2, 1]
    return small_case(seed, hq=16, hkv=4, d=128, prefix_len=[0, 300, 1000], req_agent=agents,
                      req_ctx=[(27 * i) % 298 for i in range(len(agents))],
                      req_prefill=[0] * len(agents), req_decode=[1] * len(agents), permute=True)


def _step_inputs(w, n, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    def r(*shape):
        return torch.randn(*shape, generator=g, device="cuda").to(torch.bfloat16)
    return (r(n, w.num_q_heads, w.head_dim), r(n, w.num_kv_heads, w.head_dim),
            r(n, w.num_kv_heads, w.head_dim))


def _bits(x):
    return x.contiguous().view(torch.int16) if x.dtype == torch.bfloat16 else x.view(torch.int32)


def _suffix_pages(s, ids):
    w = s.w
    out = []
    for r in ids:
        n = s.ctx.query(B.Q_SUFFIX_LEN, r)
        k = torch.empty(n, w.num_kv_heads, w.head_dim, dtype=torch.bfloat16, device="cuda")
        v = torch.empty_like(k)
        s.ctx.gather(r, True, k, v)
        out.append((k, v))
    torch.cuda.synchronize()
    return out


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
def test_two_steps_bit_identical_to_decode(mode):
    w = _workload(11 + mode)
    t = to_device(tensors_numpy(w), "cuda")
    ref = Session(w, t)
    var = Session(w, t)
    for s in (ref, var):
        s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    ids, q, kn, vn = ref.decode_inputs()
    steps = [(q, kn, vn), _step_inputs(w, len(ids), 1234 + mode)]
    for k, (q, kn, vn) in enumerate(steps):
        o_ref, l_ref = ref.new_outputs(len(ids))
        o_var, l_var = var.new_outputs(len(ids))
        o_var.fill_(7.0)
        l_var.fill_(7.0)
        ref.ctx.decode(ids, q, kn, vn, o_ref, l_ref)
        var.ctx.decode_static_scratch(ids, q, kn, vn, o_var, l_var)
        torch.cuda.synchronize()
        assert ref.ctx.device_status() == 0 and var.ctx.device_status() == 0
        assert torch.equal(_bits(o_var), _bits(o_ref)), f"step {k}: out differs"
        assert torch.equal(_bits(l_var), _bits(l_ref)), f"step {k}: lse differs"
    for (kr, vr), (kv, vv) in zip(_suffix_pages(ref, ids), _suffix_pages(var, ids)):
        assert torch.equal(_bits(kr), _bits(kv)) and torch.equal(_bits(vr), _bits(vv))
    ref.ctx.close()
    var.ctx.close()


@pytest.mark.parametrize("mode", [0, 1], ids=["cascade", "flat"])
def test_workspace_partials_untouched(mode):
    """The partials really live in the static array: after a tpa_decode
    step, the same step with other inputs through tpa_decode_static_scratch
    changes only the plan upload in the context workspace, while through
    tpa_decode it rewrites the workspace's partials (far more bytes)."""
    w = _workload(71 + mode)
    s = Session(w, to_device(tensors_numpy(w), "cuda"))
    s.ctx.set_option(B.OPT_DECODE_MODE, mode)
    ids = list(range(w.num_requests))
    lens = [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids]
    out, lse = s.new_outputs(len(ids))
    ws = s.ctx.workspace

    def changed_by(fn, seed):
        q, kn, vn = _step_inputs(w, len(ids), seed)
        before = ws.clone()
        fn(ids, q, kn, vn, out, lse)
        torch.cuda.synchronize()
        s.ctx.request_truncate(ids, lens)
        return int((ws != before).sum())

    changed_by(s.ctx.decode, 1)
    static = changed_by(s.ctx.decode_static_scratch, 2)
    regular = changed_by(s.ctx.decode, 3)
    assert s.ctx.device_status() == 0
    # the step's partials: at least one per (token, q head), (d + 1) fp32 each
    partial_bytes = len(ids) * w.num_q_heads * (w.head_dim + 1) * 4
    assert static < partial_bytes // 4, (static, partial_bytes)
    assert regular > partial_bytes // 2, (regular, partial_bytes)
    s.ctx.close()


def test_oversize_step_refused():
    # 64 requests x 32 q heads with 16-key suffix ranges need ~260k partial
    # slots, far more than the 16 MiB array holds at head_dim 128
    agents = [i % 4 for i in range(64)]
    w = small_case(5, hq=32, hkv=8, d=128, prefix_len=[2048] * 4, req_agent=agents,
                   req_ctx=[2000] * 64, req_prefill=[0] * 64, req_decode=[1] * 64, permute=False)
    t = to_device(tensors_numpy(w), "cuda")
    s = Session(w, t, max_splits=256)
    s.ctx.set_option(B.OPT_SUFFIX_SPLIT_KEYS, 16)
    ids, q, kn, vn = s.decode_inputs()
    out, lse = s.new_outputs(len(ids))
    before = [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids]
    free = s.ctx.query(B.Q_FREE_PAGES)
    with pytest.raises(B.TpaError) as e:
        s.ctx.decode_static_scratch(ids, q, kn, vn, out, lse)
    assert e.value.code == B.TPA_ERR_CAPACITY
    assert "static scratch" in str(e.value)
    assert [s.ctx.query(B.Q_SUFFIX_LEN, r) for r in ids] == before
    assert s.ctx.query(B.Q_FREE_PAGES) == free
    s.ctx.close()
