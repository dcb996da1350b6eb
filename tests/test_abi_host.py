"""Host-side checks of the C ABI (no GPU needed).

The library is built here with nvcc and loaded; contexts are created with
TPA_FLAG_PLAN_ONLY, which runs the page tables and the planner but makes
no CUDA call.  Covers: every declared symbol is exported, lifecycle and
error codes (the pool budget of Eq. 2 -> NO_SPACE, evicted prefixes ->
NOT_RESIDENT), all-or-nothing failures, page accounting, and the plan's
work decomposition for the decode cascade.
"""
import ctypes
import math

import pytest

from paper_2608_25523_gb300 import binding as B
from paper_2608_25523_gb300.build import build


@pytest.fixture(scope="module")
def lib():
    build()
    return B.load()


def plan_ctx(num_pages=64, hq=8, hkv=2, d=128, agents=4, reqs=8, tokens=64, seq=1024, seed=0,
             splits=0):
    cfg = B.make_config(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, num_pages=num_pages,
                        max_agents=agents, max_requests=reqs, max_tokens=tokens,
                        max_seq_len=seq, max_splits=splits, page_order_seed=seed,
                        flags=B.TPA_FLAG_PLAN_ONLY)
    return B.Context(cfg)


def test_exports_every_declared_symbol(lib):
    names = B.header_functions()
    assert len(names) >= 18
    for n in names:
        assert hasattr(lib, n), n
    # and nothing else with the library's prefix is declared but missing
    assert set(names) == set(B._SIGS), set(names) ^ set(B._SIGS)


def test_workspace_size(lib):
    ok = B.make_config(num_q_heads=32, num_kv_heads=8, head_dim=128, num_pages=10, max_agents=1,
                       max_requests=100, max_tokens=64, max_seq_len=1000)
    # partial results: min(max_tokens, max_requests) x Hq x 32 splits x (d + 1) floats
    assert B.workspace_size(ok) > 64 * 32 * 32 * 129 * 4
    for hq, hkv, d in [(32, 8, 96), (12, 4, 128), (32, 2, 128)]:
        bad = B.make_config(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, num_pages=10,
                            max_agents=1, max_requests=1, max_tokens=64, max_seq_len=1000)
        assert B.workspace_size(bad) == 0


def test_unsupported_shape(lib):
    cfg = B.make_config(num_q_heads=12, num_kv_heads=4, head_dim=128, num_pages=8, max_agents=1,
                        max_requests=1, max_tokens=8, max_seq_len=64, flags=B.TPA_FLAG_PLAN_ONLY)
    with pytest.raises(B.TpaError) as e:
        B.Context(cfg)
    assert e.value.code == B.TPA_ERR_UNSUPPORTED


def test_prefix_lifecycle_and_budget(lib):
    ctx = plan_ctx(num_pages=10)
    assert ctx.query(B.Q_FREE_PAGES) == 10
    ctx.prefix_register(0, 33)                       # 3 pages
    assert ctx.query(B.Q_FREE_PAGES) == 7
    assert ctx.query(B.Q_PREFIX_LEN, 0) == 33
    assert ctx.query(B.Q_PREFIX_RESIDENT, 0) == 1
    with pytest.raises(B.TpaError) as e:
        ctx.prefix_register(0, 5)
    assert e.value.code == B.TPA_ERR_STATE
    with pytest.raises(B.TpaError) as e:
        ctx.prefix_register(1, 16 * 8)               # 8 pages > 7 free: the KV budget
    assert e.value.code == B.TPA_ERR_NO_SPACE
    assert ctx.query(B.Q_FREE_PAGES) == 7            # failed call changed nothing
    assert ctx.query(B.Q_PREFIX_LEN, 1) == -1
    ctx.prefix_register(1, 0)                        # empty prefix is allowed
    assert ctx.query(B.Q_FREE_PAGES) == 7
    ctx.prefix_evict(0)
    assert ctx.query(B.Q_FREE_PAGES) == 10
    assert ctx.query(B.Q_PREFIX_RESIDENT, 0) == 0
    with pytest.raises(B.TpaError) as e:
        ctx.prefix_evict(0)
    assert e.value.code == B.TPA_ERR_NOT_RESIDENT
    with pytest.raises(B.TpaError) as e:
        ctx.prefix_register(-1, 4)
    assert e.value.code == B.TPA_ERR_INVALID_ARG
    with pytest.raises(B.TpaError) as e:
        ctx.prefix_register(9, 4)
    assert e.value.code == B.TPA_ERR_INVALID_ARG


def test_reload_needs_evicted_prefix_and_space(lib):
    ctx = plan_ctx(num_pages=6)
    ctx.prefix_register(0, 40)                       # 3 pages
    with pytest.raises(B.TpaError) as e:
        ctx.prefix_reload(0, 1, 1)
    assert e.value.code == B.TPA_ERR_STATE
    ctx.prefix_evict(0)
    ctx.prefix_register(1, 64)                       # 4 pages, 2 left
    with pytest.raises(B.TpaError) as e:
        ctx.prefix_reload(0, 1, 1)
    assert e.value.code == B.TPA_ERR_NO_SPACE
    assert ctx.query(B.Q_PREFIX_RESIDENT, 0) == 0
    ctx.prefix_evict(1)
    ctx.prefix_reload(0, 1, 1)                       # plan-only: pointers are not touched
    assert ctx.query(B.Q_PREFIX_RESIDENT, 0) == 1
    assert ctx.query(B.Q_FREE_PAGES) == 3


def test_request_lifecycle_and_append_accounting(lib):
    ctx = plan_ctx(num_pages=12, tokens=256)
    with pytest.raises(B.TpaError) as e:
        ctx.request_open(0, 0)                       # agent not registered
    assert e.value.code == B.TPA_ERR_STATE
    ctx.prefix_register(0, 20)                       # 2 pages
    ctx.request_open(0, 0)
    ctx.request_open(1, 0)
    with pytest.raises(B.TpaError) as e:
        ctx.request_open(1, 0)
    assert e.value.code == B.TPA_ERR_STATE
    ctx.kv_append([0, 1], [17, 0], 1, 1)             # 2 pages for request 0
    assert ctx.query(B.Q_SUFFIX_LEN, 0) == 17
    assert ctx.query(B.Q_FREE_PAGES) == 8
    ctx.kv_append([0], [15], 1, 1)                   # 32 tokens: still 2 pages
    assert ctx.query(B.Q_FREE_PAGES) == 8
    ctx.kv_append([0], [1], 1, 1)                    # 33 -> third page
    assert ctx.query(B.Q_FREE_PAGES) == 7
    with pytest.raises(B.TpaError) as e:
        ctx.kv_append([0, 0], [1, 1], 1, 1)          # duplicate id in a batch
    assert e.value.code == B.TPA_ERR_INVALID_ARG
    with pytest.raises(B.TpaError) as e:
        ctx.kv_append([1, 0], [16 * 7 + 1, 1], 1, 1)  # needs 8 pages, 7 free: all or nothing
    assert e.value.code == B.TPA_ERR_NO_SPACE
    assert ctx.query(B.Q_SUFFIX_LEN, 0) == 33 and ctx.query(B.Q_SUFFIX_LEN, 1) == 0
    assert ctx.query(B.Q_FREE_PAGES) == 7
    ctx.request_close(0)
    assert ctx.query(B.Q_FREE_PAGES) == 10
    assert ctx.query(B.Q_SUFFIX_LEN, 0) == -1
    with pytest.raises(B.TpaError) as e:
        ctx.request_close(0)
    assert e.value.code == B.TPA_ERR_STATE


def test_decode_requires_resident_prefix(lib):
    ctx = plan_ctx(num_pages=20)
    ctx.prefix_register(0, 16)
    ctx.request_open(0, 0)
    ctx.prefix_evict(0)
    with pytest.raises(B.TpaError) as e:
        ctx.decode([0], 1, 1, 1, 1, 1)
    assert e.value.code == B.TPA_ERR_NOT_RESIDENT
    with pytest.raises(B.TpaError) as e:
        ctx.prefill_chunk([0], [4], 1, 1, 1, 1, 1)
    assert e.value.code == B.TPA_ERR_NOT_RESIDENT
    assert ctx.query(B.Q_SUFFIX_LEN, 0) == 0


def test_capacity_limits(lib):
    ctx = plan_ctx(num_pages=200, tokens=8, seq=100)
    ctx.prefix_register(0, 16)
    for r in range(8):
        ctx.request_open(r, 0)
    with pytest.raises(B.TpaError) as e:
        ctx.kv_append([0], [101], 1, 1)              # beyond max_seq_len
    assert e.value.code == B.TPA_ERR_CAPACITY
    with pytest.raises(B.TpaError) as e:
        ctx.kv_append([0, 1], [5, 4], 1, 1)          # 9 tokens > max_tokens
    assert e.value.code == B.TPA_ERR_CAPACITY


def test_degenerate_batches_are_refused_and_leave_tables_unchanged(lib):
    ctx = plan_ctx(num_pages=100, reqs=4, tokens=64)
    ctx.prefix_register(0, 40)
    for r in range(3):
        ctx.request_open(r, 0)
    ctx.kv_append([0, 1, 2], [5, 17, 1], 1, 1)
    lens = [ctx.query(B.Q_SUFFIX_LEN, r) for r in range(3)]
    free = ctx.query(B.Q_FREE_PAGES)
    cases = [
        (lambda: ctx.decode([], 1, 1, 1, 1, 1), B.TPA_ERR_INVALID_ARG),              # empty batch
        (lambda: ctx.prefill_chunk([], [], 1, 1, 1, 1, 1), B.TPA_ERR_INVALID_ARG),
        (lambda: ctx.kv_append([], [], 1, 1), B.TPA_ERR_INVALID_ARG),
        (lambda: ctx.decode([0, 1, 0], 1, 1, 1, 1, 1), B.TPA_ERR_INVALID_ARG),       # a request twice
        (lambda: ctx.prefill_chunk([1, 1], [4, 4], 1, 1, 1, 1, 1), B.TPA_ERR_INVALID_ARG),
        (lambda: ctx.prefill_chunk([0, 1], [4, 0], 1, 1, 1, 1, 1), B.TPA_ERR_INVALID_ARG),  # empty chunk
        (lambda: ctx.decode([0, 4], 1, 1, 1, 1, 1), B.TPA_ERR_INVALID_ARG),          # id out of range
        (lambda: ctx.decode([0, -1], 1, 1, 1, 1, 1), B.TPA_ERR_INVALID_ARG),
        (lambda: ctx.decode([0, 3], 1, 1, 1, 1, 1), B.TPA_ERR_STATE),                # not open
    ]
    for call, code in cases:
        with pytest.raises(B.TpaError) as e:
            call()
        assert e.value.code == code
        assert [ctx.query(B.Q_SUFFIX_LEN, r) for r in range(3)] == lens
        assert ctx.query(B.Q_FREE_PAGES) == free
    ctx.decode([0, 1, 2], 1, 1, 1, 1, 1)         # and the context still works
    assert [ctx.query(B.Q_SUFFIX_LEN, r) for r in range(3)] == [n + 1 for n in lens]


def test_decode_plan_decomposition(lib):
    """Llama-3-8B decode shape: 4 agents x 4096-token prefixes, 16 requests each."""
    hq, hkv, G = 32, 8, 4
    ctx = plan_ctx(num_pages=4 * 256 + 64 * 70, hq=hq, hkv=hkv, agents=4, reqs=64, tokens=1024,
                   seq=4096)
    lens = [256 + 12 * r for r in range(64)]
    for a in range(4):
        ctx.prefix_register(a, 4096)
    for r in range(64):
        ctx.request_open(r, r // 16)
        ctx.kv_append([r], [lens[r]], 1, 1)
    ctx.set_option(B.OPT_PREFIX_SPLITS, 4)
    ctx.set_option(B.OPT_SUFFIX_SPLIT_KEYS, 256)
    ctx.decode(list(range(64)), 1, 1, 1, 1, 1)
    # one launch: level 1 (dense CTAs) = (agent, kv head) x one 128-row tile
    # (16 tokens x G=4 rows) x 4 key splits; level 2 (split-KV CTAs) = per
    # token and kv head, ceil((len+1)/256) suffix items
    assert ctx.query(B.Q_LAST_DENSE_ITEMS) == 4 * hkv * 1 * 4
    assert ctx.query(B.Q_LAST_SUFFIX_ITEMS) == sum(hkv * math.ceil((l + 1) / 256) for l in lens)
    assert ctx.query(B.Q_LAST_LAUNCHES) == 0        # plan-only: nothing launched
    for r in range(64):
        assert ctx.query(B.Q_SUFFIX_LEN, r) == lens[r] + 1
    # flat mode: no dense items, the prefix goes through the split-KV kernel
    ctx.set_option(B.OPT_DECODE_MODE, 1)
    ctx.decode(list(range(64)), 1, 1, 1, 1, 1)
    assert ctx.query(B.Q_LAST_DENSE_ITEMS) == 0
    assert ctx.query(B.Q_LAST_SUFFIX_ITEMS) == sum(
        hkv * (math.ceil((l + 2) / 256) + 4096 // 256) for l in lens)


def test_prefill_plan_decomposition(lib):
    hq, hkv, G = 8, 2, 4
    ctx = plan_ctx(num_pages=400, hq=hq, hkv=hkv, agents=2, reqs=4, tokens=2048, seq=4096)
    ctx.prefix_register(0, 300)
    ctx.prefix_register(1, 0)
    for r in range(4):
        ctx.request_open(r, r % 2)
    # default: items of two 128-row tiles, 256/G tokens of one chunk
    ctx.prefill_chunk([0, 1, 2, 3], [512, 33, 1, 100], 1, 1, 1, 1, 1)
    items_of = lambda c, rows: math.ceil(c / (rows // G))
    assert ctx.query(B.Q_LAST_DENSE_ITEMS) == hkv * sum(items_of(c, 256) for c in (512, 33, 1, 100))
    assert [ctx.query(B.Q_SUFFIX_LEN, r) for r in range(4)] == [512, 33, 1, 100]
    # single 128-row tiles
    ctx.set_option(B.OPT_PREFILL_TILE_ROWS, 128)
    ctx.prefill_chunk([0, 1, 2, 3], [64, 33, 1, 100], 1, 1, 1, 1, 1)
    assert ctx.query(B.Q_LAST_DENSE_ITEMS) == hkv * sum(items_of(c, 128) for c in (64, 33, 1, 100))
    assert [ctx.query(B.Q_SUFFIX_LEN, r) for r in range(4)] == [576, 66, 2, 200]
    with pytest.raises(B.TpaError):
        ctx.set_option(B.OPT_PREFILL_TILE_ROWS, 64)


def test_prefill_plan_with_prefix_and_suffix_at_max_seq_len(lib):
    """An item's key tiles (prefix + causal suffix) can reach twice
    max_seq_len / 128; the planner's longest-first ordering must size for
    that."""
    hkv, G = 2, 4
    ctx = plan_ctx(num_pages=300, hq=8, hkv=hkv, agents=2, reqs=3, tokens=2048, seq=1024)
    ctx.prefix_register(0, 1024)
    ctx.prefix_register(1, 1000)
    for r, a in enumerate((0, 1, 0)):
        ctx.request_open(r, a)
    for c in (1000, 24):
        ctx.prefill_chunk([0, 1, 2], [c, c, 1], 1, 1, 1, 1, 1)
        assert ctx.query(B.Q_LAST_DENSE_ITEMS) == hkv * (2 * math.ceil(c / (256 // G)) + 1)
    assert [ctx.query(B.Q_SUFFIX_LEN, r) for r in range(3)] == [1024, 1024, 2]


def test_permuted_pool_is_a_permutation(lib):
    ctx = plan_ctx(num_pages=50, seed=12345)
    firsts = []
    for a in range(4):
        ctx.prefix_register(a, 16)
        firsts.append(ctx.query(B.Q_PAGE_OF, a))
    assert firsts != [0, 1, 2, 3]
    assert len(set(firsts)) == 4 and all(0 <= p < 50 for p in firsts)
    ctx2 = plan_ctx(num_pages=50, seed=12345)
    for a in range(4):
        ctx2.prefix_register(a, 16)
    assert [ctx2.query(B.Q_PAGE_OF, a) for a in range(4)] == firsts   # seeded, deterministic
