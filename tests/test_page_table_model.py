"""Model-based test of the host page tables (no GPU needed).

Hypothesis drives random sequences of the C ABI's table calls (register,
evict, reload, offload, open, close, truncate, append, decode, prefill
chunk, decode-mode and tile options) on plan-only contexts, next to a small
Python model of what each call does to the KV pool of Eq. 2:

- a resident prefix of length ell holds ceil(ell / 16) pages; an evicted one
  holds none;
- an open request with a suffix of L tokens holds ceil(L / 16) pages;
- every other page is free.

For every call the model predicts the return code from the order of checks
the header documents (batch shape, ids, open, resident, duplicates, token
totals, lengths, then space), and a failed call must leave every count
unchanged.  After every step the free-page count, prefix lengths and
residency and every request's suffix length are compared with the
library's answers to tpa_query.
"""
import pytest

hypothesis = pytest.importorskip("hypothesis")
from hypothesis import settings, strategies as st  # noqa: E402
from hypothesis.stateful import (RuleBasedStateMachine, initialize, invariant,  # noqa: E402
                                 rule)

from paper_2608_25523_gb300 import binding as B  # noqa: E402
from paper_2608_25523_gb300.build import build  # noqa: E402

PAGE = 16
AGENTS = 4
REQS = 6
NUM_PAGES = 40
MAX_TOKENS = 64
MAX_SEQ = 256
HKV = 2

lengths = (st.integers(0, 96) | st.integers(0, 96) | st.integers(0, 96)
           | st.sampled_from([-1, MAX_SEQ, MAX_SEQ + 1]))


def cdiv(a, b):
    return -(-a // b)


@pytest.fixture(scope="module", autouse=True)
def _lib():
    build()
    B.load()


class PageTableMachine(RuleBasedStateMachine):
    def __init__(self):
        super().__init__()
        cfg = B.make_config(num_q_heads=8, num_kv_heads=HKV, head_dim=128, num_pages=NUM_PAGES,
                            max_agents=AGENTS, max_requests=REQS, max_tokens=MAX_TOKENS,
                            max_seq_len=MAX_SEQ, flags=B.TPA_FLAG_PLAN_ONLY)
        self.ctx = B.Context(cfg)
        self.prefix = {}     # agent -> [length, resident]
        self.suffix = {}     # request -> [agent, length]
        self.cascade = True

    def teardown(self):
        self.ctx.close()

    # -- the model ----------------------------------------------------------
    def free(self):
        used = sum(cdiv(l, PAGE) for l, res in self.prefix.values() if res)
        used += sum(cdiv(l, PAGE) for _, l in self.suffix.values())
        return NUM_PAGES - used

    def batch_rc(self, reqs, need_resident):
        if len(reqs) <= 0:
            return B.TPA_ERR_INVALID_ARG
        if len(reqs) > MAX_TOKENS:
            return B.TPA_ERR_CAPACITY
        for r in reqs:
            if r < 0 or r >= REQS:
                return B.TPA_ERR_INVALID_ARG
            if r not in self.suffix:
                return B.TPA_ERR_STATE
            if need_resident and not self.prefix[self.suffix[r][0]][1]:
                return B.TPA_ERR_NOT_RESIDENT
        if len(set(reqs)) != len(reqs):
            return B.TPA_ERR_INVALID_ARG
        return B.TPA_OK

    def reserve_rc(self, reqs, ntok):
        need = 0
        for r, t in zip(reqs, ntok):
            if t < 0:
                return B.TPA_ERR_INVALID_ARG
            length = self.suffix[r][1]
            if length + t > MAX_SEQ:
                return B.TPA_ERR_CAPACITY
            need += cdiv(length + t, PAGE) - cdiv(length, PAGE)
        return B.TPA_ERR_NO_SPACE if need > self.free() else B.TPA_OK

    def counts(self, data, n, lo, hi):
        """n per-request counts in [lo, hi], sometimes one of them -1 or 0."""
        vals = data.draw(st.lists(st.integers(lo, hi), min_size=n, max_size=n))
        if vals and not data.draw(st.integers(0, 5)):
            vals[data.draw(st.integers(0, n - 1))] = data.draw(st.sampled_from([-1, 0]))
        return vals

    def grow(self, reqs, ntok):
        for r, t in zip(reqs, ntok):
            self.suffix[r][1] += t

    @staticmethod
    def pick(data, good, limit):
        """An id: mostly one of `good` (the ids the call can succeed on),
        else any id in [-1, limit], out-of-range ones included."""
        if good and data.draw(st.integers(0, 3)):
            return data.draw(st.sampled_from(sorted(good)))
        return data.draw(st.integers(-1, limit))

    def batch(self, data):
        """A batch of request ids: mostly distinct open requests, sometimes
        with a duplicate, a closed or an out-of-range id, or empty."""
        open_reqs = sorted(self.suffix)
        reqs = data.draw(st.lists(st.sampled_from(open_reqs), unique=True, min_size=1, max_size=5)
                         if open_reqs else st.just([]))
        flaw = data.draw(st.integers(0, 9))
        if flaw == 3:
            reqs = []
        elif flaw == 0 and reqs:
            reqs.insert(data.draw(st.integers(0, len(reqs))), reqs[0])
        elif flaw == 1:
            reqs.append(data.draw(st.sampled_from([-1, REQS])))
        elif flaw == 2:
            closed = [r for r in range(REQS) if r not in self.suffix]
            if closed:
                reqs.insert(0, data.draw(st.sampled_from(closed)))
        return reqs

    def call(self, expect, fn, *args):
        """Run one library call; its return code must be the model's."""
        before = self.snapshot()
        try:
            fn(*args)
            rc = B.TPA_OK
        except B.TpaError as e:
            rc = e.code
        assert rc == expect, (fn.__name__, args, rc, expect)
        if rc != B.TPA_OK:
            assert self.snapshot() == before, (fn.__name__, args, "failed call changed state")
        return rc == B.TPA_OK

    def snapshot(self):
        q = self.ctx.query
        return (q(B.Q_FREE_PAGES),
                tuple((q(B.Q_PREFIX_LEN, a), q(B.Q_PREFIX_RESIDENT, a)) for a in range(AGENTS)),
                tuple(q(B.Q_SUFFIX_LEN, r) for r in range(REQS)))

    # -- prefixes -----------------------------------------------------------
    @initialize(lens=st.lists(lengths, min_size=1, max_size=AGENTS), reqs=st.integers(1, REQS))
    def start(self, lens, reqs):
        """Some prefixes registered and requests opened up front."""
        for a, length in enumerate(lens):
            self.register_agent(a, length)
        agents = sorted(self.prefix)
        for r in range(reqs if agents else 0):
            self.open_request(r, agents[r % len(agents)])

    @rule(data=st.data(), length=lengths)
    def register(self, data, length):
        self.register_agent(self.pick(data, set(range(AGENTS)) - set(self.prefix), AGENTS), length)

    def register_agent(self, agent, length):
        if agent < 0 or agent >= AGENTS or length < 0 or length > MAX_SEQ:
            rc = B.TPA_ERR_INVALID_ARG
        elif agent in self.prefix:
            rc = B.TPA_ERR_STATE
        elif cdiv(length, PAGE) > self.free():
            rc = B.TPA_ERR_NO_SPACE
        else:
            rc = B.TPA_OK
        if self.call(rc, self.ctx.prefix_register, agent, length):
            self.prefix[agent] = [length, True]

    @rule(data=st.data(), offload=st.booleans())
    def evict(self, data, offload):
        agent = self.pick(data, {a for a, (_, res) in self.prefix.items() if res}, AGENTS)
        if agent < 0 or agent >= AGENTS:
            rc = B.TPA_ERR_INVALID_ARG
        elif agent not in self.prefix:
            rc = B.TPA_ERR_STATE
        elif not self.prefix[agent][1]:
            rc = B.TPA_ERR_NOT_RESIDENT
        else:
            rc = B.TPA_OK
        # plan-only contexts take the host pointers without touching them
        done = (self.call(rc, self.ctx.prefix_offload, agent, 1, 1) if offload
                else self.call(rc, self.ctx.prefix_evict, agent))
        if done:
            self.prefix[agent][1] = False

    @rule(data=st.data())
    def reload(self, data):
        agent = self.pick(data, {a for a, (_, res) in self.prefix.items() if not res}, AGENTS)
        if agent < 0 or agent >= AGENTS:
            rc = B.TPA_ERR_INVALID_ARG
        elif agent not in self.prefix or self.prefix[agent][1]:
            rc = B.TPA_ERR_STATE
        elif cdiv(self.prefix[agent][0], PAGE) > self.free():
            rc = B.TPA_ERR_NO_SPACE
        else:
            rc = B.TPA_OK
        if self.call(rc, self.ctx.prefix_reload, agent, 1, 1):
            self.prefix[agent][1] = True

    # -- requests -----------------------------------------------------------
    @rule(data=st.data())
    def open(self, data):
        self.open_request(self.pick(data, set(range(REQS)) - set(self.suffix), REQS),
                          self.pick(data, set(self.prefix), AGENTS))

    def open_request(self, req, agent):
        if req < 0 or req >= REQS or agent < 0 or agent >= AGENTS:
            rc = B.TPA_ERR_INVALID_ARG
        elif req in self.suffix or agent not in self.prefix:
            rc = B.TPA_ERR_STATE
        else:
            rc = B.TPA_OK
        if self.call(rc, self.ctx.request_open, req, agent):
            self.suffix[req] = [agent, 0]

    @rule(data=st.data())
    def close(self, data):
        req = self.pick(data, set(self.suffix), REQS)
        if req < 0 or req >= REQS:
            rc = B.TPA_ERR_INVALID_ARG
        elif req not in self.suffix:
            rc = B.TPA_ERR_STATE
        else:
            rc = B.TPA_OK
        if self.call(rc, self.ctx.request_close, req):
            del self.suffix[req]

    @rule(data=st.data())
    def truncate(self, data):
        reqs = self.batch(data)
        # a length within each suffix, sometimes one past its end
        lens = [data.draw(st.integers(0, self.suffix[r][1] if r in self.suffix else 0))
                for r in reqs]
        if lens and not data.draw(st.integers(0, 5)):
            i = data.draw(st.integers(0, len(lens) - 1))
            lens[i] = data.draw(st.sampled_from([-1, lens[i] + 1]))
        rc = self.batch_rc(reqs, False)
        if rc == B.TPA_OK:
            for r, l in zip(reqs, lens):
                if l < 0 or l > self.suffix[r][1]:
                    rc = B.TPA_ERR_INVALID_ARG
                    break
        if self.call(rc, self.ctx.request_truncate, reqs, lens):
            for r, l in zip(reqs, lens):
                self.suffix[r][1] = l

    @rule(data=st.data())
    def append(self, data):
        reqs = self.batch(data)
        ntok = self.counts(data, len(reqs), 0, 24)
        rc = self.batch_rc(reqs, False)
        if rc == B.TPA_OK and sum(max(t, 0) for t in ntok) > MAX_TOKENS:
            rc = B.TPA_ERR_CAPACITY
        if rc == B.TPA_OK:
            rc = self.reserve_rc(reqs, ntok)
        if self.call(rc, self.ctx.kv_append, reqs, ntok, 1, 1):
            self.grow(reqs, ntok)

    @rule(data=st.data())
    def decode(self, data):
        reqs = self.batch(data)
        rc = self.batch_rc(reqs, True)
        if rc == B.TPA_OK:
            rc = self.reserve_rc(reqs, [1] * len(reqs))
        if self.call(rc, self.ctx.decode, reqs, None, None, None, None, None):
            self.grow(reqs, [1] * len(reqs))
            q = self.ctx.query
            assert q(B.Q_LAST_LAUNCHES) == 0        # a plan-only context launches nothing
            # every token has at least its own new key: one suffix item per kv head at least
            assert q(B.Q_LAST_SUFFIX_ITEMS) >= HKV * len(reqs)
            with_prefix = any(self.prefix[self.suffix[r][0]][0] > 0 for r in reqs)
            assert (q(B.Q_LAST_DENSE_ITEMS) > 0) == (self.cascade and with_prefix)

    @rule(data=st.data())
    def prefill(self, data):
        reqs = self.batch(data)
        chunk = self.counts(data, len(reqs), 1, 24)
        rc = self.batch_rc(reqs, True)
        if rc == B.TPA_OK and any(c <= 0 for c in chunk):
            rc = B.TPA_ERR_INVALID_ARG
        if rc == B.TPA_OK and sum(chunk) > MAX_TOKENS:
            rc = B.TPA_ERR_CAPACITY
        if rc == B.TPA_OK:
            rc = self.reserve_rc(reqs, chunk)
        if self.call(rc, self.ctx.prefill_chunk, reqs, chunk, None, None, None, None, None):
            self.grow(reqs, chunk)

    # -- options that change the plans, not the tables ----------------------
    @rule(cascade=st.booleans(), rows=st.sampled_from([128, 256]),
          splits=st.sampled_from([0, 1, 2]), keys=st.sampled_from([0, 16, 64]))
    def options(self, cascade, rows, splits, keys):
        self.ctx.set_option(B.OPT_DECODE_MODE, 0 if cascade else 1)
        self.ctx.set_option(B.OPT_PREFILL_TILE_ROWS, rows)
        self.ctx.set_option(B.OPT_PREFIX_SPLITS, splits)
        self.ctx.set_option(B.OPT_SUFFIX_SPLIT_KEYS, keys)
        self.cascade = cascade

    # -- the tables against the model ---------------------------------------
    @invariant()
    def tables_match(self):
        free, prefixes, suffixes = self.snapshot()
        assert free == self.free()
        for a in range(AGENTS):
            want = (self.prefix[a][0], int(self.prefix[a][1])) if a in self.prefix else (-1, -1)
            assert prefixes[a] == want, a
        for r in range(REQS):
            assert suffixes[r] == (self.suffix[r][1] if r in self.suffix else -1), r


PageTableMachine.TestCase.settings = settings(max_examples=300, stateful_step_count=40,
                                              derandomize=True, database=None,
                                              deadline=None)
test_page_tables = PageTableMachine.TestCase
