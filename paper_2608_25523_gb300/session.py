"""Drive a synthetic serving workload through the library.

A Session owns one context sized for a workload, writes the agents'
prefixes, opens the requests and appends their cached suffix context, and
then issues the calls a serving engine would make per step: a decode step
over the decoding requests, prefill chunk rounds, prefix reloads from
pinned host memory.  It only moves tensors and ids; all arithmetic happens
in the library's kernels.
"""
from __future__ import annotations

import torch

from . import binding as B
from .workloads import PAGE, Tensors, Workload


def to_device(t: Tensors, device) -> Tensors:
    """numpy (bf16-valued float32) tensors -> torch bf16 on `device`."""
    def cv(x):
        if isinstance(x, torch.Tensor):
            return x.to(device)
        return torch.from_numpy(x).to(device).to(torch.bfloat16)
    return Tensors(cv(t.prefix_k), cv(t.prefix_v), cv(t.suffix_k), cv(t.suffix_v),
                   cv(t.q_prefill), cv(t.q_decode), t.prefix_off, t.suffix_off, t.qpf_off)


class Session:
    def __init__(self, w: Workload, t: Tensors, device="cuda", extra_tokens=64, max_splits=0,
                 max_tokens=None, setup=True):
        self.w, self.t, self.device = w, t, device
        self.dec = w.decode_requests()
        round_tokens = max([sum(c for _, _, c in w.chunks_of_round(r))
                            for r in range(w.prefill_rounds())] + [0])
        self.max_tokens = max_tokens or max(len(self.dec), round_tokens, 1024)
        slack = w.num_requests * (extra_tokens // PAGE + 1)
        max_seq = max(list(w.prefix_len) + [w.req_total(r) + extra_tokens
                                            for r in range(w.num_requests)])
        self.ctx = B.allocate(num_q_heads=w.num_q_heads, num_kv_heads=w.num_kv_heads,
                              head_dim=w.head_dim, num_pages=w.pages_needed() + slack,
                              max_agents=w.num_agents, max_requests=w.num_requests,
                              max_tokens=self.max_tokens, max_seq_len=max_seq,
                              max_splits=max_splits,
                              page_order_seed=w.page_order_seed if w.permute_pages else 0,
                              device=device)
        self.host_prefix = {}
        if setup:
            self.setup()

    # ------------------------------------------------------------------ setup
    def setup(self):
        w, t, ctx = self.w, self.t, self.ctx
        for a in range(w.num_agents):
            ctx.prefix_register(a, w.prefix_len[a])
            if w.prefix_len[a]:
                k, v = t.prefix(a, w)
                ctx.prefix_write(a, k.contiguous(), v.contiguous())
        for r in range(w.num_requests):
            ctx.request_open(r, w.req_agent[r])
        # cached suffix context, in calls of at most max_tokens rows (a long
        # context is split across calls; each call takes a request once)
        done = [0] * w.num_requests
        pending = [r for r in range(w.num_requests) if w.req_ctx[r] > 0]
        while pending:
            batch, rows = [], 0
            for r in pending:
                take = min(w.req_ctx[r] - done[r], self.max_tokens - rows)
                if take <= 0:
                    break
                batch.append((r, done[r], take))
                rows += take
            ks, vs = zip(*[t.suffix(r, w, lo, lo + n) for r, lo, n in batch])
            self.ctx.kv_append([r for r, _, _ in batch], [n for _, _, n in batch],
                               torch.cat(ks), torch.cat(vs))
            for r, lo, n in batch:
                done[r] += n
            pending = [r for r in pending if done[r] < w.req_ctx[r]]
        torch.cuda.synchronize(self.device)

    # ------------------------------------------------------------------ steps
    def decode_inputs(self, reqs=None):
        """q, k_new, v_new of a decode step over `reqs` (positions into
        decode_requests(); default all)."""
        w, t = self.w, self.t
        pos = list(range(len(self.dec))) if reqs is None else list(reqs)
        ids = [self.dec[i] for i in pos]
        rows = [t.suffix_off[r] + w.req_ctx[r] + w.req_prefill[r] for r in ids]
        idx = torch.tensor(rows, device=t.suffix_k.device, dtype=torch.long)
        q = t.q_decode[torch.tensor(pos, device=t.q_decode.device, dtype=torch.long)]
        return ids, q.contiguous(), t.suffix_k[idx].contiguous(), t.suffix_v[idx].contiguous()

    def new_outputs(self, rows):
        w = self.w
        out = torch.empty(rows, w.num_q_heads, w.head_dim, dtype=torch.bfloat16, device=self.device)
        lse = torch.empty(rows, w.num_q_heads, dtype=torch.float32, device=self.device)
        return out, lse

    def decode(self, ids, q, k_new, v_new, out, lse, stream=None):
        self.ctx.decode(ids, q, k_new, v_new, out, lse, stream)

    def prefill_inputs(self, rnd):
        w, t = self.w, self.t
        chunks = w.chunks_of_round(rnd)
        ids = [r for r, _, _ in chunks]
        lens = [c for _, _, c in chunks]
        qs, ks, vs = [], [], []
        for r, off, c in chunks:
            q0 = t.qpf_off[r] + (off - w.req_ctx[r])
            qs.append(t.q_prefill[q0:q0 + c])
            k, v = t.suffix(r, w, off, off + c)
            ks.append(k)
            vs.append(v)
        return chunks, ids, lens, torch.cat(qs), torch.cat(ks), torch.cat(vs)

    def prefill(self, ids, lens, q, k, v, out, lse, stream=None):
        self.ctx.prefill_chunk(ids, lens, q, k, v, out, lse, stream)

    # ------------------------------------------------------------- movement
    def offload_for_reload(self, agents=None):
        """Copy the given prefixes to pinned host memory and evict them, so
        a later step can reload them (the paper's prefix movement)."""
        w, t = self.w, self.t
        agents = w.reload_agents if agents is None else agents
        for a in agents:
            k, v = t.prefix(a, w)
            hk = torch.empty(k.shape, dtype=k.dtype, pin_memory=True)
            hv = torch.empty(v.shape, dtype=v.dtype, pin_memory=True)
            hk.copy_(k)
            hv.copy_(v)
            self.host_prefix[a] = (hk, hv)
            self.ctx.prefix_evict(a)
        torch.cuda.synchronize(self.device)

    def reload(self, agents=None, side_stream=None, done_event=None):
        agents = self.w.reload_agents if agents is None else agents
        for a in agents:
            hk, hv = self.host_prefix[a]
            self.ctx.prefix_reload(a, hk, hv, side_stream, done_event)
