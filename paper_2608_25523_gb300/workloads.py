"""Seeded synthetic workloads shaped like multi-agent serving.

This module only draws inputs: request structure (agents, prefix lengths,
suffix lengths, chunking) and bf16-valued Q/K/V.  It holds none of the
attention arithmetic, so both the CUDA library's tests and the fp64 oracle
can consume the same inputs without sharing any computation.

Structure follows the paper's setting: every request belongs to one agent
a(r) whose static system-prompt prefix of length ell_a is shared by all of
that agent's requests, and each request carries its own dynamic suffix plus
decode tokens (Sec. III, the joint prefix-request state and Eq. 2).  The
five named workloads below stand in for the paper's serving workloads
(Sec. V-A, Qwen2.5-32B on SGLang with MetaGPT prompts), which are neither
reproducible nor needed here: only the shapes matter to the attention path.

Values: Q, K, V ~ N(0, 1) drawn in float32 and rounded to bf16
(round-to-nearest-even).  Small workloads are drawn with numpy's PCG64
(`tensors_numpy`); the large ones are drawn on the device with a seeded
torch generator (`tensors_torch`) because numpy would need minutes and tens
of GB of host memory for them.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np

PAGE = 16


@dataclass
class Workload:
    name: str
    seed: int
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    prefix_len: list            # ell_a per agent (tokens)
    req_agent: list             # a(r) per request
    req_ctx: list               # suffix tokens already cached before the timed step
    req_prefill: list           # suffix tokens prefilled in this workload (chunked)
    req_decode: list            # 1 if the request takes one decode step, else 0
    chunk: int = 512            # prefill chunk size (tokens)
    reload_agents: list = field(default_factory=list)  # prefixes reloaded from pinned host
    permute_pages: bool = False  # free-page order randomly permuted (fragmented pool)
    q_scale: float = 1.0        # >1 sharpens the softmax ("sharp" parity variant)
    page_order_seed: int = 0    # seed of the free-list permutation when permute_pages

    # derived sizes -------------------------------------------------------
    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def num_agents(self) -> int:
        return len(self.prefix_len)

    @property
    def num_requests(self) -> int:
        return len(self.req_agent)

    def req_total(self, r: int) -> int:
        return self.req_ctx[r] + self.req_prefill[r] + self.req_decode[r]

    def decode_requests(self) -> list:
        return [r for r in range(self.num_requests) if self.req_decode[r]]

    def prefill_requests(self) -> list:
        return [r for r in range(self.num_requests) if self.req_prefill[r]]

    def kv_bytes_per_token(self) -> int:
        # K and V, bf16, all kv heads: the per-layer analogue of the paper's mu
        return 2 * self.num_kv_heads * self.head_dim * 2

    def pages_needed(self) -> int:
        n = sum(-(-l // PAGE) for l in self.prefix_len)
        n += sum(-(-self.req_total(r) // PAGE) for r in range(self.num_requests))
        return n

    def prefill_rounds(self) -> int:
        return max([-(-p // self.chunk) for p in self.req_prefill] + [0])

    def chunks_of_round(self, rnd: int):
        """(request, suffix offset, chunk length) of every chunk in round `rnd`."""
        out = []
        for r in range(self.num_requests):
            p = self.req_prefill[r]
            lo = rnd * self.chunk
            if lo < p:
                out.append((r, self.req_ctx[r] + lo, min(self.chunk, p - lo)))
        return out


def _uniform_int(rng, lo, hi, n):
    """n integers uniform on [lo, hi], both ends included."""
    return [int(x) for x in rng.integers(lo, hi + 1, size=n)]


def config(index: int) -> Workload:
    """The five named workloads, index 0..4, each with its fixed seed."""
    if index == 0:
        # Tiny: 1 agent, 256-token prefix, 4 requests with a 64-token suffix
        # prefilled in one chunk and then one decode step; Hq=8, Hkv=2, d=64.
        return Workload("tiny", 0, 8, 2, 64, [256], [0] * 4, [0] * 4, [64] * 4,
                        [1] * 4, chunk=64)
    if index == 1:
        # Llama-3-8B attention layer, decode: 4 agents x 4096-token prefixes,
        # 16 requests each, cached suffixes uniform in 256..1024.
        rng = np.random.default_rng(1)
        agents = [a for a in range(4) for _ in range(16)]
        ctx = _uniform_int(rng, 256, 1024, 64)
        return Workload("llama3_8b_decode", 1, 32, 8, 128, [4096] * 4, agents, ctx,
                        [0] * 64, [1] * 64)
    if index == 2:
        # Chunked prefill, same layer: 8 agents with prefixes uniform in
        # 2048..8192, 32 new requests each prefilling 512..2048 suffix tokens
        # in 512-token chunks.
        rng = np.random.default_rng(2)
        plen = _uniform_int(rng, 2048, 8192, 8)
        agents = [a for a in range(8) for _ in range(32)]
        pf = _uniform_int(rng, 512, 2048, 256)
        return Workload("chunked_prefill", 2, 32, 8, 128, plen, agents, [0] * 256, pf,
                        [0] * 256, chunk=512)
    if index == 3:
        # Mixed batch: 16 agents with prefixes 1024..8192, 256 decode requests
        # assigned by a Zipf(1.1) law over agent ranks 1..16 (cached suffixes
        # 256..1024), plus 8 new requests prefilling one 1024-token chunk;
        # fragmented (permuted) pool; 2 prefixes reloaded from pinned host.
        rng = np.random.default_rng(3)
        plen = _uniform_int(rng, 1024, 8192, 16)
        p = np.arange(1, 17, dtype=np.float64) ** -1.1
        p /= p.sum()
        dec_agents = [int(a) for a in rng.choice(16, size=256, p=p)]
        ctx = _uniform_int(rng, 256, 1024, 256)
        pf_agents = [int(a) for a in rng.choice(16, size=8, p=p)]
        active = sorted(set(dec_agents))
        reload = [int(a) for a in rng.choice(active, size=2, replace=False)]
        agents = dec_agents + pf_agents
        return Workload("mixed", 3, 32, 8, 128, plen, agents, ctx + [0] * 8,
                        [0] * 256 + [1024] * 8, [1] * 256 + [0] * 8, chunk=1024,
                        reload_agents=reload, permute_pages=True, page_order_seed=3)
    if index == 4:
        # Llama-3-70B attention layer, decode: 6 agents x 16384-token
        # prefixes, 512 requests split 86,86,85,85,85,85, cached suffixes
        # uniform in 512..4096.
        rng = np.random.default_rng(4)
        counts = [86, 86, 85, 85, 85, 85]
        agents = [a for a in range(6) for _ in range(counts[a])]
        ctx = _uniform_int(rng, 512, 4096, 512)
        return Workload("llama3_70b_decode", 4, 64, 8, 128, [16384] * 6, agents, ctx,
                        [0] * 512, [1] * 512)
    raise ValueError(f"no workload {index}")


def small_case(seed, *, hq=8, hkv=2, d=128, prefix_len=(40,), req_agent=(0,),
               req_ctx=(0,), req_prefill=(0,), req_decode=(1,), chunk=64,
               permute=False, q_scale=1.0, reload_agents=()) -> Workload:
    """A free-form small workload for parity tests (sizes the oracle finishes
    in well under a second)."""
    return Workload(f"case{seed}", seed, hq, hkv, d, list(prefix_len), list(req_agent),
                    list(req_ctx), list(req_prefill), list(req_decode), chunk=chunk,
                    reload_agents=list(reload_agents), permute_pages=permute,
                    q_scale=q_scale, page_order_seed=seed + 1 if permute else 0)


def sharp(w: Workload, q_scale: float = 8.0) -> Workload:
    return replace(w, name=w.name + "_sharp", q_scale=q_scale)


# --------------------------------------------------------------------------
# bf16 values
# --------------------------------------------------------------------------

def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round float32 to the nearest bf16 (ties to even); returned as float32
    holding exactly the bf16 value.  Inputs are finite."""
    b = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    b = (b + (((b >> 16) & 1) + 0x7FFF)) & 0xFFFF0000
    return b.astype(np.uint32).view(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """uint16 bit patterns of float32 values that are already bf16-exact."""
    return (np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


@dataclass
class Tensors:
    """Flat bf16-valued tensors of a workload plus per-entity offsets.

    prefix_k/v  [sum ell_a, Hkv, d]   agent a at rows prefix_off[a] ...
    suffix_k/v  [sum total_r, Hkv, d] request r at rows suffix_off[r]; its
                first req_ctx[r] rows are cached context, then the prefill
                tokens, then (if it decodes) the decode token's K/V
    q_prefill   [sum prefill_r, Hq, d] request r at rows qpf_off[r]
    q_decode    [n_decode, Hq, d]      in the order of decode_requests()
    """
    prefix_k: object
    prefix_v: object
    suffix_k: object
    suffix_v: object
    q_prefill: object
    q_decode: object
    prefix_off: list
    suffix_off: list
    qpf_off: list

    def prefix(self, a, w):
        o = self.prefix_off[a]
        return self.prefix_k[o:o + w.prefix_len[a]], self.prefix_v[o:o + w.prefix_len[a]]

    def suffix(self, r, w, lo=0, hi=None):
        o = self.suffix_off[r]
        hi = w.req_total(r) if hi is None else hi
        return self.suffix_k[o + lo:o + hi], self.suffix_v[o + lo:o + hi]


def _offsets(sizes):
    off, acc = [], 0
    for s in sizes:
        off.append(acc)
        acc += s
    return off, acc


def tensors_numpy(w: Workload) -> Tensors:
    rng = np.random.default_rng([w.seed, 7])
    hkv, hq, d = w.num_kv_heads, w.num_q_heads, w.head_dim
    poff, pn = _offsets(w.prefix_len)
    soff, sn = _offsets([w.req_total(r) for r in range(w.num_requests)])
    qoff, qn = _offsets(w.req_prefill)
    nd = len(w.decode_requests())

    def draw(*shape, scale=1.0):
        x = rng.standard_normal(shape, dtype=np.float32)
        if scale != 1.0:
            x *= np.float32(scale)
        return bf16_round(x)

    return Tensors(draw(pn, hkv, d), draw(pn, hkv, d), draw(sn, hkv, d), draw(sn, hkv, d),
                   draw(qn, hq, d, scale=w.q_scale), draw(nd, hq, d, scale=w.q_scale),
                   poff, soff, qoff)


def tensors_torch(w: Workload, device) -> Tensors:
    """Same layout as tensors_numpy, drawn on `device` with a seeded torch
    generator (different values than the numpy draw)."""
    import torch
    g = torch.Generator(device=device)
    g.manual_seed(1_000_003 * w.seed + 17)
    hkv, hq, d = w.num_kv_heads, w.num_q_heads, w.head_dim
    poff, pn = _offsets(w.prefix_len)
    soff, sn = _offsets([w.req_total(r) for r in range(w.num_requests)])
    qoff, qn = _offsets(w.req_prefill)
    nd = len(w.decode_requests())

    def draw(*shape, scale=1.0):
        x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
        if scale != 1.0:
            x.mul_(scale)
        return x.to(torch.bfloat16)

    return Tensors(draw(pn, hkv, d), draw(pn, hkv, d), draw(sn, hkv, d), draw(sn, hkv, d),
                   draw(qn, hq, d, scale=w.q_scale), draw(nd, hq, d, scale=w.q_scale),
                   poff, soff, qoff)


def replicate(w: Workload, copies: int) -> Workload:
    """`copies` independent copies of a workload in one pool (agents and
    requests renumbered per copy).  Cycling a benchmark over the copies keeps
    the bytes touched between two visits of the same data far above the L2
    size, so every step reads its KV from HBM."""
    na, nr = w.num_agents, w.num_requests
    return replace(
        w, name=f"{w.name}_x{copies}",
        prefix_len=list(w.prefix_len) * copies,
        req_agent=[a + c * na for c in range(copies) for a in w.req_agent],
        req_ctx=list(w.req_ctx) * copies,
        req_prefill=list(w.req_prefill) * copies,
        req_decode=list(w.req_decode) * copies,
        reload_agents=[a + c * na for c in range(copies) for a in w.reload_agents])


def request_subset(w: Workload, stride: int) -> Workload:
    """Every `stride`-th request of a workload (all its agents kept): the
    same shapes and prefixes with fewer new tokens, for profiler captures
    that must hold little device memory."""
    keep = list(range(0, w.num_requests, stride))
    return replace(
        w, name=f"{w.name}_every{stride}",
        req_agent=[w.req_agent[r] for r in keep],
        req_ctx=[w.req_ctx[r] for r in keep],
        req_prefill=[w.req_prefill[r] for r in keep],
        req_decode=[w.req_decode[r] for r in keep])


def copy_requests(w: Workload, copies: int, c: int) -> list:
    """Request ids of copy `c` of replicate(w, copies)."""
    n = w.num_requests // copies
    return list(range(c * n, (c + 1) * n))
