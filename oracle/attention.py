"""fp64 CPU oracle for shared-prefix paged attention.

TEST INFRASTRUCTURE.  Only tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline / reference leg may import this module.  The CUDA library never
calls it, and it shares no code, header or table with the library.

What is computed.  The paper (TOPAS) serves requests of agent a that share a
static system-prompt prefix of length ell_a whose KV cache is resident once
per agent, while every request r adds its own dynamic suffix, retained output
tokens and decode tokens on top (Sec. I: requests of one agent walk the same
static path of the prefix cache and append request-specific content;
Sec. III, Eq. 2: the prefix is paid once per agent plus d_r(t) per request).
The attention those requests run is therefore ordinary attention over the
request's own key sequence

    K_r = [ K_prefix(a(r)) ; K_suffix(r) ]      (and likewise V_r)

The paper states no attention formula (Sec. VI cites FlashAttention,
PagedAttention and chunked prefill for the kernels), so the textbook
definition is used, in float64, over fully materialised per-request K/V:

    s_j = <q, k_j> / sqrt(d)            for every visible key j
    m   = max_j s_j
    w_j = exp(s_j - m)
    o   = sum_j w_j v_j / sum_j w_j
    lse = m + ln(sum_j w_j)             (natural logarithm)

Readings where the paper is silent (the paper prints no attention arithmetic):
  * scale 1/sqrt(d); inputs are post-rotary, synthetic;
  * grouped-query attention: q head h reads kv head h // (Hq / Hkv);
  * decode appends the new token's K/V first, then attends to all
    ell_a + |suffix| + 1 keys, itself included;
  * a prefill chunk at suffix offset o attends to the whole prefix and to
    suffix positions 0 .. o + i for its row i (causal, diagonal included);
  * the prefix may be empty (plain attention over the suffix).

Everything here is the definition written out; the only library primitive is
numpy's matrix product.  Rows are processed in blocks only to bound memory;
blocking over rows does not change any row's arithmetic.
"""
from __future__ import annotations

import numpy as np

ROW_BLOCK = 512


def attend(q, k, v, visible=None, scale=None):
    """Attention of query rows q [n, d] over keys k [m, d] and values v [m, dv].

    visible: optional bool [n, m]; False hides key j from row i.  Every row
    must see at least one key (in the method a row always sees its own
    position or the prefix).  Returns (o [n, dv], lse [n]) in float64.
    """
    q = np.asarray(q, dtype=np.float64)
    k = np.asarray(k, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    if scale is None:
        scale = 1.0 / np.sqrt(q.shape[1])
    s = (q @ k.T) * scale
    if visible is not None:
        s = np.where(visible, s, -np.inf)
    m = s.max(axis=1, keepdims=True)
    if not np.all(np.isfinite(m)):
        raise ValueError("a query row sees no key")
    w = np.exp(s - m)
    l = w.sum(axis=1, keepdims=True)
    o = (w @ v) / l
    lse = m[:, 0] + np.log(l[:, 0])
    return o, lse


def lse_merge(parts):
    """Exact combination of attention results over disjoint key subsets.

    parts: list of (o_i [n, dv], lse_i [n]) where o_i is the normalised
    attention over subset i.  With M = max_i lse_i and c_i = exp(lse_i - M):
        o = sum_i c_i o_i / sum_i c_i,   lse = M + ln(sum_i c_i).
    This is the algebra that lets split-KV and two-level (prefix / suffix)
    attention equal single-pass attention.
    """
    lses = np.stack([np.asarray(p[1], np.float64) for p in parts])      # [k, n]
    os_ = np.stack([np.asarray(p[0], np.float64) for p in parts])       # [k, n, dv]
    mx = lses.max(axis=0)
    c = np.exp(lses - mx)
    tot = c.sum(axis=0)
    o = (c[:, :, None] * os_).sum(axis=0) / tot[:, None]
    return o, mx + np.log(tot)


def kv_head_of(h, num_q_heads, num_kv_heads):
    """Grouped-query mapping: consecutive groups of Hq/Hkv q heads share one kv head."""
    return h // (num_q_heads // num_kv_heads)


def _heads_attend(q, K, V, visible_rows=None):
    """q [n, Hq, d]; K, V [L, Hkv, d]; visible_rows: bool [n, L] or None.
    Each q head attends through its kv head; returns o [n, Hq, d], lse [n, Hq]."""
    n, hq, d = q.shape
    hkv = K.shape[1]
    o = np.empty((n, hq, V.shape[2]), np.float64)
    lse = np.empty((n, hq), np.float64)
    for h in range(hq):
        g = kv_head_of(h, hq, hkv)
        Kg = np.asarray(K[:, g, :], np.float64)
        Vg = np.asarray(V[:, g, :], np.float64)
        for i0 in range(0, n, ROW_BLOCK):
            i1 = min(n, i0 + ROW_BLOCK)
            vis = None if visible_rows is None else visible_rows[i0:i1]
            o[i0:i1, h], lse[i0:i1, h] = attend(q[i0:i1, h, :], Kg, Vg, vis)
    return o, lse


def decode_step(q, prefix_k, prefix_v, suffix_k, suffix_v, k_new, v_new):
    """One decode step of one request.

    q [Hq, d]; prefix_k/v [ell_a, Hkv, d]; suffix_k/v [n_s, Hkv, d] cached
    before the step; k_new/v_new [Hkv, d] of the decoded token.  The token's
    K/V is appended first, so the query sees ell_a + n_s + 1 keys.
    Returns (o [Hq, d], lse [Hq]).
    """
    K = np.concatenate([np.asarray(prefix_k), np.asarray(suffix_k), np.asarray(k_new)[None]], 0)
    V = np.concatenate([np.asarray(prefix_v), np.asarray(suffix_v), np.asarray(v_new)[None]], 0)
    o, lse = _heads_attend(np.asarray(q)[None], K, V)
    return o[0], lse[0]


def prefill_chunk(q, prefix_k, prefix_v, suffix_k, suffix_v, k_new, v_new):
    """One prefill chunk of one request.

    q [c, Hq, d] are the chunk's queries at suffix positions o .. o+c-1,
    where o = len(suffix_k) tokens were cached before the chunk;
    k_new/v_new [c, Hkv, d] are the chunk's own K/V (appended first).
    Row i sees every prefix key and suffix positions 0 .. o + i.
    Returns (o [c, Hq, d], lse [c, Hq]).
    """
    q = np.asarray(q)
    lp = np.asarray(prefix_k).shape[0]
    off = np.asarray(suffix_k).shape[0]
    c = q.shape[0]
    K = np.concatenate([np.asarray(prefix_k), np.asarray(suffix_k), np.asarray(k_new)], 0)
    V = np.concatenate([np.asarray(prefix_v), np.asarray(suffix_v), np.asarray(v_new)], 0)
    L = K.shape[0]
    key = np.arange(L)[None, :]
    row = np.arange(c)[:, None]
    visible = (key < lp) | (key - lp <= off + row)
    return _heads_attend(q, K, V, visible)


# --------------------------------------------------------------------------
# whole-workload drivers (inputs come from the seeded generator)
# --------------------------------------------------------------------------

def workload_decode(w, t, requests=None):
    """Decode outputs of the workload's decode requests (or a subset, given
    as positions into w.decode_requests()).  Returns dict pos -> (o, lse)."""
    dec = w.decode_requests()
    pos = range(len(dec)) if requests is None else requests
    out = {}
    for i in pos:
        r = dec[i]
        a = w.req_agent[r]
        pk, pv = t.prefix(a, w)
        n_cached = w.req_ctx[r] + w.req_prefill[r]
        sk, sv = t.suffix(r, w, 0, n_cached)
        nk, nv = t.suffix(r, w, n_cached, n_cached + 1)
        out[i] = decode_step(t.q_decode[i], pk, pv, sk, sv, nk[0], nv[0])
    return out


def workload_prefill_chunk(w, t, r, offset, length):
    """Outputs of request r's prefill chunk covering suffix positions
    offset .. offset+length-1."""
    a = w.req_agent[r]
    pk, pv = t.prefix(a, w)
    sk, sv = t.suffix(r, w, 0, offset)
    nk, nv = t.suffix(r, w, offset, offset + length)
    q0 = t.qpf_off[r] + (offset - w.req_ctx[r])
    q = t.q_prefill[q0:q0 + length]
    return prefill_chunk(q, pk, pv, sk, sv, nk, nv)
