"""Pins of the fp64 oracle against facts that do not come from the oracle.

Each pin is checked against something fixed outside the oracle's code:
hand-derived closed forms (tests/golden/closed_forms.json), a brute-force
high-precision evaluation of the definition with mpmath on tiny inputs,
torch's own scaled_dot_product_attention (a library routine) in float64,
and invariants of the mathematics (weights sum to one, split-and-merge
equals single pass).  test_planted_mistakes_are_caught shows that typical
mistakes planted into the oracle (wrong scale, dropped term, wrong sign,
wrong head mapping, wrong causal diagonal, missing decode token) each make
at least one pin fail.
"""
import json
import math
import os

import numpy as np
import pytest

import oracle
from oracle import attention as A

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "closed_forms.json")


def _num(x):
    if isinstance(x, str):
        table = {"2ln3": 2 * math.log(3), "ln4": math.log(4), "ln5": math.log(5),
                 "ln6": math.log(6), "ln8": math.log(8)}
        return table[x]
    return float(x)


def _arr(rows):
    return np.array([[_num(x) for x in r] for r in rows], np.float64)


# ---------------------------------------------------------------- pins ----

def pin_closed_forms_attend():
    g = json.load(open(GOLDEN))
    for case in g["attend"]:
        o, lse = A.attend(_arr(case["q"]), _arr(case["k"]), _arr(case["v"]))
        np.testing.assert_allclose(o, _arr(case["o"]), rtol=0, atol=1e-12, err_msg=case["name"])
        np.testing.assert_allclose(lse, [_num(x) for x in case["lse"]], rtol=0, atol=1e-12,
                                   err_msg=case["name"])


def pin_closed_form_decode():
    c = json.load(open(GOLDEN))["decode"]
    hq, hkv, d, lp, ns = c["Hq"], c["Hkv"], c["d"], c["prefix_len"], c["cached"]
    L = lp + ns + 1
    rng = np.random.default_rng(11)
    K = rng.standard_normal((L, hkv, d))
    V = np.zeros((L, hkv, d))
    for j in range(L):
        V[j, 0, :] = j
        V[j, 1, :] = 100 + j
    o, lse = A.decode_step(np.zeros((hq, d)), K[:lp], V[:lp], K[lp:lp + ns], V[lp:lp + ns],
                           K[L - 1], V[L - 1])
    np.testing.assert_allclose(o, np.array(c["o_head"])[:, None] * np.ones((1, d)), atol=1e-12)
    np.testing.assert_allclose(lse, [_num(c["lse"])] * hq, atol=1e-12)


def pin_closed_form_prefill():
    c = json.load(open(GOLDEN))["prefill"]
    hq, hkv, d, lp, off, ch = c["Hq"], c["Hkv"], c["d"], c["prefix_len"], c["cached"], c["chunk"]
    L = lp + off + ch
    rng = np.random.default_rng(12)
    K = rng.standard_normal((L, hkv, d))
    V = np.arange(L, dtype=np.float64)[:, None, None] * np.ones((1, hkv, d))
    o, lse = A.prefill_chunk(np.zeros((ch, hq, d)), K[:lp], V[:lp], K[lp:lp + off],
                             V[lp:lp + off], K[lp + off:], V[lp + off:])
    for i in range(ch):
        np.testing.assert_allclose(o[i], c["o_row"][i], atol=1e-12)
        np.testing.assert_allclose(lse[i], _num(c["lse_row"][i]), atol=1e-12)


def _brute_mp(q, k, v):
    """Definition evaluated element by element in 50-digit arithmetic."""
    import mpmath
    mpmath.mp.dps = 50
    n, d = q.shape
    m = k.shape[0]
    o = np.zeros((n, v.shape[1]))
    lse = np.zeros(n)
    for i in range(n):
        s = [mpmath.fsum(mpmath.mpf(float(q[i, t])) * mpmath.mpf(float(k[j, t]))
                         for t in range(d)) / mpmath.sqrt(d) for j in range(m)]
        w = [mpmath.e ** sj for sj in s]
        tot = mpmath.fsum(w)
        for c in range(v.shape[1]):
            o[i, c] = float(mpmath.fsum(w[j] * mpmath.mpf(float(v[j, c])) for j in range(m)) / tot)
        lse[i] = float(mpmath.log(tot))
    return o, lse


def pin_brute_force_tiny():
    rng = np.random.default_rng(5)
    for m in range(1, 9):
        d = int(rng.integers(1, 9))
        q = rng.standard_normal((3, d)) * 2
        k = rng.standard_normal((m, d))
        v = rng.standard_normal((m, 5))
        o, lse = A.attend(q, k, v)
        ob, lb = _brute_mp(q, k, v)
        np.testing.assert_allclose(o, ob, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, lb, rtol=0, atol=1e-12)


def pin_weights_sum_to_one():
    # with one-hot values the output row IS the weight vector
    rng = np.random.default_rng(6)
    m, d = 37, 16
    q = rng.standard_normal((4, d)) * 3
    k = rng.standard_normal((m, d))
    o, lse = A.attend(q, k, np.eye(m))
    assert np.all(o >= 0)
    np.testing.assert_allclose(o.sum(axis=1), 1.0, atol=1e-12)
    # and each weight equals exp(s_j - lse)
    s = (q @ k.T) / math.sqrt(d)
    np.testing.assert_allclose(o, np.exp(s - lse[:, None]), rtol=1e-12, atol=1e-15)


def pin_split_merge_equals_single_pass():
    rng = np.random.default_rng(7)
    m, d = 300, 32
    q = rng.standard_normal((6, d)) * 2
    k = rng.standard_normal((m, d))
    v = rng.standard_normal((m, d))
    o, lse = A.attend(q, k, v)
    for parts in (2, 3, 7):
        cuts = np.sort(rng.choice(np.arange(1, m), size=parts - 1, replace=False))
        bounds = [0, *cuts.tolist(), m]
        pieces = [A.attend(q, k[a:b], v[a:b]) for a, b in zip(bounds[:-1], bounds[1:])]
        om, lm = A.lse_merge(pieces)
        np.testing.assert_allclose(om, o, rtol=0, atol=1e-12)
        np.testing.assert_allclose(lm, lse, rtol=0, atol=1e-12)


def pin_torch_sdpa():
    """torch's SDPA (float64, CPU, explicit boolean mask, grouped kv heads)
    must agree with the oracle's decode and prefill drivers."""
    torch = pytest.importorskip("torch")
    F = torch.nn.functional
    rng = np.random.default_rng(8)
    hq, hkv, d, lp, off, ch = 8, 2, 16, 23, 9, 13
    L = lp + off + ch
    K = rng.standard_normal((L, hkv, d))
    V = rng.standard_normal((L, hkv, d))
    q = rng.standard_normal((ch, hq, d)) * 2
    o, _ = A.prefill_chunk(q, K[:lp], V[:lp], K[lp:lp + off], V[lp:lp + off],
                           K[lp + off:], V[lp + off:])
    key = torch.arange(L)[None, :]
    row = torch.arange(ch)[:, None]
    mask = (key < lp) | (key - lp <= off + row)
    ref = F.scaled_dot_product_attention(
        torch.from_numpy(q).permute(1, 0, 2)[None], torch.from_numpy(K).permute(1, 0, 2)[None],
        torch.from_numpy(V).permute(1, 0, 2)[None], attn_mask=mask, enable_gqa=True)
    np.testing.assert_allclose(o, ref[0].permute(1, 0, 2).numpy(), rtol=0, atol=1e-12)
    # decode: one query over all L keys (the last one is the new token)
    qd = rng.standard_normal((hq, d))
    od, _ = A.decode_step(qd, K[:lp], V[:lp], K[lp:L - 1], V[lp:L - 1], K[L - 1], V[L - 1])
    refd = F.scaled_dot_product_attention(
        torch.from_numpy(qd)[:, None, :][None], torch.from_numpy(K).permute(1, 0, 2)[None],
        torch.from_numpy(V).permute(1, 0, 2)[None], enable_gqa=True)
    np.testing.assert_allclose(od, refd[0, :, 0, :].numpy(), rtol=0, atol=1e-12)


def pin_empty_prefix_is_plain_attention():
    rng = np.random.default_rng(9)
    hq, hkv, d, n = 4, 1, 8, 10
    K = rng.standard_normal((n + 1, hkv, d))
    V = rng.standard_normal((n + 1, hkv, d))
    q = rng.standard_normal((hq, d))
    o, lse = A.decode_step(q, K[:0], V[:0], K[:n], V[:n], K[n], V[n])
    ob, lb = _brute_mp(q, K[:, 0], V[:, 0])
    np.testing.assert_allclose(o, ob, atol=1e-12)
    np.testing.assert_allclose(lse, lb, atol=1e-12)


PINS = [pin_closed_forms_attend, pin_closed_form_decode, pin_closed_form_prefill,
        pin_brute_force_tiny, pin_weights_sum_to_one, pin_split_merge_equals_single_pass,
        pin_torch_sdpa, pin_empty_prefix_is_plain_attention]


@pytest.mark.parametrize("pin", PINS, ids=[p.__name__ for p in PINS])
def test_pin(pin):
    pin()


# ------------------------------------------------- planted mistakes -----

def _attend_factory(mistake):
    def attend(q, k, v, visible=None, scale=None):
        q = np.asarray(q, np.float64); k = np.asarray(k, np.float64); v = np.asarray(v, np.float64)
        d = q.shape[1]
        sc = (1.0 / d) if mistake == "scale_1_over_d" else 1.0 / np.sqrt(d)
        s = (q @ k.T) * sc
        if visible is not None:
            s = np.where(visible, s, -np.inf)
        m = s.max(axis=1, keepdims=True)
        w = np.exp(m - s) if mistake == "sign" else np.exp(s - m)
        if visible is not None and mistake == "sign":
            w = np.where(visible, w, 0.0)
        l = w.sum(axis=1, keepdims=True)
        o = (w @ v) if mistake == "no_normalise" else (w @ v) / l
        lse = np.log(l[:, 0]) if mistake == "lse_drops_max" else m[:, 0] + np.log(l[:, 0])
        if mistake == "lse_log2":
            lse = m[:, 0] + np.log2(l[:, 0])
        return o, lse
    return attend


def _merge_without_weights(parts):
    os_ = np.stack([np.asarray(p[0], np.float64) for p in parts])
    lses = np.stack([np.asarray(p[1], np.float64) for p in parts])
    return os_.mean(axis=0), lses.max(axis=0)


def _prefill_excluding_diagonal(q, prefix_k, prefix_v, suffix_k, suffix_v, k_new, v_new):
    q = np.asarray(q)
    lp, off, c = np.asarray(prefix_k).shape[0], np.asarray(suffix_k).shape[0], q.shape[0]
    K = np.concatenate([prefix_k, suffix_k, k_new], 0)
    V = np.concatenate([prefix_v, suffix_v, v_new], 0)
    key = np.arange(K.shape[0])[None, :]
    row = np.arange(c)[:, None]
    visible = (key < lp) | (key - lp < off + row + (1 if off + lp == 0 else 0))
    visible[:, 0] = True
    return A._heads_attend(q, K, V, visible)


def _decode_without_new_token(q, prefix_k, prefix_v, suffix_k, suffix_v, k_new, v_new):
    K = np.concatenate([prefix_k, suffix_k], 0)
    V = np.concatenate([prefix_v, suffix_v], 0)
    o, lse = A._heads_attend(np.asarray(q)[None], K, V)
    return o[0], lse[0]


MISTAKES = {
    "scale_1_over_d": ("attend", _attend_factory("scale_1_over_d")),
    "sign": ("attend", _attend_factory("sign")),
    "no_normalise": ("attend", _attend_factory("no_normalise")),
    "lse_drops_max": ("attend", _attend_factory("lse_drops_max")),
    "lse_log2": ("attend", _attend_factory("lse_log2")),
    "gqa_interleaved": ("kv_head_of", lambda h, hq, hkv: h % hkv),
    "merge_unweighted": ("lse_merge", _merge_without_weights),
    "causal_no_diagonal": ("prefill_chunk", _prefill_excluding_diagonal),
    "decode_skips_new_token": ("decode_step", _decode_without_new_token),
}


@pytest.mark.parametrize("name", sorted(MISTAKES))
def test_planted_mistakes_are_caught(name, monkeypatch):
    attr, fn = MISTAKES[name]
    monkeypatch.setattr(A, attr, fn)
    failed = []
    for pin in PINS:
        try:
            pin()
        except (AssertionError, ValueError, FloatingPointError):
            failed.append(pin.__name__)
    assert failed, f"planted mistake {name!r} passed every pin"
