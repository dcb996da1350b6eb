"""ctypes binding of libtopas_attn.so (include/topas_attn.h, include/topas_sched.h).

Argument marshalling only: every step of the attention path runs in the
library's CUDA kernels.  Loading fails loudly when the library has not been
built; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import re
from ctypes import (POINTER, c_char_p, c_double, c_int, c_int8, c_int32, c_int64, c_size_t, c_uint8,
                    c_uint32, c_uint64, c_void_p)

from .build import HEADER, LIB, SCHED_HEADER

# status codes
TPA_OK = 0
TPA_ERR_INVALID_ARG = 1
TPA_ERR_NO_SPACE = 2
TPA_ERR_NOT_RESIDENT = 3
TPA_ERR_STATE = 4
TPA_ERR_UNSUPPORTED = 5
TPA_ERR_CUDA = 6
TPA_ERR_TIMEOUT = 7
TPA_ERR_CAPACITY = 8
ERROR_NAMES = {0: "OK", 1: "INVALID_ARG", 2: "NO_SPACE", 3: "NOT_RESIDENT", 4: "STATE",
               5: "UNSUPPORTED", 6: "CUDA", 7: "TIMEOUT", 8: "CAPACITY"}

TPA_FLAG_PLAN_ONLY = 1

# tpa_query
Q_FREE_PAGES, Q_PREFIX_LEN, Q_PREFIX_RESIDENT, Q_SUFFIX_LEN, Q_NUM_SMS = 0, 1, 2, 3, 4
Q_LAST_DENSE_ITEMS, Q_LAST_SUFFIX_ITEMS, Q_LAST_LAUNCHES, Q_PAGE_OF = 5, 6, 7, 8
# tpa_set_option
OPT_DECODE_MODE, OPT_PREFIX_SPLITS, OPT_SUFFIX_SPLIT_KEYS = 0, 1, 2
OPT_KERNEL_TIMING = 4
OPT_TEST_PLAN_WAIT = 5
OPT_PREFILL_TILE_ROWS = 6
OPT_TEST_BAD_PAGE = 7
OPT_MOVEMENT_STAGED = 8
OPT_TEST_BAD_SLOT = 9
# kernel kinds of tpa_kernel_times
KERNEL_NAMES = ["kv_append", "dense_tcgen05", "split_kv", "lse_merge", "page_copy",
                "prefill_pair_tcgen05"]


class TpaError(RuntimeError):
    def __init__(self, code: int, msg: str):
        super().__init__(f"TPA_ERR_{ERROR_NAMES.get(code, code)}: {msg}")
        self.code = code


class Config(ctypes.Structure):
    _fields_ = [("num_q_heads", c_int32), ("num_kv_heads", c_int32), ("head_dim", c_int32),
                ("page_size", c_int32), ("num_pages", c_int64), ("k_pool", c_void_p),
                ("v_pool", c_void_p), ("workspace", c_void_p), ("workspace_bytes", c_size_t),
                ("max_agents", c_int32), ("max_requests", c_int32), ("max_tokens", c_int32),
                ("max_seq_len", c_int32), ("max_splits", c_int32), ("flags", c_int32),
                ("page_order_seed", c_uint64)]


_I32P = POINTER(c_int32)
class SchedParams(ctypes.Structure):
    _fields_ = [("budget", c_double), ("mu", c_double), ("b_swap", c_double), ("t_decode", c_double),
                ("beta", c_double), ("rho", c_double), ("h_age", c_double), ("M", c_int32),
                ("K", c_int32), ("mc_samples", c_int32), ("pad", c_int32), ("seed", c_uint64)]


class SchedSnapshot(ctypes.Structure):
    _fields_ = [("t", c_double), ("n_stages", c_int32), ("n_agents", c_int32), ("n_tasks", c_int32),
                ("n_reqs", c_int32), ("stage_agent", POINTER(c_int32)), ("pred_off", POINTER(c_int32)),
                ("pred_idx", POINTER(c_int32)), ("prefix_len", POINTER(c_int64)),
                ("sample_off", POINTER(c_int32)), ("samples", POINTER(c_double)),
                ("task_id", POINTER(c_uint64)), ("task_arrival", POINTER(c_double)),
                ("stage_state", POINTER(c_int8)), ("stage_served", POINTER(c_double)),
                ("req_task", POINTER(c_int32)), ("req_stage", POINTER(c_int32)),
                ("req_kv", POINTER(c_double)), ("req_dhat", POINTER(c_double)),
                ("req_redo", POINTER(c_double)), ("req_credit", POINTER(c_double)),
                ("req_running", POINTER(c_uint8)), ("resident", POINTER(c_uint8))]


class SchedDecision(ctypes.Structure):
    _fields_ = [("agents", POINTER(c_uint8)), ("running", POINTER(c_uint8)),
                ("admitted", POINTER(c_int32)), ("credits", POINTER(c_double)),
                ("n_admitted", c_int32), ("n_preempted", c_int32), ("score", c_double),
                ("j_admit", c_double), ("j_move", c_double), ("j_redo", c_double),
                ("j_revoke", c_double), ("v_reuse", c_double), ("n_candidates", c_int64)]


_SIGS = {
    "tpa_workspace_size": (c_size_t, [POINTER(Config)]),
    "tpa_create": (c_int, [POINTER(Config), POINTER(c_void_p)]),
    "tpa_destroy": (c_int, [c_void_p]),
    "tpa_prefix_register": (c_int, [c_void_p, c_int32, c_int32]),
    "tpa_prefix_write": (c_int, [c_void_p, c_int32, c_void_p, c_void_p, c_void_p]),
    "tpa_prefix_evict": (c_int, [c_void_p, c_int32]),
    "tpa_prefix_reload": (c_int, [c_void_p, c_int32, c_void_p, c_void_p, c_void_p, c_void_p]),
    "tpa_prefix_offload": (c_int, [c_void_p, c_int32, c_void_p, c_void_p, c_void_p, c_void_p]),
    "tpa_request_open": (c_int, [c_void_p, c_int32, c_int32]),
    "tpa_request_close": (c_int, [c_void_p, c_int32]),
    "tpa_request_truncate": (c_int, [c_void_p, c_int32, _I32P, _I32P]),
    "tpa_kv_append": (c_int, [c_void_p, c_int32, _I32P, _I32P, c_void_p, c_void_p, c_void_p]),
    "tpa_prefill_chunk": (c_int, [c_void_p, c_int32, _I32P, _I32P, c_void_p, c_void_p,
                                  c_void_p, c_void_p, c_void_p, c_void_p]),
    "tpa_decode": (c_int, [c_void_p, c_int32, _I32P, c_void_p, c_void_p, c_void_p, c_void_p,
                           c_void_p, c_void_p]),
    "tpa_decode_static_scratch": (c_int, [c_void_p, c_int32, _I32P, c_void_p, c_void_p,
                                          c_void_p, c_void_p, c_void_p, c_void_p]),
    "tpa_gather": (c_int, [c_void_p, c_int32, c_int32, c_void_p, c_void_p, c_void_p]),
    "tpa_query": (c_int, [c_void_p, c_int32, c_int32, POINTER(c_int64)]),
    "tpa_set_option": (c_int, [c_void_p, c_int32, c_int64]),
    "tpa_device_status": (c_int, [c_void_p, c_void_p, POINTER(c_uint32)]),
    "tpa_kernel_times": (c_int, [c_void_p, c_int32, POINTER(ctypes.c_double), POINTER(c_int64),
                                 c_int32]),
    "tpa_last_error": (c_char_p, []),
    "tpa_sched_decide": (c_int, [POINTER(SchedParams), POINTER(SchedSnapshot), POINTER(SchedDecision)]),
}

_lib = None


def header_functions() -> list:
    """Names of the functions include/topas_attn.h and include/topas_sched.h declare."""
    text = open(HEADER).read() + open(SCHED_HEADER).read()
    return sorted(set(re.findall(r"^TPA_API\s+[\w\s\*]+?\b(tpa_\w+)\s*\(", text, re.M)))


def load():
    """Load the built library (raises if it is missing)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} is not built: run paper_2608_25523_gb300.build.build()")
        lib = ctypes.CDLL(LIB)
        for name, (res, args) in _SIGS.items():
            f = getattr(lib, name)
            f.restype = res
            f.argtypes = args
        _lib = lib
    return _lib


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return x.data_ptr()
    raise TypeError(f"cannot pass {type(x)} as a pointer")


def _stream(s):
    if s is None:
        import torch
        return torch.cuda.current_stream().cuda_stream if torch.cuda.is_available() else None
    if isinstance(s, int):
        return s
    return s.cuda_stream


def _event(e):
    if e is None:
        return None
    if isinstance(e, int):
        return e
    if not e.cuda_event:
        # torch creates the CUDA event lazily on its first record; the library
        # records it again on the stream of the call
        e.record()
    return e.cuda_event


def _i32(vals):
    if isinstance(vals, ctypes.Array):
        return vals
    vals = list(int(v) for v in vals)
    return (c_int32 * max(1, len(vals)))(*vals)


class Context:
    """One library context (tpa_ctx) over caller-owned pools and workspace."""

    def __init__(self, cfg: Config, keep=()):
        self.lib = load()
        self._keep = keep  # device tensors that must outlive the context
        self.cfg = cfg
        h = c_void_p()
        self._check(self.lib.tpa_create(ctypes.byref(cfg), ctypes.byref(h)))
        self.handle = h

    # -- plumbing ---------------------------------------------------------
    def _check(self, rc):
        if rc != TPA_OK:
            raise TpaError(rc, self.lib.tpa_last_error().decode())
        return rc

    def close(self):
        if getattr(self, "handle", None):
            self.lib.tpa_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # -- C ABI, same names --------------------------------------------------
    def prefix_register(self, agent, length):
        return self._check(self.lib.tpa_prefix_register(self.handle, agent, length))

    def prefix_write(self, agent, k, v, stream=None):
        return self._check(self.lib.tpa_prefix_write(self.handle, agent, _ptr(k), _ptr(v),
                                                     _stream(stream)))

    def prefix_evict(self, agent):
        return self._check(self.lib.tpa_prefix_evict(self.handle, agent))

    def prefix_reload(self, agent, host_k, host_v, side_stream=None, done_event=None):
        return self._check(self.lib.tpa_prefix_reload(self.handle, agent, _ptr(host_k),
                                                      _ptr(host_v), _stream(side_stream),
                                                      _event(done_event)))

    def prefix_offload(self, agent, host_k, host_v, side_stream=None, done_event=None):
        return self._check(self.lib.tpa_prefix_offload(self.handle, agent, _ptr(host_k),
                                                       _ptr(host_v), _stream(side_stream),
                                                       _event(done_event)))

    def request_open(self, req, agent):
        return self._check(self.lib.tpa_request_open(self.handle, req, agent))

    def request_close(self, req):
        return self._check(self.lib.tpa_request_close(self.handle, req))

    def request_truncate(self, reqs, lens):
        return self._check(self.lib.tpa_request_truncate(self.handle, len(reqs), _i32(reqs),
                                                         _i32(lens)))

    def kv_append(self, reqs, ntok, k_new, v_new, stream=None):
        return self._check(self.lib.tpa_kv_append(self.handle, len(reqs), _i32(reqs), _i32(ntok),
                                                  _ptr(k_new), _ptr(v_new), _stream(stream)))

    def prefill_chunk(self, reqs, chunk_len, q, k_new, v_new, out, lse, stream=None):
        return self._check(self.lib.tpa_prefill_chunk(
            self.handle, len(reqs), _i32(reqs), _i32(chunk_len), _ptr(q), _ptr(k_new),
            _ptr(v_new), _ptr(out), _ptr(lse), _stream(stream)))

    def decode(self, reqs, q, k_new, v_new, out, lse, stream=None):
        return self._check(self.lib.tpa_decode(self.handle, len(reqs), _i32(reqs), _ptr(q),
                                               _ptr(k_new), _ptr(v_new), _ptr(out), _ptr(lse),
                                               _stream(stream)))

    def decode_static_scratch(self, reqs, q, k_new, v_new, out, lse, stream=None):
        """decode() with its split partials in the library's static device array."""
        return self._check(self.lib.tpa_decode_static_scratch(
            self.handle, len(reqs), _i32(reqs), _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(out),
            _ptr(lse), _stream(stream)))

    def gather(self, ident, is_request, k_out, v_out, stream=None):
        return self._check(self.lib.tpa_gather(self.handle, ident, 1 if is_request else 0,
                                               _ptr(k_out), _ptr(v_out), _stream(stream)))

    def query(self, what, ident=0):
        v = c_int64()
        self._check(self.lib.tpa_query(self.handle, what, ident, ctypes.byref(v)))
        return v.value

    def set_option(self, option, value):
        return self._check(self.lib.tpa_set_option(self.handle, option, value))

    def kernel_times(self, reset=False):
        """{kernel name: (total ms, launches)} accumulated while kernel timing is on."""
        n = len(KERNEL_NAMES)
        ms = (ctypes.c_double * n)()
        cnt = (c_int64 * n)()
        self._check(self.lib.tpa_kernel_times(self.handle, n, ms, cnt, 1 if reset else 0))
        return {KERNEL_NAMES[i]: (ms[i], cnt[i]) for i in range(n)}

    def device_status(self, stream=None):
        v = c_uint32()
        rc = self.lib.tpa_device_status(self.handle, _stream(stream), ctypes.byref(v))
        if rc not in (TPA_OK, TPA_ERR_TIMEOUT):
            self._check(rc)
        return v.value


def i32_array(vals):
    """Pre-built id array for repeated calls (skips per-call marshalling)."""
    return _i32(vals)


def make_config(*, num_q_heads, num_kv_heads, head_dim, num_pages, max_agents, max_requests,
                max_tokens, max_seq_len, max_splits=0, page_order_seed=0, flags=0,
                k_pool=None, v_pool=None, workspace=None, workspace_bytes=0) -> Config:
    return Config(num_q_heads, num_kv_heads, head_dim, 16, num_pages, _ptr(k_pool), _ptr(v_pool),
                  _ptr(workspace), workspace_bytes, max_agents, max_requests, max_tokens,
                  max_seq_len, max_splits, flags, page_order_seed)


def workspace_size(cfg: Config) -> int:
    return load().tpa_workspace_size(ctypes.byref(cfg))


def allocate(*, num_q_heads, num_kv_heads, head_dim, num_pages, max_agents, max_requests,
             max_tokens, max_seq_len, max_splits=0, page_order_seed=0, device="cuda") -> Context:
    """Allocate zeroed KV pools and a workspace with torch on `device` and
    create a context over them."""
    import torch
    shape = (num_pages, num_kv_heads, 16, head_dim)
    k_pool = torch.zeros(shape, dtype=torch.bfloat16, device=device)
    v_pool = torch.zeros(shape, dtype=torch.bfloat16, device=device)
    cfg = make_config(num_q_heads=num_q_heads, num_kv_heads=num_kv_heads, head_dim=head_dim,
                      num_pages=num_pages, max_agents=max_agents, max_requests=max_requests,
                      max_tokens=max_tokens, max_seq_len=max_seq_len, max_splits=max_splits,
                      page_order_seed=page_order_seed)
    ws_bytes = workspace_size(cfg)
    if ws_bytes == 0:
        raise TpaError(TPA_ERR_UNSUPPORTED, "unsupported configuration")
    ws = torch.empty(ws_bytes + 256, dtype=torch.uint8, device=device)
    base = (ws.data_ptr() + 255) // 256 * 256
    cfg.k_pool, cfg.v_pool = k_pool.data_ptr(), v_pool.data_ptr()
    cfg.workspace, cfg.workspace_bytes = base, ws_bytes
    ctx = Context(cfg, keep=(k_pool, v_pool, ws))
    ctx.k_pool, ctx.v_pool, ctx.workspace = k_pool, v_pool, ws
    return ctx


# ---------------------------------------------------------------- scheduler

def _arr(ctype, vals):
    vals = list(vals)
    return (ctype * max(1, len(vals)))(*vals)


def sched_decide(params, snap, repeat: int = 1) -> dict:
    """tpa_sched_decide (include/topas_sched.h).

    `params` and `snap` are any objects with the header's field names, the
    snapshot's per-stage predecessors and samples as `stage_preds` and
    `stage_samples` (lists of lists) and its [task][stage] arrays as lists of
    lists.  Returns the selected state: R' and Q' (sorted ids), the admitted
    requests in order with their credits, the preempted count and the score
    terms of Eq. 12.  With repeat > 1 the native call runs that many times
    on the marshalled arguments and `native_us` is its mean duration."""
    import time
    lib = load()
    ns, na, nt, nr = (len(snap.stage_agent), len(snap.prefix_len), len(snap.task_id),
                      len(snap.req_task))
    pred_off, pred_idx = [0], []
    for preds in snap.stage_preds:
        pred_idx += list(preds)
        pred_off.append(len(pred_idx))
    sample_off, samples = [0], []
    for xs in snap.stage_samples:
        samples += list(xs)
        sample_off.append(len(samples))
    keep = dict(
        stage_agent=_arr(c_int32, snap.stage_agent), pred_off=_arr(c_int32, pred_off),
        pred_idx=_arr(c_int32, pred_idx), prefix_len=_arr(c_int64, snap.prefix_len),
        sample_off=_arr(c_int32, sample_off), samples=_arr(c_double, samples),
        task_id=_arr(c_uint64, snap.task_id), task_arrival=_arr(c_double, snap.task_arrival),
        stage_state=_arr(c_int8, [x for row in snap.stage_state for x in row]),
        stage_served=_arr(c_double, [x for row in snap.stage_served for x in row]),
        req_task=_arr(c_int32, snap.req_task), req_stage=_arr(c_int32, snap.req_stage),
        req_kv=_arr(c_double, snap.req_kv), req_dhat=_arr(c_double, snap.req_dhat),
        req_redo=_arr(c_double, snap.req_redo), req_credit=_arr(c_double, snap.req_credit),
        req_running=_arr(c_uint8, [1 if x else 0 for x in snap.req_running]),
        resident=_arr(c_uint8, [1 if x else 0 for x in snap.resident]))
    cs = SchedSnapshot(snap.t, ns, na, nt, nr,
                       *(ctypes.cast(keep[f], ptype) for f, ptype in SchedSnapshot._fields_[5:]))
    cp = SchedParams(params.budget, params.mu, params.b_swap, params.t_decode, params.beta,
                     params.rho, params.h_age, params.M, params.K, params.mc_samples, 0,
                     params.seed)
    out_agents, out_running = (c_uint8 * na)(), (c_uint8 * max(1, nr))()
    out_adm, out_cred = (c_int32 * max(1, nr))(), (c_double * max(1, nr))()
    cd = SchedDecision(out_agents, out_running, out_adm, out_cred)
    t0 = time.perf_counter()
    for _ in range(max(1, repeat)):
        rc = lib.tpa_sched_decide(ctypes.byref(cp), ctypes.byref(cs), ctypes.byref(cd))
        if rc != TPA_OK:
            raise TpaError(rc, lib.tpa_last_error().decode())
    native_us = (time.perf_counter() - t0) / max(1, repeat) * 1e6
    n = cd.n_admitted
    return {"agents": tuple(a for a in range(na) if out_agents[a]),
            "running": tuple(r for r in range(nr) if out_running[r]),
            "admitted": tuple(out_adm[k] for k in range(n)),
            "credits": tuple(out_cred[k] for k in range(n)),
            "n_preempted": cd.n_preempted, "score": cd.score, "j_admit": cd.j_admit,
            "j_move": cd.j_move, "j_redo": cd.j_redo, "j_revoke": cd.j_revoke,
            "v_reuse": cd.v_reuse, "n_candidates": cd.n_candidates, "native_us": native_us}
