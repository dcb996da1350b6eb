"""ctypes binding of libtopas_attn.so (include/topas_attn.h).

Argument marshalling only: every step of the attention path runs in the
library's CUDA kernels.  Loading fails loudly when the library has not been
built; there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
import re
from ctypes import POINTER, c_char_p, c_int, c_int32, c_int64, c_size_t, c_uint32, c_uint64, c_void_p

from .build import HEADER, LIB

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
}

_lib = None


def header_functions() -> list:
    """Names of the functions include/topas_attn.h declares."""
    text = open(HEADER).read()
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
