"""fp64 CPU oracle (test infrastructure only).

Imported only by tests/, __graft_entry__.smoke() and bench.py's CPU-baseline
and reference legs.  The CUDA library and its Python binding never import it.

attention  exact attention over materialised per-request KV (the hot path)
sched      one TOPAS scheduling decision from a state snapshot (Sec. IV),
           imported as `oracle.sched`
"""
from .attention import (attend, lse_merge, kv_head_of, decode_step, prefill_chunk,
                        workload_decode, workload_prefill_chunk)

__all__ = ["attend", "lse_merge", "kv_head_of", "decode_step", "prefill_chunk",
           "workload_decode", "workload_prefill_chunk"]
