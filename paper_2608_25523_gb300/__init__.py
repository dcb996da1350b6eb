"""GB300 (sm_103a) shared-prefix paged attention: C-ABI CUDA library plus a
thin ctypes binding.

    build        compile libtopas_attn.so in-tree (nvcc, sm_103a)
    binding      the C ABI of include/topas_attn.h, same names
    session      drives a synthetic multi-agent serving workload through it
    workloads    seeded synthetic inputs (structure and bf16 values only)
"""
__all__ = ["build", "binding", "session", "workloads"]
