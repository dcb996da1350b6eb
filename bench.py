"""Benchmark of shared-prefix paged attention on one GB300 (or N replicas).

Default workload: the Llama-3-8B attention layer decode step (32 q heads,
8 kv heads, head_dim 128, bf16): 4 agents with 4096-token prefixes, 64
decode requests (16 per agent) with cached suffixes uniform in 256..1024,
page size 16.  One step = one tpa_decode call over the 64 requests (host plan,
one upload, one persistent tcgen05 launch that appends the new tokens and
runs the stacked shared-prefix tiles and the per-request suffixes, and the
log-sum-exp merge launched as its programmatic dependent), followed by a
table-only truncate that drops
the appended token again so every step sees the same workload.  Four
independent copies of the workload are cycled so that ~0.94 GB of KV lies
between two visits of the same bytes (L2 is 129 MB): every step reads HBM.

value  = algorithmic bytes per step (each prefix once, each suffix once,
         Q, the new tokens' K/V in and out, O and LSE) / device time, GB/s.
e2e    = the same metric through the public call with host buffers: the
         step's q / k_new / v_new sit in pinned host memory and O / LSE go
         back to it, inside the timed region.  tpa_decode takes the host
         arrays themselves and its kernels move those bytes over the
         CPU-GPU link; the variant with copy-engine copies to and from
         device buffers is reported beside it (e2e.copy_engine).
Also reported (rank 0, N=1): the tcgen05 chunked-prefill workload
(TFLOP/s), the mixed workload (reload + prefill + Zipf decode, ms/step),
the Llama-3-70B decode workload (GB/s), each with its own roofline, the
prefix-movement calibration (reload / offload bandwidth, the paper's
mu / B_swap), the redo trade of a preempted suffix (decode steps vs
chunked prefill), a kernel-level analogue of the paper's co-residency
diagnostic (one vs two resident prefixes under one KV budget), and the
TOPAS scheduler driving the library on Chain-3 tasks (decision latency,
native and oracle).

Under torchrun every rank runs its own copy on its own GPU (the path has
no exchange step: replicas only); value aggregates all ranks over the
slowest rank's time.

--impl reference times the fp64 CPU oracle on this host's cores on a
bounded sample of the same workload and metric.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "decode KV HBM GB/s (% of peak) + prefill TFLOP/s, tokens/s at 1×GB300"
COPIES = 4


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained", d["bf16_tflops"]), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


# ------------------------------------------------------------ accounting --

# Sources of the unified decode kernel; the DRAM traffic recorded in its ncu
# summary counts only while they are unchanged.
KERNEL_SOURCES = ["k_dense.cu", "dense_common.cuh", "split_kv.cuh", "ptx.cuh", "plan.h", "kernels.h"]
PROFILE = os.path.join(ROOT, "profiles", "dense_tcgen05_c2_decode.md")


def kernel_source_hash():
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_25523_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic():
    """DRAM bytes (read + write) per launch of the unified decode kernel from
    the committed ncu summary, or None if it was taken on other sources."""
    try:
        vals = {}
        with open(PROFILE) as fh:
            for line in fh:
                if ":" in line and line.split(":")[0] in ("traffic_bytes_per_launch",
                                                          "kernel_sources_sha256_16"):
                    k, v = line.split(":", 1)
                    vals[k.strip()] = v.strip()
        if vals.get("kernel_sources_sha256_16") != kernel_source_hash():
            return None
        return int(vals["traffic_bytes_per_launch"])
    except (OSError, KeyError, ValueError):
        return None


def decode_bytes(w, reqs):
    """Algorithmic HBM bytes of one decode step over `reqs`: each distinct
    prefix once, each suffix (with the new token) once, Q in, the new
    tokens' K/V in and into the pool, O and LSE out."""
    mu = w.kv_bytes_per_token()
    agents = sorted({w.req_agent[r] for r in reqs})
    prefix = sum(w.prefix_len[a] for a in agents) * mu
    suffix = sum(w.req_ctx[r] + w.req_prefill[r] + 1 for r in reqs) * mu
    n = len(reqs)
    qo = 2 * n * w.num_q_heads * w.head_dim * 2 + n * w.num_q_heads * 4
    new = 2 * n * mu
    return prefix, suffix, prefix + suffix + qo + new


def prefill_flops(w, chunks):
    """Unmasked (query row, key) pairs x 4 d flops of the chunks (QK^T and PV)."""
    pairs = 0
    for r, off, c in chunks:
        lp = w.prefix_len[w.req_agent[r]]
        # positions off..off+c-1 see lp prefix keys and p+1 suffix keys
        pairs += c * lp + c * off + c * (c + 1) // 2
    return pairs * w.num_q_heads * 4 * w.head_dim


def job_rate(ms, units_per_rank, world, device):
    """Slowest rank's timed region (max over ranks) and the whole-job rate:
    the units all ranks processed over that time (per second)."""
    if world > 1:
        import torch
        import torch.distributed as dist
        t = torch.tensor([ms], device=device, dtype=torch.float64)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return ms, units_per_rank * world / (ms / 1e3)


# ---------------------------------------------------------------- clocks --

class Clocks:
    """nvidia-smi samples of SM clock and throttle reasons during a region."""
    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def start(self):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "20", "-i", str(self.index)], stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None
        time.sleep(0.3)  # first sample lands before the timed region starts
        self.t0 = time.time()

    def stop(self):
        self.t1 = time.time()
        time.sleep(0.05)
        if self.proc:
            self.proc.terminate()
            self.proc.wait()
        self.f.flush()
        rows = []
        for line in open(self.f.name):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                ts += float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                rows.append((ts, float(parts[1]), float(parts[2]), parts[5:9]))
            except (ValueError, IndexError):
                continue
        os.unlink(self.f.name)
        inside = [r for r in rows if self.t0 - 0.05 <= r[0] <= self.t1 + 0.05]
        if not inside and rows:
            inside = [min(rows, key=lambda r: abs(r[0] - (self.t0 + self.t1) / 2))]
        if not inside:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in inside for i, v in enumerate(r[3]) if v == "Active"})
        sm = sorted(r[1] for r in inside)
        return {"sm_mhz": sm[len(sm) // 2], "sm_max_mhz": max(r[2] for r in inside),
                "reasons": reasons, "samples": len(inside)}


# ------------------------------------------------------------- our arm ---

def run_ours(args, rank, world, local_rank):
    import torch
    import torch.distributed as dist

    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.build import build
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import config, copy_requests, replicate, tensors_torch

    build()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    hbm_peak, tf_peak, tf_sust, peak_src = peaks()

    base = config(1)
    w = replicate(base, COPIES)
    t = tensors_torch(w, dev)
    s = Session(w, t, device=dev, extra_tokens=16)
    n = base.num_requests
    steps = []
    for c in range(COPIES):
        reqs = copy_requests(w, COPIES, c)
        ids, q, kn, vn = s.decode_inputs(reqs)   # decode positions == request ids here
        out, lse = s.new_outputs(len(ids))
        lens = [w.req_ctx[r] for r in ids]
        steps.append((B.i32_array(ids), q, kn, vn, out, lse, B.i32_array(lens)))
    prefix_b, suffix_b, step_bytes = decode_bytes(w, copy_requests(w, COPIES, 0))
    stream = torch.cuda.current_stream(dev)

    def step(i):
        ids, q, kn, vn, out, lse, lens = steps[i % COPIES]
        s.ctx.decode(ids, q, kn, vn, out, lse, stream)
        s.ctx.request_truncate(ids, lens)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    for i in range(args.warmup):
        step(i)
    barrier()
    props = torch.cuda.get_device_properties(dev)
    clocks = Clocks(f"GPU-{props.uuid}" if getattr(props, "uuid", None) else str(local_rank))
    if rank == 0:
        clocks.start()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(args.steps):
        step(args.warmup + i)
    e1.record(stream)
    e1.synchronize()
    ms = e0.elapsed_time(e1)
    barrier()
    clk = clocks.stop() if rank == 0 else None
    ms, bytes_s = job_rate(ms, step_bytes * args.steps, world, dev)
    launches_per_step = s.ctx.query(B.Q_LAST_LAUNCHES)
    ms_step = ms / args.steps
    value = bytes_s / 1e9
    tokens_s = n * args.steps * world / (ms / 1e3)
    status = s.ctx.device_status()

    # per-kernel device time (CUDA events on each kernel's stream)
    s.ctx.set_option(B.OPT_KERNEL_TIMING, 1)
    s.ctx.kernel_times(reset=True)
    kt_steps = min(args.steps, 400)
    for i in range(kt_steps):
        step(i)
    torch.cuda.synchronize(dev)
    kt = s.ctx.kernel_times(reset=True)
    s.ctx.set_option(B.OPT_KERNEL_TIMING, 0)
    # the unified launch does all of the step's algorithmic HBM work (append,
    # both levels); the merge that follows only reads the L2-resident partials
    kbytes = {"dense_tcgen05": step_bytes}
    share = {k: v[0] for k, v in kt.items() if v[1]}
    dom = "dense_tcgen05"
    dom_ms = kt[dom][0] / max(1, kt[dom][1])
    achieved = kbytes[dom] / (dom_ms / 1e3) / 1e9
    kernels = {k: {"launches": v[1], "avg_us": round(1e3 * v[0] / v[1], 2) if v[1] else None,
                   "share": round(v[0] / sum(share.values()), 3) if v[1] else 0.0}
               for k, v in kt.items() if v[1]}

    # end to end through the public call with host buffers.  A step's inputs
    # (q, k_new, v_new) sit back to back in one pinned host buffer and its
    # outputs (out, lse) in another.  tpa_decode takes the pinned host arrays
    # themselves: its kernels read the inputs and write the outputs over the
    # CPU-GPU link (NVLink-C2C), so each step moves exactly those bytes across
    # the link inside the timed region, with no staging copy.  The same step
    # with copy-engine copies into device buffers and back is timed too.
    import torch as _t

    def packed(tensors, device):
        sizes = [x.numel() * x.element_size() for x in tensors]
        buf = _t.empty(sum(sizes), dtype=_t.uint8, device=device,
                       pin_memory=device == "cpu")
        views, off = [], 0
        for x, n in zip(tensors, sizes):
            views.append(buf[off:off + n].view(x.dtype).view(x.shape))
            off += n
        return buf, views

    host, dev_io = [], []
    for ids, q, kn, vn, out, lse, lens in steps:
        hin, hviews = packed((q, kn, vn), "cpu")
        for hv_, x in zip(hviews, (q, kn, vn)):
            hv_.copy_(x.cpu())
        hout, houts = packed((out, lse), "cpu")
        din, (dq, dkn, dvn) = packed((q, kn, vn), dev)
        dout, (dou, dls) = packed((out, lse), dev)
        host.append((hin, hout, hviews, houts))
        dev_io.append((din, dq, dkn, dvn, dout, dou, dls))
    h2d = host[0][0].numel()
    d2h = host[0][1].numel()
    e2e_steps = args.steps

    def e2e_step(i):
        ids, _, _, _, _, _, lens = steps[i % COPIES]
        _, _, (hq, hkn, hvn), (hou, hls) = host[i % COPIES]
        s.ctx.decode(ids, hq, hkn, hvn, hou, hls, stream)
        s.ctx.request_truncate(ids, lens)

    def staged_step(i):
        ids, _, _, _, _, _, lens = steps[i % COPIES]
        hin, hout, _, _ = host[i % COPIES]
        din, dq, dkn, dvn, dout, dou, dls = dev_io[i % COPIES]
        din.copy_(hin, non_blocking=True)
        s.ctx.decode(ids, dq, dkn, dvn, dou, dls, stream)
        hout.copy_(dout, non_blocking=True)
        s.ctx.request_truncate(ids, lens)

    def timed_loop(fn, n):
        for i in range(args.warmup):
            fn(i)
        barrier()
        e0.record(stream)
        for i in range(n):
            fn(i)
        e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1)

    ms_e2e, e2e_bytes_s = job_rate(timed_loop(e2e_step, e2e_steps), step_bytes * e2e_steps, world, dev)
    staged_n = min(e2e_steps, 500)
    ms_st, st_bytes_s = job_rate(timed_loop(staged_step, staged_n), step_bytes * staged_n, world, dev)
    e2e = {"value": round(e2e_bytes_s / 1e9, 1), "unit": "GB/s",
           "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
           "ms_per_step": round(ms_e2e / e2e_steps, 4),
           "io": "pinned host buffers passed to tpa_decode; its kernels read q/k_new/v_new and "
                 "write out/lse over NVLink-C2C (no staging copy)",
           "copy_engine": {"value": round(st_bytes_s / 1e9, 1), "unit": "GB/s",
                           "ms_per_step": round(ms_st / staged_n, 4),
                           "io": "cudaMemcpyAsync of the packed inputs to device buffers, "
                                 "tpa_decode on those, cudaMemcpyAsync of the outputs back"}}

    result = {
        "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) bf16 Q/K/V, random-init; no model weights)",
        "config": {"workload": "llama3_8b_decode: Hq=32 Hkv=8 d=128 bf16, 4 agents x 4096-token "
                               "prefixes, 64 decode requests (16/agent), cached suffixes U[256,1024], "
                               "page 16, contiguous pages",
                   "l2": f"inputs larger than L2: {COPIES} copies cycled, "
                         f"{COPIES * step_bytes / 1e9:.2f} GB between reuses",
                   "bytes_per_step": step_bytes, "prefix_bytes": prefix_b, "suffix_bytes": suffix_b,
                   "parallelism": f"replicas x{world}"},
        "hbm_frac_of_measured": round(value / world / hbm_peak, 4),
        "hbm_frac_of_8tbs": round(value / world / 8000.0, 4),
        "tokens_per_s": round(tokens_s, 1),
        "roofline": {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 1),
                     "peak": hbm_peak, "unit": "GB/s", "frac": round(achieved / hbm_peak, 4),
                     "peak_source": peak_src, "traffic": profiled_traffic(),
                     "bytes_per_launch": kbytes[dom], "avg_launch_us": round(dom_ms * 1e3, 2)},
        "kernels": kernels,
        "e2e": e2e,
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clk,
        "device_status": status,
    }
    s.ctx.close()
    del s, t
    torch.cuda.empty_cache()
    if rank == 0 and world == 1 and not args.no_extras:
        result["prefill"] = bench_prefill(args, dev, tf_peak, peak_src)
        result["decode_70b"] = bench_70b(args, dev, hbm_peak, peak_src)
        result["mixed"] = bench_mixed(args, dev)
        result["movement"] = bench_movement(args, dev)
        result["redo"] = bench_redo(args, dev)
        result["coresidency"] = bench_coresidency(args, dev)
        result["sched"] = bench_sched(args, dev)
    if rank == 0 and world == 1 and not args.no_cpu:
        result["cpu_baseline"] = cpu_baseline(budget_s=15.0)
    return result


def bench_prefill(args, dev, tf_peak, peak_src):
    """Chunked causal prefill workload: all 512-token chunk rounds of 256
    new requests over 8 agents' prefixes, timed as one pass (with
    --prefill-stride k, every k-th request only: a small case of the same
    shapes for profiler captures)."""
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import config, request_subset, tensors_torch

    stride = max(1, getattr(args, "prefill_stride", 1))
    w = config(2) if stride == 1 else request_subset(config(2), stride)
    stream = torch.cuda.current_stream(dev)

    def one_pass(kernel_timing=False):
        t = tensors_torch(w, dev)
        s = Session(w, t, device=dev, extra_tokens=0)
        s.ctx.set_option(B.OPT_KERNEL_TIMING, 1 if kernel_timing else 0)
        rounds = []
        for rnd in range(w.prefill_rounds()):
            chunks, ids, lens, q, k, v = s.prefill_inputs(rnd)
            out, lse = s.new_outputs(sum(lens))
            rounds.append((chunks, ids, lens, q, k, v, out, lse))
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for chunks, ids, lens, q, k, v, out, lse in rounds:
            s.prefill(ids, lens, q, k, v, out, lse, stream)
        e1.record(stream)
        e1.synchronize()
        kt = s.ctx.kernel_times(reset=True) if kernel_timing else None
        st = s.ctx.device_status()
        s.ctx.close()
        return e0.elapsed_time(e1), kt, st, rounds

    one_pass()                                  # warm-up (first-touch, clocks)
    ms, _, st, rounds = one_pass()
    _, kt, _, _ = one_pass(kernel_timing=True)
    flops = sum(prefill_flops(w, r[0]) for r in rounds)
    tokens = sum(sum(r[2]) for r in rounds)
    kname = "prefill_pair_tcgen05"  # the default 256-row items
    dense_ms = kt[kname][0]
    ach = flops / (dense_ms / 1e3) / 1e12
    nreq = w.num_requests
    return {"workload": f"chunked_prefill: 8 agents, prefixes U[2048,8192], {nreq} requests, suffixes "
                        "U[512,2048] in 512-token chunks (all rounds)" +
                        (f", every {stride}th request of the 256" if stride > 1 else ""),
            "tflops": round(flops / (ms / 1e3) / 1e12, 1), "ms": round(ms, 3),
            "tokens_per_s": round(tokens / (ms / 1e3), 1), "flops": flops,
            "roofline": {"bound": "tensor", "kernel": kname, "achieved": round(ach, 1),
                         "peak": tf_peak, "unit": "TFLOP/s", "frac": round(ach / tf_peak, 4),
                         "peak_source": peak_src, "traffic": None,
                         "avg_launch_us": round(1e3 * dense_ms / max(1, kt[kname][1]), 1)},
            "device_status": st}


def bench_sched(args, dev):
    """TOPAS decisions driving the library (the scheduler of Sec. IV as a host
    module): Chain-3 tasks on the Llama-3-8B attention layer under a KV budget
    that forces prefix moves and preemptions.  Service times are synthetic;
    the page table and the attention kernels are real.  Reports the native
    decision latency and, as its CPU baseline, the oracle's on the same
    recorded snapshots."""
    import time
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.workflow_sim import WorkflowSim, chain3

    wf = chain3()
    pages = 900     # the three prefixes need 576 pages: room for a few requests
    ctx = B.allocate(num_q_heads=32, num_kv_heads=8, head_dim=128, num_pages=pages, max_agents=8,
                     max_requests=64, max_tokens=1024, max_seq_len=8192, device=str(dev))
    ctx.set_option(B.OPT_KERNEL_TIMING, 1)
    rec = []
    sim = WorkflowSim(wf, ctx, n_tasks=40, rate=1.5, seed=7, dims=(32, 8, 128), budget_pages=pages,
                      max_tokens=1024, max_requests=64, device=str(dev), record=rec)
    res = sim.run()
    torch.cuda.synchronize(dev)
    kt = ctx.kernel_times(reset=True)
    st = ctx.device_status()
    ctx.close()
    native = [B.sched_decide(prm, snap, repeat=20)["native_us"] for prm, snap, _ in rec]
    out = res.summary()
    out.update({
        "workload": "chain3 workflow (3 agents, prefixes 2048/4096/3072 tokens), 40 tasks, "
                    "Poisson 1.5/s, KV budget 900 pages; Llama-3-8B layer (Hq 32, Hkv 8, d 128); "
                    "synthetic service times (20 us/prefill token, 20 ms/decode step)",
        "native_decide_us_mean": round(sum(native) / len(native), 1),
        "native_decide_us_max": round(max(native), 1),
        "gpu_ms": {k: round(v[0], 3) for k, v in kt.items() if v[1]},
        "device_status": st})
    if not args.no_cpu:
        import oracle.sched as OS   # CPU baseline: the oracle on the same snapshots
        t0 = time.perf_counter()
        n = 0
        for prm, snap, _ in rec:
            OS.decide(OS.Snapshot(**vars(snap)), OS.Params(**vars(prm)))
            n += 1
            if time.perf_counter() - t0 > 10.0:
                break
        out["cpu_baseline"] = {"value": round((time.perf_counter() - t0) / n * 1e6, 1), "unit": "us/decision",
                               "cores": 1, "kind": "oracle",
                               "sample": f"the first {n} of {len(rec)} recorded decisions"}
    return out


def bench_70b(args, dev, hbm_peak, peak_src):
    """Llama-3-70B layer decode: 6 agents x 16384-token prefixes, 512
    requests, suffixes U[512,4096]; 5.3 GB of KV per layer per step.

    The workload is sized to fill most of a 180 GB HBM: L layer pools (one
    context per layer, all with the same page and request tables, each with
    its own seeded KV and queries) take about 80 % of 180 GB, capped by the
    free memory.  A step runs the decode of every layer in turn, as a model's
    forward pass would, so consecutive decodes never share an L2-resident
    byte; the numbers are per layer (the step time divided by L)."""
    import dataclasses
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import config, tensors_torch

    w = config(4)
    stream = torch.cuda.current_stream(dev)
    prefix_b, suffix_b, step_bytes = decode_bytes(w, w.decode_requests())
    layers = []   # (session, ids array, lens array, q, k_new, v_new)
    t_setup = time.perf_counter()

    def add_layer(l):
        wl = w if l == 0 else dataclasses.replace(w, seed=w.seed + 1000 * l)
        t = tensors_torch(wl, dev)
        s = Session(wl, t, device=dev, extra_tokens=16, max_tokens=len(w.decode_requests()))
        ids, q, kn, vn = s.decode_inputs()
        s.t = None    # the drawn KV now lives in the pool only
        lens = [w.req_ctx[r] for r in ids]
        layers.append((s, B.i32_array(ids), B.i32_array(lens), q, kn, vn))

    add_layer(0)
    torch.cuda.synchronize(dev)
    s0 = layers[0][0]
    per_layer = (s0.ctx.k_pool.numel() * 2 * 2 + s0.ctx.workspace.numel()
                 + 3 * layers[0][3].numel() * 2)
    free, _ = torch.cuda.mem_get_info(dev)
    n_layers = max(1, min(args.layers_70b, 1 + int((free - 8e9) // per_layer)))
    for l in range(1, n_layers):
        add_layer(l)
    torch.cuda.synchronize(dev)
    t_setup = time.perf_counter() - t_setup
    n_dec = len(w.decode_requests())
    out, lse = s0.new_outputs(n_dec)

    def step():
        for s, ida, lna, q, kn, vn in layers:
            s.ctx.decode(ida, q, kn, vn, out, lse, stream)
            s.ctx.request_truncate(ida, lna)

    for _ in range(2):
        step()
    torch.cuda.synchronize(dev)
    k = 4
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(k):
        step()
    e1.record(stream)
    e1.synchronize()
    ms = e0.elapsed_time(e1) / (k * n_layers)
    for s, *_ in layers:
        s.ctx.set_option(B.OPT_KERNEL_TIMING, 1)
    step()
    kt = {}
    for s, *_ in layers:
        for kk, v in s.ctx.kernel_times(reset=True).items():
            a = kt.setdefault(kk, [0.0, 0])
            a[0] += v[0]
            a[1] += v[1]
    st = 0
    for s, *_ in layers:
        st |= s.ctx.device_status()
        s.ctx.close()
    resident = n_layers * per_layer
    del layers, s0, out, lse
    torch.cuda.empty_cache()
    gbs = step_bytes / (ms / 1e3) / 1e9
    return {"workload": "llama3_70b_decode: Hq=64 Hkv=8 d=128, 6 agents x 16384-token prefixes, "
                        "512 requests, suffixes U[512,4096]; %d layer pools (%.0f GB resident), "
                        "every step decodes all layers in turn" % (n_layers, resident / 1e9),
            "layers": n_layers, "resident_gb": round(resident / 1e9, 1),
            "value": round(gbs, 1), "unit": "GB/s", "ms_per_step": round(ms, 4),
            "ms_per_step_all_layers": round(ms * n_layers, 3),
            "hbm_frac_of_measured": round(gbs / hbm_peak, 4), "hbm_frac_of_8tbs": round(gbs / 8000, 4),
            "tokens_per_s": round(n_dec / (ms / 1e3), 1), "bytes_per_step": step_bytes,
            "kernels": {kk: {"avg_us": round(1e3 * v[0] / v[1], 1), "launches": v[1]}
                        for kk, v in kt.items() if v[1]},
            "setup_s": round(t_setup, 1), "device_status": st}


def bench_mixed(args, dev):
    """Mixed step: 2 prefixes reloaded from pinned host on a side stream,
    8 x 1024-token prefill chunks and 256 Zipf-assigned decode requests on
    a permuted (fragmented) pool."""
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import config, tensors_torch

    w = config(3)
    t = tensors_torch(w, dev)
    s = Session(w, t, device=dev, extra_tokens=16)
    s.offload_for_reload()
    stream = torch.cuda.current_stream(dev)
    side = torch.cuda.Stream(device=dev)
    chunks, pids, plens, pq, pk, pv = s.prefill_inputs(0)
    pout, plse = s.new_outputs(sum(plens))
    dids, dq, dkn, dvn = s.decode_inputs()
    dout, dlse = s.new_outputs(len(dids))
    ida = B.i32_array(dids)
    lna = B.i32_array([w.req_ctx[r] for r in dids])
    pida = B.i32_array(pids)
    zeros = B.i32_array([0] * len(pids))

    def step():
        s.reload(side_stream=side)
        s.prefill(pida, plens, pq, pk, pv, pout, plse, stream)
        s.ctx.decode(ida, dq, dkn, dvn, dout, dlse, stream)
        s.ctx.request_truncate(ida, lna)
        s.ctx.request_truncate(pida, zeros)
        for a in w.reload_agents:
            s.ctx.prefix_evict(a)

    step()
    torch.cuda.synchronize(dev)
    k = 10
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(k):
        step()
    e1.record(stream)
    side.synchronize()
    e1.synchronize()
    ms = e0.elapsed_time(e1) / k
    # per-kernel device time (events around each launch, which also counts a
    # launch's wait for free SMs, e.g. the reload scatter behind the prefill)
    s.ctx.set_option(B.OPT_KERNEL_TIMING, 1)
    s.ctx.kernel_times(reset=True)
    for _ in range(5):
        step()
    side.synchronize()
    torch.cuda.synchronize(dev)
    kt = s.ctx.kernel_times(reset=True)
    st = s.ctx.device_status()
    reload_bytes = sum(w.prefix_len[a] for a in w.reload_agents) * w.kv_bytes_per_token()
    pf = prefill_flops(w, chunks)
    _, _, dec_bytes = decode_bytes(w, dids)
    s.ctx.close()
    per_step = {kk: {"us": round(1e3 * v[0] / 5, 1), "launches": v[1] // 5}
                for kk, v in kt.items() if v[1]}
    if "prefill_pair_tcgen05" in per_step:
        per_step["prefill_pair_tcgen05"]["tflops"] = round(
            pf / (per_step["prefill_pair_tcgen05"]["us"] * 1e-6) / 1e12, 1)
    if "dense_tcgen05" in per_step:
        per_step["dense_tcgen05"]["gbs"] = round(
            dec_bytes / (per_step["dense_tcgen05"]["us"] * 1e-6) / 1e9, 1)
    return {"workload": "mixed: 16 agents prefixes U[1024,8192], 256 Zipf(1.1) decode requests "
                        "(suffixes U[256,1024]), 8 x 1024-token prefill chunks, permuted pool, "
                        "2 prefixes reloaded from pinned host on a side stream",
            "ms_per_step": round(ms, 4), "decode_tokens_per_s": round(len(dids) / (ms / 1e3), 1),
            "prefill_flops": pf, "decode_bytes": dec_bytes, "reload_bytes": reload_bytes,
            "kernels_per_step": per_step, "device_status": st}


def bench_movement(args, dev):
    """Prefix movement between GPU and pinned host memory (Sec. IV, Eq. 7:
    T_move = mu / B_swap x the moved prefix lengths; the same mu l_a / B_swap
    prices reuse in Eq. 10).  For prefixes of the Llama-3-8B layer (mu = 4096
    B per token) of several lengths: reload = host -> free, permuted pages on
    a side stream; offload = pages -> host.  Each is fitted as t = t0 + bytes
    / B and compared with a plain pinned copy of the same bytes."""
    import torch
    from paper_2608_25523_gb300 import binding as B

    hkv, d, hq = 8, 128, 32
    mu = 2 * hkv * d * 2
    sizes = [1024, 4096, 16384, 65536]
    lmax = max(sizes)
    ctx = B.allocate(num_q_heads=hq, num_kv_heads=hkv, head_dim=d, num_pages=lmax // 16 + 64,
                     max_agents=len(sizes), max_requests=1, max_tokens=1024,
                     max_seq_len=lmax + 64, page_order_seed=3, device=dev)
    side = torch.cuda.Stream(device=dev)
    g = torch.Generator().manual_seed(11)
    hk = torch.randn(lmax, hkv, d, generator=g).to(torch.bfloat16).pin_memory()
    hv = torch.randn(lmax, hkv, d, generator=g).to(torch.bfloat16).pin_memory()
    ok = torch.empty_like(hk).pin_memory()
    ov = torch.empty_like(hv).pin_memory()
    dk = torch.empty(lmax, hkv, d, dtype=torch.bfloat16, device=dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed(fn, before=None, reps=5):
        ts = []
        for _ in range(reps + 1):
            if before:
                before()
            e0.record(side)
            fn()
            e1.record(side)
            e1.synchronize()
            ts.append(e0.elapsed_time(e1) * 1e3)
        return sorted(ts[1:])[len(ts[1:]) // 2]   # median, first run dropped

    rows = []
    for a, ell in enumerate(sizes):
        ctx.prefix_register(a, ell)
        ctx.prefix_write(a, hk[:ell], hv[:ell], side)
        side.synchronize()

        resident = [True]

        def evict():       # untimed: free the pages (table only)
            if resident[0]:
                ctx.prefix_evict(a)
                resident[0] = False

        def reload():      # pinned host -> free (permuted) pages
            ctx.prefix_reload(a, hk[:ell], hv[:ell], side)
            resident[0] = True

        def offload():     # pages -> pinned host, then evicted
            ctx.prefix_offload(a, ok[:ell], ov[:ell], side)
            resident[0] = False

        def make_resident():
            if not resident[0]:
                reload()

        def h2d():
            dk[:ell].copy_(hk[:ell], non_blocking=True)
            dk[:ell].copy_(hv[:ell], non_blocking=True)

        def d2h():
            ok[:ell].copy_(dk[:ell], non_blocking=True)
            ov[:ell].copy_(dk[:ell], non_blocking=True)

        with torch.cuda.stream(side):
            # the page kernel on the mapped host arrays (TPA_OPT_MOVEMENT_STAGED 0) ...
            ctx.set_option(B.OPT_MOVEMENT_STAGED, 0)
            t_re_d = timed(reload, before=evict)
            t_off_d = timed(offload, before=make_resident)
            # ... and the default: copy engine through the staging area
            ctx.set_option(B.OPT_MOVEMENT_STAGED, 1)
            t_re = timed(reload, before=evict)
            t_off = timed(offload, before=make_resident)
            side.synchronize()
            exact = bool(torch.equal(ok[:ell].view(torch.int16), hk[:ell].view(torch.int16)) and
                         torch.equal(ov[:ell].view(torch.int16), hv[:ell].view(torch.int16)))
            t_h2d, t_d2h = timed(h2d), timed(d2h)
        side.synchronize()
        rows.append({"tokens": ell, "bytes": ell * mu, "reload_us": round(t_re, 1),
                     "offload_us": round(t_off, 1), "reload_direct_us": round(t_re_d, 1),
                     "offload_direct_us": round(t_off_d, 1), "h2d_copy_us": round(t_h2d, 1),
                     "d2h_copy_us": round(t_d2h, 1), "round_trip_bit_exact": exact})
        evict()

    def fit(key):
        xs = [r["bytes"] for r in rows]
        ys = [r[key] for r in rows]
        n = len(xs)
        mx, my = sum(xs) / n, sum(ys) / n
        slope = sum((x - mx) * (y - my) for x, y in zip(xs, ys)) / sum((x - mx) ** 2 for x in xs)
        return {"B_gbs": round(1e-3 / slope, 1), "t0_us": round(my - slope * mx, 1)}

    ctx.close()
    res = {"workload": "prefix movement, llama3_8b layer (mu = 4096 B/token), prefixes of "
                       + ", ".join(str(x) for x in sizes) + " tokens, permuted pool",
           "rows": rows, "reload": fit("reload_us"), "offload": fit("offload_us"),
           "reload_direct": fit("reload_direct_us"), "offload_direct": fit("offload_direct_us"),
           "h2d_copy": fit("h2d_copy_us"), "d2h_copy": fit("d2h_copy_us")}
    res["mu_over_B_swap_ns_per_token"] = {
        "reload": round(mu / (res["reload"]["B_gbs"] * 1e9) * 1e9, 3),
        "offload": round(mu / (res["offload"]["B_gbs"] * 1e9) * 1e9, 3)}
    return res


def bench_redo(args, dev):
    """Rebuilding a preempted request's suffix KV (Sec. IV, Eq. 8 charges
    T_decode y_r for redoing y_r tokens one decode step at a time) against
    rebuilding it with chunked causal prefill (512-token chunks), both
    through this library on one Llama-3-8B layer: one agent with a
    4096-token prefix, one request whose suffix is rebuilt from empty."""
    import torch
    from paper_2608_25523_gb300 import binding as B

    hq, hkv, d, lp = 32, 8, 128, 4096
    ys = [256, 1024, 4096]
    ymax = max(ys)
    ctx = B.allocate(num_q_heads=hq, num_kv_heads=hkv, head_dim=d,
                     num_pages=(lp + ymax) // 16 + 64, max_agents=1, max_requests=1,
                     max_tokens=512, max_seq_len=lp + ymax + 64, device=dev)
    g = torch.Generator(device=dev).manual_seed(5)

    def rnd(*shape):
        return torch.randn(*shape, generator=g, device=dev).to(torch.bfloat16)
    pk, pv = rnd(lp, hkv, d), rnd(lp, hkv, d)
    q, k, v = rnd(ymax, hq, d), rnd(ymax, hkv, d), rnd(ymax, hkv, d)
    out, lse = torch.empty(512, hq, d, dtype=torch.bfloat16, device=dev), \
        torch.empty(512, hq, dtype=torch.float32, device=dev)
    ctx.prefix_register(0, lp)
    ctx.prefix_write(0, pk, pv)
    ctx.request_open(0, 0)
    one, zero = B.i32_array([0]), B.i32_array([0])
    stream = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def run(fn):
        ctx.request_truncate(one, zero)
        fn()                                  # warm-up pass
        torch.cuda.synchronize(dev)
        ctx.request_truncate(one, zero)
        ctx.set_option(B.OPT_KERNEL_TIMING, 1)
        ctx.kernel_times(reset=True)
        e0.record(stream)
        fn()
        e1.record(stream)
        e1.synchronize()
        kt = ctx.kernel_times(reset=True)
        ctx.set_option(B.OPT_KERNEL_TIMING, 0)
        return e0.elapsed_time(e1), sum(t for t, n in kt.values())

    rows = []
    for y in ys:
        def by_decode():
            for i in range(y):
                ctx.decode(one, q[i:i + 1], k[i:i + 1], v[i:i + 1], out[:1], lse[:1], stream)

        def by_prefill():
            for o in range(0, y, 512):
                c = min(512, y - o)
                ctx.prefill_chunk(one, [c], q[o:o + c], k[o:o + c], v[o:o + c], out[:c], lse[:c],
                                  stream)

        wd, kd = run(by_decode)
        wp, kp = run(by_prefill)
        rows.append({"tokens": y, "decode_redo_ms": round(wd, 3), "decode_redo_kernel_ms": round(kd, 3),
                     "prefill_rebuild_ms": round(wp, 3), "prefill_rebuild_kernel_ms": round(kp, 3),
                     "T_decode_us_per_token": round(1e3 * kd / y, 2),
                     "kernel_speedup": round(kd / kp, 1)})
    st = ctx.device_status()
    ctx.close()
    return {"workload": "redo of a preempted request's suffix: llama3_8b layer, prefix 4096, "
                        "suffix rebuilt from empty, decode (y steps) vs chunked prefill (512)",
            "rows": rows, "device_status": st}


def bench_coresidency(args, dev):
    """Kernel-level analogue of the paper's Diagnostic 1 (Sec. II, Table 1):
    under one KV budget, keeping one agent's long prefix resident (Grouped)
    admits twice the decode batch of keeping two (Alternating).  Budget
    49152 tokens of one Llama-3-8B layer; prefixes of 16384 tokens; each
    request holds a 2048-token suffix.  Grouped: agent A resident, 16
    requests; Alternating: A and B resident, 4 + 4 requests.  Each decode
    step reads the whole budget either way; throughput follows the batch."""
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import small_case, tensors_torch

    lp, ls, budget = 16384, 2048, 49152
    cases = {"grouped": ([lp], [0] * 16), "alternating": ([lp, lp], [0, 1] * 4)}
    res = {"workload": f"KV budget {budget} tokens (llama3_8b layer), prefixes {lp}, "
                       f"suffixes {ls}; decode steps of the admitted batch"}
    stream = torch.cuda.current_stream(dev)
    for name, (plens, agents) in cases.items():
        n = len(agents)
        assert sum(plens) + n * ls <= budget
        w = small_case(7, hq=32, hkv=8, d=128, prefix_len=plens, req_agent=agents,
                       req_ctx=[ls - 1] * n, req_prefill=[0] * n, req_decode=[1] * n)
        t = tensors_torch(w, dev)
        s = Session(w, t, device=dev, extra_tokens=16)
        ids, q, kn, vn = s.decode_inputs()
        out, lse = s.new_outputs(n)
        ida, lna = B.i32_array(ids), B.i32_array([w.req_ctx[r] for r in ids])

        def step():
            s.ctx.decode(ida, q, kn, vn, out, lse, stream)
            s.ctx.request_truncate(ida, lna)
        for _ in range(10):
            step()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        k = 200
        e0.record(stream)
        for _ in range(k):
            step()
        e1.record(stream)
        e1.synchronize()
        us = e0.elapsed_time(e1) / k * 1e3
        step_bytes = decode_bytes(w, ids)[2]
        res[name] = {"resident_prefixes": len(plens), "batch": n, "step_us": round(us, 2),
                     "tokens_per_s": round(n / (us / 1e6), 1),
                     "gbs": round(step_bytes / (us / 1e6) / 1e9, 1),
                     "device_status": s.ctx.device_status()}
        s.ctx.close()
        del s, t
    res["grouped_over_alternating_tokens_per_s"] = round(
        res["grouped"]["tokens_per_s"] / res["alternating"]["tokens_per_s"], 2)
    return res


# ------------------------------------------------------ oracle baseline --

def _blas_threads():
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 0) for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return max(n)
    except Exception:
        pass
    return os.cpu_count()


def cpu_baseline(budget_s=20.0, per_step_s=None, steps=1, warmup=0):
    """Time the fp64 oracle on this host's cores over a bounded sample of
    the decode workload.  The sample unit is one (request, kv head): the
    oracle's decode step for the G query heads of that kv head.  The value
    scales the step's algorithmic bytes by the fraction of units done."""
    import oracle
    from paper_2608_25523_gb300.workloads import config, tensors_numpy

    w = config(1)
    t = tensors_numpy(w)
    dec = w.decode_requests()
    G, hkv = w.group, w.num_kv_heads
    units = [(i, g) for i in range(len(dec)) for g in range(hkv)]
    step_bytes = decode_bytes(w, dec)[2]

    def run(us):
        for i, g in us:
            r = dec[i]
            pk, pv = t.prefix(w.req_agent[r], w)
            n_cached = w.req_ctx[r] + w.req_prefill[r]
            sk, sv = t.suffix(r, w, 0, n_cached)
            nk, nv = t.suffix(r, w, n_cached, n_cached + 1)
            oracle.decode_step(t.q_decode[i, g * G:(g + 1) * G], pk[:, g:g + 1], pv[:, g:g + 1],
                               sk[:, g:g + 1], sv[:, g:g + 1], nk[0, g:g + 1], nv[0, g:g + 1])

    t0 = time.perf_counter()
    run(units[:1])
    one = time.perf_counter() - t0
    total_s, done, pos = 0.0, 0, 0
    if per_step_s is None:
        # one timed region of about budget_s seconds: units cycled over the step
        t_end = time.perf_counter() + budget_s
        t0 = time.perf_counter()
        while done == 0 or time.perf_counter() < t_end:
            k = max(1, min(len(units), int(0.5 / max(one, 1e-6))))
            run([units[(pos + j) % len(units)] for j in range(k)])
            pos += k
            done += k
        total_s = time.perf_counter() - t0
        per = done
    else:
        per = max(1, min(len(units), int(per_step_s / max(one, 1e-6))))
        for i in range(warmup + steps):
            sample = [units[(pos + j) % len(units)] for j in range(per)]
            pos += per
            t0 = time.perf_counter()
            run(sample)
            dt = time.perf_counter() - t0
            if i >= warmup:
                total_s += dt
                done += per
    value = step_bytes * (done / len(units)) / total_s / 1e9
    return {"value": round(value, 4), "unit": "GB/s", "cores": _blas_threads(), "kind": "oracle",
            "sample": (f"{done} (request, kv head) units of the llama3_8b_decode step "
                       f"({len(units)} units per step; {done / len(units):.2f} steps' worth)"
                       if per_step_s is None else
                       f"{per} of {len(units)} (request, kv head) units of one llama3_8b_decode "
                       f"step per timed step, {steps} step(s)")
                      + "; float64 numpy over per-request materialised KV; value = step bytes x "
                        "steps' worth done / time",
            "seconds": round(total_s, 2)}


def run_reference(args, rank, world):
    if rank != 0:
        return None
    budget_total = 150.0
    per_step = budget_total / max(1, args.steps + args.warmup)
    cb = cpu_baseline(per_step_s=per_step, steps=args.steps, warmup=args.warmup)
    return {"impl": "reference", "metric": METRIC, "value": cb["value"], "unit": "GB/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": round(1e3 * cb["seconds"] / args.steps, 3),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": "llama3_8b_decode (bounded sample per step, see cpu_baseline)"},
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-extras", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--only", choices=["prefill", "decode_70b", "mixed", "movement", "redo",
                                       "coresidency", "sched"],
                    help="run just one of the extra workloads (1 GPU) and print its result")
    ap.add_argument("--layers-70b", type=int, default=26,
                    help="layer pools of the 70B decode workload (5.4 GB of KV each; "
                         "26 fill 80 %% of 180 GB), capped by the free memory")
    ap.add_argument("--prefill-stride", type=int, default=1,
                    help="prefill workload: every k-th request only (a small case for profiling)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3)
    rank = int(os.environ.get("RANK", 0))
    world = int(os.environ.get("WORLD_SIZE", 1))
    local_rank = int(os.environ.get("LOCAL_RANK", 0))
    if args.impl == "reference":
        res = run_reference(args, rank, world)
        if res is not None:
            print(json.dumps(res))
        return
    if args.only:
        import torch
        from paper_2608_25523_gb300.build import build
        build()
        dev = torch.device("cuda", 0)
        torch.cuda.set_device(dev)
        hbm_peak, tf_peak, _, peak_src = peaks()
        fn = {"prefill": lambda: bench_prefill(args, dev, tf_peak, peak_src),
              "decode_70b": lambda: bench_70b(args, dev, hbm_peak, peak_src),
              "mixed": lambda: bench_mixed(args, dev),
              "movement": lambda: bench_movement(args, dev),
              "redo": lambda: bench_redo(args, dev),
              "coresidency": lambda: bench_coresidency(args, dev),
              "sched": lambda: bench_sched(args, dev)}[args.only]
        print(json.dumps({"only": args.only, "result": fn()}))
        return
    if world > 1:
        import torch
        import torch.distributed as dist
        torch.cuda.set_device(local_rank)
        dist.init_process_group("nccl")
    res = run_ours(args, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(res))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
