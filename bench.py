"""Benchmark of shared-prefix paged attention on one GB300 (or N replicas).

Headline workload: the Llama-3-70B attention layer decode step (64 q heads,
8 kv heads, head_dim 128, bf16): 6 agents with 16384-token prefixes, 512
decode requests (86,86,85,85,85,85) with cached suffixes uniform in
512..4096, page size 16, contiguous pages; 5.35 GB of KV per layer.  The
workload is sized to fill most of a 180 GB HBM: L layer pools (26 by
default, one context each, the same page and request tables, each with its
own seeded KV and queries), 157 GB resident.  One step = one tpa_decode
call per layer, layer after layer, as a model's forward pass makes them
(host plan, one upload, one persistent tcgen05 launch that appends the new
tokens and runs the stacked shared-prefix tiles and the per-request
suffixes, and the log-sum-exp merge launched as its programmatic
dependent), each followed by a table-only truncate that drops the appended
token again so every step sees the same workload.  Consecutive decodes
never share an L2-resident byte (each layer's KV is 41x the L2).

value  = algorithmic bytes per step (per layer: each prefix once, each
         suffix once, Q, the new tokens' K/V in and into the pool, O and
         LSE; times L) / device time, GB/s.
e2e    = the same metric through the public call with host buffers: each
         layer's q / k_new / v_new sit in pinned host memory and its O / LSE
         go back to it, inside the timed region.  tpa_decode takes the host
         arrays themselves and its kernels move those bytes over the
         CPU-GPU link; the variant with copy-engine copies to and from
         device buffers is reported beside it (e2e.copy_engine).

Also reported (rank 0, N=1), each reduced to its headline fields in the
printed line (--detail PATH writes everything):
  decode_8b    the Llama-3-8B layer decode step (4 agents x 4096-token
               prefixes, 64 requests), 4 copies cycled, its own step count;
  prefill      the chunked-prefill workload (TFLOP/s, tensor roofline);
  mixed        reload + prefill + Zipf decode on a fragmented pool (ms/step);
  movement     prefix reload / offload bandwidth, the paper's mu / B_swap;
  redo         the redo trade of a preempted suffix (decode steps against
               chunked prefill);
  coresidency  a kernel-level analogue of the paper's co-residency
               diagnostic: admissible batch and tokens/s as the number of
               co-resident prefixes grows under one KV budget;
  sched        the TOPAS scheduler driving the library on Chain-3 tasks
               (decision latency, native and oracle).

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
COPIES = 4          # copies of the 8B decode workload cycled to defeat L2
LAYERS_70B = 26     # layer pools of the 70B workload (5.4 GB of KV each)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained", d["bf16_tflops"]), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


# ------------------------------------------------------------ accounting --

# Sources of the unified decode kernel; the DRAM traffic recorded in an ncu
# summary counts only while they are unchanged.
KERNEL_SOURCES = ["k_dense.cu", "dense_common.cuh", "split_kv.cuh", "ptx.cuh", "plan.h", "kernels.h"]
PROFILE_8B = os.path.join(ROOT, "profiles", "dense_tcgen05_c2_decode.md")
PROFILE_70B = os.path.join(ROOT, "profiles", "dense_tcgen05_70b_decode.md")


def kernel_source_hash():
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, "paper_2608_25523_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def profiled_traffic(path):
    """DRAM bytes (read + write) per launch of the unified decode kernel from
    a committed ncu summary, or None if it was taken on other sources."""
    try:
        vals = {}
        with open(path) as fh:
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


def headline_config(n_layers, world):
    """`config` of the headline line, shared by both arms."""
    from paper_2608_25523_gb300.workloads import config
    w = config(4)
    layer_bytes = decode_bytes(w, w.decode_requests())[2]
    return {"workload": f"llama3_70b_decode: Hq64 Hkv8 d128 bf16, 6 x 16384-token prefixes, "
                        f"512 requests, suffixes U[512,4096], {n_layers} layers",
            "layers": n_layers,
            "step": "one decode step of the 512 requests in every layer pool, layer after layer",
            "l2": "inputs larger than L2: each layer's KV (5.35 GB) is read once per step",
            "bytes_per_layer": layer_bytes, "bytes_per_step": layer_bytes * n_layers,
            "parallelism": f"replicas x{world}"}


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

def _packed(tensors, device):
    """One buffer (pinned when on the host) holding `tensors` back to back,
    and views of it shaped like them."""
    import torch
    sizes = [x.numel() * x.element_size() for x in tensors]
    buf = torch.empty(sum(sizes), dtype=torch.uint8, device=device, pin_memory=device == "cpu")
    views, off = [], 0
    for x, n in zip(tensors, sizes):
        views.append(buf[off:off + n].view(x.dtype).view(x.shape))
        off += n
    return buf, views


def build_70b_layers(dev, max_layers):
    """The 70B decode workload's layer pools: one Session per layer with the
    same page and request tables and its own seeded KV and queries, as many
    as fit (at most `max_layers`).  Returns (workload, layers, bytes held
    per layer, setup seconds); a layer is (session, ids, lens, q, k_new, v_new)."""
    import dataclasses
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import config, tensors_torch

    w = config(4)
    layers = []
    t0 = time.perf_counter()

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
    n_layers = max(1, min(max_layers, 1 + int((free - 8e9) // per_layer)))
    for l in range(1, n_layers):
        add_layer(l)
    torch.cuda.synchronize(dev)
    return w, layers, per_layer, time.perf_counter() - t0


def measure_70b(args, rank, world, dev, hbm_peak, peak_src, steps, warmup, with_e2e=True):
    """The headline: decode steps of the 70B workload over every layer pool.

    Timed region: `steps` steps after `warmup` untimed ones, a barrier and a
    device synchronize on both sides, CUDA events on the launching stream,
    nvidia-smi clocks sampled during it (rank 0).  The unified kernel's
    launches run back to back (the merge of each layer is its programmatic
    dependent, and the next layer's unified kernel the merge's), so its
    average launch duration is the timed region over its launches; a short
    second region with every launch bracketed by events (which breaks that
    overlap) gives each kernel's share."""
    import torch
    import torch.distributed as dist
    from paper_2608_25523_gb300 import binding as B

    w, layers, per_layer, setup_s = build_70b_layers(dev, args.layers_70b)
    n_layers = len(layers)
    n_dec = len(w.decode_requests())
    out, lse = layers[0][0].new_outputs(n_dec)
    stream = torch.cuda.current_stream(dev)
    prefix_b, suffix_b, layer_bytes = decode_bytes(w, w.decode_requests())
    step_bytes = layer_bytes * n_layers

    def step(_i):
        for s, ida, lna, q, kn, vn in layers:
            s.ctx.decode(ida, q, kn, vn, out, lse, stream)
            s.ctx.request_truncate(ida, lna)

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def timed_loop(fn, n, clocks=None):
        for i in range(warmup):
            fn(i)
        barrier()
        if clocks is not None:
            clocks.start()
        e0.record(stream)
        for i in range(n):
            fn(warmup + i)
        e1.record(stream)
        e1.synchronize()
        ms = e0.elapsed_time(e1)
        barrier()
        clk = clocks.stop() if clocks is not None else None
        return ms, clk

    props = torch.cuda.get_device_properties(dev)
    clocks = Clocks(f"GPU-{props.uuid}" if getattr(props, "uuid", None) else str(dev.index or 0)) \
        if rank == 0 else None
    ms, clk = timed_loop(step, steps, clocks)
    ms, bytes_s = job_rate(ms, step_bytes * steps, world, dev)
    launches = sum(s.ctx.query(B.Q_LAST_LAUNCHES) for s, *_ in layers)
    status = 0
    for s, *_ in layers:
        status |= s.ctx.device_status()
    value = bytes_s / 1e9
    period_us = 1e3 * ms / (steps * n_layers)

    # per-kernel shares: every launch bracketed by events (two steps, after
    # one that creates the events)
    for s, *_ in layers:
        s.ctx.set_option(B.OPT_KERNEL_TIMING, 1)
    step(0)
    torch.cuda.synchronize(dev)
    for s, *_ in layers:
        s.ctx.kernel_times(reset=True)
    for i in range(2):
        step(i)
    torch.cuda.synchronize(dev)
    kt = {}
    for s, *_ in layers:
        for k, v in s.ctx.kernel_times(reset=True).items():
            a = kt.setdefault(k, [0.0, 0])
            a[0] += v[0]
            a[1] += v[1]
        s.ctx.set_option(B.OPT_KERNEL_TIMING, 0)
    tot = sum(v[0] for v in kt.values() if v[1]) or 1.0
    kernels = {k: {"launches": v[1], "bracketed_avg_us": round(1e3 * v[0] / v[1], 1),
                   "share": round(v[0] / tot, 3)} for k, v in kt.items() if v[1]}
    dom = "dense_tcgen05"
    achieved = layer_bytes / (period_us * 1e-6) / 1e9
    res = {
        "metric": METRIC, "value": round(value, 1), "unit": "GB/s", "n_gpus": world,
        "steps": steps, "warmup": warmup, "ms_per_step": round(ms / steps, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded N(0,1) bf16 Q/K/V, random-init; no model weights)",
        "config": headline_config(n_layers, world),
        "ms_per_layer": round(ms / (steps * n_layers), 4),
        "hbm_frac_of_measured": round(value / world / hbm_peak, 4),
        "hbm_frac_of_8tbs": round(value / world / 8000.0, 4),
        "tokens_per_s": round(n_dec * steps * world / (ms / 1e3), 1),
        "tokens_per_s_note": "decode tokens per second through all layers (one token per request per step)",
        "roofline": {"bound": "hbm", "kernel": dom, "achieved": round(achieved, 1),
                     "peak": hbm_peak, "unit": "GB/s", "frac": round(achieved / hbm_peak, 4),
                     "peak_source": peak_src, "traffic": profiled_traffic(PROFILE_70B),
                     "bytes_per_launch": layer_bytes, "avg_launch_us": round(period_us, 1),
                     "avg_launch_from": "timed region / unified-kernel launches (back to back)",
                     "bracketed_avg_us": kernels.get(dom, {}).get("bracketed_avg_us")},
        "kernels": kernels,
        "gpu_launches": launches * steps,
        "clocks": clk,
        "resident_gb": round(n_layers * per_layer / 1e9, 1),
        "setup_s": round(setup_s, 1),
        "prefix_bytes_per_layer": prefix_b, "suffix_bytes_per_layer": suffix_b,
    }

    if with_e2e:
        # end to end through the public call with host buffers: each layer's
        # q, k_new, v_new sit back to back in one pinned host buffer and its
        # out, lse in another.  tpa_decode takes the pinned host arrays
        # themselves (its kernels read the inputs and write the outputs over
        # NVLink-C2C); the same step with copy-engine copies into device
        # buffers and back is timed too.
        host, dev_io = [], []
        for s, ida, lna, q, kn, vn in layers:
            hin, hviews = _packed((q, kn, vn), "cpu")
            for hv_, x in zip(hviews, (q, kn, vn)):
                hv_.copy_(x.cpu())
            hout, houts = _packed((out, lse), "cpu")
            din, dviews = _packed((q, kn, vn), dev)
            dout, douts = _packed((out, lse), dev)
            host.append((hin, hout, hviews, houts))
            dev_io.append((din, dout, dviews, douts))
        h2d = sum(h[0].numel() for h in host)
        d2h = sum(h[1].numel() for h in host)

        def e2e_step(_i):
            for (s, ida, lna, *_), (_, _, (hq, hkn, hvn), (hou, hls)) in zip(layers, host):
                s.ctx.decode(ida, hq, hkn, hvn, hou, hls, stream)
                s.ctx.request_truncate(ida, lna)

        def staged_step(_i):
            for (s, ida, lna, *_), (hin, hout, _, _), (din, dout, (dq, dkn, dvn), (dou, dls)) \
                    in zip(layers, host, dev_io):
                din.copy_(hin, non_blocking=True)
                s.ctx.decode(ida, dq, dkn, dvn, dou, dls, stream)
                hout.copy_(dout, non_blocking=True)
                s.ctx.request_truncate(ida, lna)

        ms_e, e_bytes_s = job_rate(timed_loop(e2e_step, steps)[0], step_bytes * steps, world, dev)
        ms_c, c_bytes_s = job_rate(timed_loop(staged_step, steps)[0], step_bytes * steps, world, dev)
        res["e2e"] = {"value": round(e_bytes_s / 1e9, 1), "unit": "GB/s",
                      "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                      "ms_per_step": round(ms_e / steps, 4),
                      "io": "pinned host q/k_new/v_new/out/lse passed to tpa_decode (zero copy)",
                      "copy_engine": {"value": round(c_bytes_s / 1e9, 1), "unit": "GB/s",
                                      "ms_per_step": round(ms_c / steps, 4),
                                      "io": "cudaMemcpyAsync in, tpa_decode, cudaMemcpyAsync out"}}
        for s, *_ in layers:
            status |= s.ctx.device_status()
        del host, dev_io
    res["device_status"] = status
    for s, *_ in layers:
        s.ctx.close()
    del layers, out, lse
    torch.cuda.empty_cache()
    return res


def run_ours(args, rank, world, local_rank):
    import torch

    from paper_2608_25523_gb300.build import build

    build()
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    hbm_peak, tf_peak, tf_sust, peak_src = peaks()
    result = measure_70b(args, rank, world, dev, hbm_peak, peak_src, args.steps, args.warmup)
    if rank == 0 and world == 1 and not args.no_extras:
        result["decode_8b"] = bench_decode_8b(args, dev, hbm_peak, peak_src)
        result["prefill"] = bench_prefill(args, dev, tf_peak, peak_src)
        result["mixed"] = bench_mixed(args, dev)
        result["movement"] = bench_movement(args, dev)
        result["redo"] = bench_redo(args, dev)
        result["coresidency"] = bench_coresidency(args, dev)
        result["sched"] = bench_sched(args, dev)
    if rank == 0 and world == 1 and not args.no_cpu:
        result["cpu_baseline"] = cpu_baseline(budget_s=15.0)
    return result


def bench_decode_8b(args, dev, hbm_peak, peak_src, steps=2000, warmup=20):
    """The Llama-3-8B layer decode step: 4 agents x 4096-token prefixes, 64
    decode requests (16/agent), cached suffixes U[256,1024].  Four copies of
    the workload are cycled so ~0.93 GB of KV lies between two visits of
    the same bytes.  Timed over its own `steps` (a 45 us step needs a long
    region to average out the first step's host latency), with the same e2e
    variants as the headline."""
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import config, copy_requests, replicate, tensors_torch

    base = config(1)
    w = replicate(base, COPIES)
    t = tensors_torch(w, dev)
    s = Session(w, t, device=dev, extra_tokens=16)
    n = base.num_requests
    steps_io = []
    for c in range(COPIES):
        reqs = copy_requests(w, COPIES, c)
        ids, q, kn, vn = s.decode_inputs(reqs)   # decode positions == request ids here
        out, lse = s.new_outputs(len(ids))
        lens = [w.req_ctx[r] for r in ids]
        steps_io.append((B.i32_array(ids), q, kn, vn, out, lse, B.i32_array(lens)))
    prefix_b, suffix_b, step_bytes = decode_bytes(w, copy_requests(w, COPIES, 0))
    stream = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)

    def step(i):
        ids, q, kn, vn, out, lse, lens = steps_io[i % COPIES]
        s.ctx.decode(ids, q, kn, vn, out, lse, stream)
        s.ctx.request_truncate(ids, lens)

    def timed_loop(fn, k):
        for i in range(warmup):
            fn(i)
        torch.cuda.synchronize(dev)
        e0.record(stream)
        for i in range(k):
            fn(warmup + i)
        e1.record(stream)
        e1.synchronize()
        return e0.elapsed_time(e1)

    ms = timed_loop(step, steps)
    period_us = 1e3 * ms / steps
    value = step_bytes / (period_us * 1e-6) / 1e9
    # a short region at the driver's default size, for comparison
    ms20 = timed_loop(step, 20)

    s.ctx.set_option(B.OPT_KERNEL_TIMING, 1)
    s.ctx.kernel_times(reset=True)
    for i in range(400):
        step(i)
    torch.cuda.synchronize(dev)
    kt = s.ctx.kernel_times(reset=True)
    s.ctx.set_option(B.OPT_KERNEL_TIMING, 0)
    tot = sum(v[0] for v in kt.values() if v[1]) or 1.0
    kernels = {k: {"launches": v[1], "bracketed_avg_us": round(1e3 * v[0] / v[1], 2),
                   "share": round(v[0] / tot, 3)} for k, v in kt.items() if v[1]}

    host, dev_io = [], []
    for ids, q, kn, vn, out, lse, lens in steps_io:
        hin, hviews = _packed((q, kn, vn), "cpu")
        for hv_, x in zip(hviews, (q, kn, vn)):
            hv_.copy_(x.cpu())
        hout, houts = _packed((out, lse), "cpu")
        din, dviews = _packed((q, kn, vn), dev)
        dout, douts = _packed((out, lse), dev)
        host.append((hin, hout, hviews, houts))
        dev_io.append((din, dout, dviews, douts))

    def e2e_step(i):
        ids, _, _, _, _, _, lens = steps_io[i % COPIES]
        _, _, (hq, hkn, hvn), (hou, hls) = host[i % COPIES]
        s.ctx.decode(ids, hq, hkn, hvn, hou, hls, stream)
        s.ctx.request_truncate(ids, lens)

    def staged_step(i):
        ids, _, _, _, _, _, lens = steps_io[i % COPIES]
        hin, hout, _, _ = host[i % COPIES]
        din, dout, (dq, dkn, dvn), (dou, dls) = dev_io[i % COPIES]
        din.copy_(hin, non_blocking=True)
        s.ctx.decode(ids, dq, dkn, dvn, dou, dls, stream)
        hout.copy_(dout, non_blocking=True)
        s.ctx.request_truncate(ids, lens)

    ms_e = timed_loop(e2e_step, steps)
    ms_c = timed_loop(staged_step, min(steps, 500))
    status = s.ctx.device_status()
    s.ctx.close()
    del s, t, host, dev_io
    torch.cuda.empty_cache()
    dom = "dense_tcgen05"
    return {"workload": "llama3_8b_decode: Hq32 Hkv8 d128, 4 x 4096-token prefixes, 64 requests, "
                        "suffixes U[256,1024]",
            "value": round(value, 1), "unit": "GB/s", "steps": steps, "warmup": warmup,
            "ms_per_step": round(ms / steps, 5),
            "hbm_frac_of_measured": round(value / hbm_peak, 4),
            "hbm_frac_of_8tbs": round(value / 8000.0, 4),
            "tokens_per_s": round(n / (period_us * 1e-6), 1),
            "bytes_per_step": step_bytes, "prefix_bytes": prefix_b, "suffix_bytes": suffix_b,
            "l2": f"{COPIES} copies cycled, {COPIES * step_bytes / 1e9:.2f} GB between reuses",
            "steps20_ms_per_step": round(ms20 / 20, 5),
            "roofline": {"bound": "hbm", "kernel": dom, "achieved": round(value, 1),
                         "peak": hbm_peak, "unit": "GB/s", "frac": round(value / hbm_peak, 4),
                         "peak_source": peak_src, "traffic": profiled_traffic(PROFILE_8B),
                         "bytes_per_launch": step_bytes, "avg_launch_us": round(period_us, 2),
                         "avg_launch_from": "timed region / unified-kernel launches (back to back)",
                         "bracketed_avg_us": kernels.get(dom, {}).get("bracketed_avg_us")},
            "kernels": kernels,
            "e2e": {"value": round(step_bytes * steps / (ms_e / 1e3) / 1e9, 1), "unit": "GB/s",
                    "ms_per_step": round(ms_e / steps, 4),
                    "copy_engine_value": round(step_bytes * min(steps, 500) / (ms_c / 1e3) / 1e9, 1)},
            "device_status": status}


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
                         "frac_of_sustained": round(ach / peaks()[2], 4),
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
            # the staged reload's page scatter alone (its kernel bracketed by events):
            # it reads the staging area and writes the pages, 2 x bytes of HBM traffic
            ctx.set_option(B.OPT_KERNEL_TIMING, 1)
            ctx.kernel_times(reset=True)
            timed(reload, before=evict)
            kt = ctx.kernel_times(reset=True)
            ctx.set_option(B.OPT_KERNEL_TIMING, 0)
            scatter_us = 1e3 * kt["page_copy"][0] / max(1, kt["page_copy"][1])
        side.synchronize()
        rows.append({"tokens": ell, "bytes": ell * mu, "reload_us": round(t_re, 1),
                     "scatter_kernel_us": round(scatter_us, 1),
                     "scatter_hbm_gbs": round(2 * ell * mu / (scatter_us * 1e-6) / 1e9, 1),
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
    big = rows[-1]
    hbm_peak = peaks()[0]
    res["reload_scatter"] = {
        "tokens": big["tokens"], "kernel_us": big["scatter_kernel_us"],
        "hbm_gbs": big["scatter_hbm_gbs"], "frac": round(big["scatter_hbm_gbs"] / hbm_peak, 4),
        "frac_of_8tbs": round(big["scatter_hbm_gbs"] / 8000.0, 4),
        "bytes": "staging area read + pages written, 2 x the prefix's bytes"}
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
    under one KV budget, every further co-resident prefix takes pages that
    would otherwise hold request suffixes, so the admissible decode batch
    shrinks.  Budget 49152 tokens of one Llama-3-8B layer; every request
    holds a 2048-token suffix.  Two prefix lengths:

      16384 tokens  the Grouped / Alternating pair (1 resident prefix
                    admits 16 requests, 2 admit 8);
      4096 tokens   1, 2, 3, 4, 6 and 8 resident prefixes.

    The batch is the largest the budget admits, its requests spread
    round-robin over the resident prefixes.  Each step reads about the
    whole budget whatever the split, so tokens/s follows the batch.  Two
    copies of each point's workload are cycled (0.4 GB between reuses)."""
    import torch
    from paper_2608_25523_gb300 import binding as B
    from paper_2608_25523_gb300.session import Session
    from paper_2608_25523_gb300.workloads import copy_requests, replicate, small_case, tensors_torch

    budget, ls = 49152, 2048
    series = {16384: [1, 2], 4096: [1, 2, 3, 4, 6, 8]}
    res = {"workload": f"KV budget {budget} tokens (llama3_8b layer), suffixes {ls}; "
                       "decode steps of the admitted batch", "budget_tokens": budget,
           "suffix_tokens": ls, "series": {}}
    stream = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    for lp, ks in series.items():
        pts = []
        for k in ks:
            n = (budget - k * lp) // ls
            agents = [i % k for i in range(n)]
            base = small_case(7, hq=32, hkv=8, d=128, prefix_len=[lp] * k, req_agent=agents,
                              req_ctx=[ls - 1] * n, req_prefill=[0] * n, req_decode=[1] * n)
            assert base.pages_needed() * 16 <= budget
            w = replicate(base, 2)
            t = tensors_torch(w, dev)
            s = Session(w, t, device=dev, extra_tokens=16)
            io = []
            for c in range(2):
                ids, q, kn, vn = s.decode_inputs(copy_requests(w, 2, c))
                out, lse = s.new_outputs(n)
                io.append((B.i32_array(ids), B.i32_array([w.req_ctx[r] for r in ids]), q, kn, vn,
                           out, lse))

            def step(i):
                ida, lna, q, kn, vn, out, lse = io[i % 2]
                s.ctx.decode(ida, q, kn, vn, out, lse, stream)
                s.ctx.request_truncate(ida, lna)
            for i in range(10):
                step(i)
            torch.cuda.synchronize(dev)
            reps = 400
            e0.record(stream)
            for i in range(reps):
                step(i)
            e1.record(stream)
            e1.synchronize()
            us = e0.elapsed_time(e1) / reps * 1e3
            step_bytes = decode_bytes(w, copy_requests(w, 2, 0))[2]
            pts.append({"resident_prefixes": k, "batch": n, "step_us": round(us, 2),
                        "tokens_per_s": round(n / (us / 1e6), 1),
                        "gbs": round(step_bytes / (us / 1e6) / 1e9, 1),
                        "device_status": s.ctx.device_status()})
            s.ctx.close()
            del s, t, io
        res["series"][str(lp)] = pts
    g, a = res["series"]["16384"]
    res["grouped_over_alternating_tokens_per_s"] = round(g["tokens_per_s"] / a["tokens_per_s"], 2)
    torch.cuda.empty_cache()
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
    """Time the fp64 oracle on this host's cores over a bounded sample of the
    llama3_70b_decode step (one layer; the per-layer rate is the rate of a
    step through every layer).  The sample unit is one (request, kv head):
    the oracle's decode step for the G query heads of that kv head over the
    request's materialised prefix + suffix + new token.  The units come from
    16 of the 512 requests, drawn with a fixed seed, with their own suffix
    lengths; all six prefixes have 16384 tokens, so one drawn prefix stands
    for each request's.  A unit is credited with the step's algorithmic
    bytes in proportion to its keys: value = step bytes x (keys of the
    units done / keys of all 4096 units) / time."""
    import numpy as np

    import oracle
    from paper_2608_25523_gb300.workloads import config, small_case, tensors_numpy

    full = config(4)
    dec = full.decode_requests()
    step_bytes = decode_bytes(full, dec)[2]
    hkv, G = full.num_kv_heads, full.group
    keys_all = sum(full.prefix_len[full.req_agent[r]] + full.req_ctx[r] + 1 for r in dec) * hkv
    rng = np.random.default_rng(2024)
    pick = sorted(int(x) for x in rng.choice(len(dec), size=16, replace=False))
    ctx = [full.req_ctx[dec[i]] for i in pick]
    lp = full.prefix_len[0]
    w = small_case(4, hq=full.num_q_heads, hkv=hkv, d=full.head_dim, prefix_len=[lp],
                   req_agent=[0] * len(pick), req_ctx=ctx, req_prefill=[0] * len(pick),
                   req_decode=[1] * len(pick))
    t = tensors_numpy(w)
    pk, pv = t.prefix(0, w)
    units = [(i, g) for i in range(len(pick)) for g in range(hkv)]

    def run(us):
        keys = 0
        for i, g in us:
            n_cached = w.req_ctx[i]
            sk, sv = t.suffix(i, w, 0, n_cached)
            nk, nv = t.suffix(i, w, n_cached, n_cached + 1)
            oracle.decode_step(t.q_decode[i, g * G:(g + 1) * G], pk[:, g:g + 1], pv[:, g:g + 1],
                               sk[:, g:g + 1], sv[:, g:g + 1], nk[0, g:g + 1], nv[0, g:g + 1])
            keys += lp + n_cached + 1
        return keys

    t0 = time.perf_counter()
    run(units[:1])
    one = time.perf_counter() - t0
    total_s, done_keys, done, pos = 0.0, 0, 0, 0
    if per_step_s is None:
        # one timed region of about budget_s seconds, units cycled over the sample
        t_end = time.perf_counter() + budget_s
        t0 = time.perf_counter()
        while done == 0 or time.perf_counter() < t_end:
            k = max(1, min(len(units), int(0.5 / max(one, 1e-6))))
            done_keys += run([units[(pos + j) % len(units)] for j in range(k)])
            pos += k
            done += k
        total_s = time.perf_counter() - t0
        per = done
    else:
        per = max(1, int(per_step_s / max(one, 1e-6)))
        for i in range(warmup + steps):
            sample = [units[(pos + j) % len(units)] for j in range(per)]
            pos += per
            t0 = time.perf_counter()
            kk = run(sample)
            dt = time.perf_counter() - t0
            if i >= warmup:
                total_s += dt
                done += per
                done_keys += kk
    frac = done_keys / keys_all
    value = step_bytes * frac / total_s / 1e9
    return {"value": round(value, 4), "unit": "GB/s", "cores": _blas_threads(), "kind": "oracle",
            "sample": (f"{done} (request, kv head) units of one llama3_70b_decode layer step "
                       f"(16 seeded requests x 8 kv heads, cycled; {frac:.3f} layer steps' worth)"
                       + ("" if per_step_s is None else f", {per} per timed step, {steps} steps")
                       + "; fp64 numpy over materialised K/V"),
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
            "data": "synthetic (seeded N(0,1) bf16-valued Q/K/V)",
            "config": headline_config(args.layers_70b, world),
            "cpu_baseline": cb,
            "e2e": {"value": cb["value"], "unit": "GB/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


# ------------------------------------------------------------ the line ---

CONTRACT_KEYS = ["metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
                 "higher_is_better", "scaling", "vs_baseline", "dtype", "data", "config",
                 "ms_per_layer", "hbm_frac_of_measured", "hbm_frac_of_8tbs", "tokens_per_s",
                 "roofline", "kernels", "e2e", "gpu_launches", "clocks", "device_status",
                 "cpu_baseline"]


def _csv(xs):
    return ",".join(str(x) for x in xs)


def compact(res):
    """The printed line: the headline's keys in full and every extra reduced
    to a few scalars, so the whole line stays short."""
    out = {k: res[k] for k in CONTRACT_KEYS if k in res}
    x = res.get("decode_8b")
    if x:
        out["decode_8b"] = {"value": x["value"], "unit": "GB/s", "steps": x["steps"],
                            "ms_per_step": x["ms_per_step"], "frac": x["roofline"]["frac"],
                            "frac_of_8tbs": x.get("hbm_frac_of_8tbs"),
                            "bracketed_kernel_us": x["roofline"]["bracketed_avg_us"],
                            "steps20_ms_per_step": x["steps20_ms_per_step"],
                            "tokens_per_s": x["tokens_per_s"], "e2e_gbs": x["e2e"]["value"],
                            "traffic": x["roofline"]["traffic"], "device_status": x["device_status"]}
    x = res.get("prefill")
    if x:
        out["prefill"] = {"tflops": x["tflops"], "ms": x["ms"], "tokens_per_s": x["tokens_per_s"],
                          "kernel_tflops": x["roofline"]["achieved"], "frac": x["roofline"]["frac"],
                          "peak": x["roofline"]["peak"],
                          "frac_of_sustained": x["roofline"].get("frac_of_sustained"),
                          "device_status": x["device_status"]}
    x = res.get("mixed")
    if x:
        k = x["kernels_per_step"]
        out["mixed"] = {"ms_per_step": x["ms_per_step"],
                        "decode_tokens_per_s": x["decode_tokens_per_s"],
                        "prefill_kernel_tflops": k.get("prefill_pair_tcgen05", {}).get("tflops"),
                        "decode_kernel_gbs": k.get("dense_tcgen05", {}).get("gbs"),
                        "device_status": x["device_status"]}
    x = res.get("movement")
    if x:
        out["movement"] = {"reload_gbs": x["reload"]["B_gbs"], "offload_gbs": x["offload"]["B_gbs"],
                           "reload_direct_gbs": x["reload_direct"]["B_gbs"],
                           "offload_direct_gbs": x["offload_direct"]["B_gbs"],
                           "h2d_copy_gbs": x["h2d_copy"]["B_gbs"],
                           "mu_over_B_swap_ns": x["mu_over_B_swap_ns_per_token"]["reload"],
                           "reload_scatter_hbm_gbs": (x.get("reload_scatter") or {}).get("hbm_gbs"),
                           "reload_scatter_frac": (x.get("reload_scatter") or {}).get("frac"),
                           "bit_exact": all(r["round_trip_bit_exact"] for r in x["rows"])}
    x = res.get("redo")
    if x:
        out["redo"] = {"tokens": _csv(r["tokens"] for r in x["rows"]),
                       "decode_kernel_ms": _csv(r["decode_redo_kernel_ms"] for r in x["rows"]),
                       "prefill_kernel_ms": _csv(r["prefill_rebuild_kernel_ms"] for r in x["rows"]),
                       "T_decode_us_per_token": x["rows"][-1]["T_decode_us_per_token"],
                       "device_status": x["device_status"]}
    x = res.get("coresidency")
    if x:
        c = {"budget_tokens": x["budget_tokens"], "suffix_tokens": x["suffix_tokens"]}
        for lp, pts in x["series"].items():
            c[f"p{lp}_prefixes"] = _csv(p["resident_prefixes"] for p in pts)
            c[f"p{lp}_batch"] = _csv(p["batch"] for p in pts)
            c[f"p{lp}_step_us"] = _csv(p["step_us"] for p in pts)
            c[f"p{lp}_tokens_per_s"] = _csv(int(p["tokens_per_s"]) for p in pts)
        c["grouped_over_alternating"] = x["grouped_over_alternating_tokens_per_s"]
        out["coresidency"] = c
    x = res.get("sched")
    if x:
        out["sched"] = {"tasks": x["tasks"], "decisions": x["decisions"],
                        "native_decide_us_mean": x["native_decide_us_mean"],
                        "native_decide_us_max": x["native_decide_us_max"],
                        "oracle_decide_us": (x.get("cpu_baseline") or {}).get("value"),
                        "preemptions": x["preemptions"], "prefix_moves_in": x["prefix_moves_in"],
                        "mean_jct_s": x["mean_jct_s"], "device_status": x["device_status"]}
    return out


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-extras", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--only", choices=["decode_70b", "decode_8b", "prefill", "mixed", "movement",
                                       "redo", "coresidency", "sched"],
                    help="run just one workload (1 GPU) and print its full result")
    ap.add_argument("--layers-70b", type=int, default=LAYERS_70B,
                    help="layer pools of the 70B decode workload (5.4 GB of KV each; "
                         "26 fill 80 %% of 180 GB), capped by the free memory")
    ap.add_argument("--prefill-stride", type=int, default=1,
                    help="prefill workload: every k-th request only (a small case for profiling)")
    ap.add_argument("--detail", default=None,
                    help="also write the full result (every extra in full) to this JSON file")
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
        fn = {"decode_70b": lambda: measure_70b(args, 0, 1, dev, hbm_peak, peak_src, args.steps,
                                                args.warmup, with_e2e=False),
              "decode_8b": lambda: bench_decode_8b(args, dev, hbm_peak, peak_src, steps=args.steps,
                                                   warmup=args.warmup),
              "prefill": lambda: bench_prefill(args, dev, tf_peak, peak_src),
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
        if args.detail:
            with open(args.detail, "w") as fh:
                json.dump(res, fh, indent=1)
        print(json.dumps(compact(res)))
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
